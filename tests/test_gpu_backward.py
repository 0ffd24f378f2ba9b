"""GPU parity of dla_backward: the gradients of the read-out with the forward
pass's decisions held fixed, against the fp64 gradient oracle (oracle/grad.py,
itself pinned by finite differences of the recurrent oracle in
test_oracle_grad.py).

The decision trace given to both sides is the oracle's forward trace of the
same inputs, so the backward kernels are checked on their own; upstream
gradients are seeded N(0, 1).  Outputs must be within the bf16-input tolerance
(max-abs 2e-2) and, as a sharper check of the hi + lo operand splits, within
1e-4 of the largest gradient magnitude (a single bf16 rounding of the
weighted products would give about 2e-3)."""
import numpy as np
import pytest
import torch

import oracle
from oracle import grad as G
from paper_2606_10650_gb300 import dla
from paper_2606_10650_gb300 import workloads as W
from parity_util import upload

pytestmark = pytest.mark.gpu

CASES = {
    # name: (workload, overrides)
    "standard_bf16": ("standard", dict(B=1, H=2, T=700)),
    "churn_bf16": ("long", dict(B=1, H=2, T=1500, block=256)),      # a merge at most tokens of the i.i.d. spans
    "small_cache_bf16": ("regime", dict(B=2, H=2, T=300, C=3, tau=1.2)),
    "d64_bf16": ("standard", dict(B=2, H=2, T=700, d=64, C=8, tau=1.4215)),
}


def _grads_gpu(w, q, k, v, lam, bnd, mlog, g, want_lam=True):
    dev = torch.device("cuda:0")
    qt, kt, vt, lt = upload(w, q, k, v, lam)
    gt = torch.from_numpy(np.ascontiguousarray(g, dtype=np.float32)).to(dev)
    bt = torch.from_numpy(np.ascontiguousarray(bnd, dtype=np.uint8)).to(dev)
    mt = torch.from_numpy(np.ascontiguousarray(mlog, dtype=np.int32)).to(dev)
    out = dla.backward(qt, kt, vt, lt, bt, mt, gt, capacity=w.C, want_lam=want_lam)
    st = dla.dla_sync_status()
    return {k_: (None if x is None else x.double().cpu().numpy()) for k_, x in out.items()}, st


def _grads_oracle(w, q, k, v, lam, bnd, mlog, g):
    B, T, H, d = k.shape
    r = dict(dq=np.zeros((B, T, H, d)), dk=np.zeros((B, T, H, d)), dv=np.zeros((B, T, H, d)),
             dlam=None if lam is None else np.zeros((B, T, H, w.C)))
    for b in range(B):
        for h in range(H):
            x = G.readout_grads(q[b, :, h], k[b, :, h], v[b, :, h], None if lam is None else lam[b, :, h],
                                bnd[b, h], mlog[b, h], g[b, :, h])
            r["dq"][b, :, h], r["dk"][b, :, h], r["dv"][b, :, h] = x["dq"], x["dk"], x["dv"]
            if lam is not None:
                r["dlam"][b, :, h] = x["dlam"]
    return r


def _check(gpu, ref, keys=("dq", "dk", "dv", "dlam")):
    rep = {}
    for key in keys:
        if ref.get(key) is None:
            continue
        err = np.abs(gpu[key] - ref[key]).max()
        scale = max(1.0, np.abs(ref[key]).max())
        rep[key] = (float(err), float(err / scale))
        assert err <= 2e-2, (key, err)
        assert err <= 1e-4 * scale, (key, err, scale)
    return rep


def _inputs(w, seed=7):
    q, k, v, lam = W.host_batch(w, T=w.T)
    r = oracle.forward(q, k, v, lam, tau=w.tau, C=w.C, eps=w.eps, rms_eps=w.rms_eps,
                       want_o=np.zeros(w.T, bool))
    g = np.random.default_rng(seed).standard_normal(q.shape)
    return q, k, v, lam, r["boundary"], r["merge_log"], g


@pytest.mark.parametrize("case", list(CASES))
def test_backward_parity(case):
    name, ov = CASES[case]
    w = W.get(name, **ov)
    q, k, v, lam, bnd, mlog, g = _inputs(w)
    gpu, st = _grads_gpu(w, q, k, v, lam, bnd, mlog, g)
    assert st == 0
    rep = _check(gpu, _grads_oracle(w, q, k, v, lam, bnd, mlog, g))
    print(case, "boundaries", int(bnd.sum()), "merges", int((mlog >= 0).sum()), rep)


def test_backward_churn_case_merges():
    """The churn case is not vacuous: most of its boundaries merge."""
    w = W.get("long", B=1, H=2, T=1500, block=256)
    _, _, _, _, bnd, mlog, _ = _inputs(w)
    assert (mlog >= 0).sum() > 300


def test_backward_lambda_null():
    """lambda = NULL: every weight is 1 (the gradient of causal linear
    attention); no dlambda is asked for."""
    w = W.get("standard", B=1, H=2, T=333)
    q, k, v, _, bnd, mlog, g = _inputs(w)
    gpu, st = _grads_gpu(w, q, k, v, None, bnd, mlog, g, want_lam=False)
    assert st == 0
    _check(gpu, _grads_oracle(w, q, k, v, None, bnd, mlog, g), keys=("dq", "dk", "dv"))


def test_backward_reports_an_inconsistent_trace():
    """A merge index outside the live pairs is found by the slot-list replay:
    status 6, and the next call on the stream is correct."""
    w = W.get("standard", B=1, H=1, T=256)
    q, k, v, lam, bnd, mlog, g = _inputs(w)
    bad = mlog.copy()
    t = int(np.flatnonzero(bnd[0, 0])[1])  # the second boundary: one live state before it
    bad[0, 0, t] = 5
    _, st = _grads_gpu(w, q, k, v, lam, bnd, bad, g)
    assert st == 6
    gpu, st = _grads_gpu(w, q, k, v, lam, bnd, mlog, g)
    assert st == 0
    _check(gpu, _grads_oracle(w, q, k, v, lam, bnd, mlog, g))
