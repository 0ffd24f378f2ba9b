"""GPU parity of the CUDA path (through the C ABI) against the fp64 oracle on
decision-safe seeded inputs, at sizes where the oracle checks every stream,
token and state.  Sizes span several scan chunks / read-out intervals and a
ragged tail."""
import dataclasses

import numpy as np
import pytest
import torch

import oracle
from paper_2606_10650_gb300 import dla
from paper_2606_10650_gb300 import workloads as W
from parity_util import TOL, compare, run_gpu, run_oracle, structural_checks, upload
from safe_inputs import safe_batch, safe_stream

pytestmark = pytest.mark.gpu


def _safe(w, T=None, seed=None, score_mode=0):
    T = w.total_tokens if T is None else T
    q, k, v, lam = W.host_batch(w, seed=seed, T=T)
    for b in range(w.B):
        for h in range(w.H):
            r = safe_stream(w, b, h, T=T, seed=seed, score_mode=score_mode)
            q[b, :, h], k[b, :, h], v[b, :, h], lam[b, :, h] = r["q"], r["k"], r["v"], r["lam"]
    return q, k, v, lam


CASES = {
    # name: (workload, overrides)
    "tiny_fp32": ("tiny", dict()),
    "standard_bf16": ("standard", dict(B=1, H=3, T=1000)),
    "regime_bf16": ("regime", dict(B=1, H=2, T=2500)),
    "long_churn_bf16": ("long", dict(B=1, H=2, T=1500, block=256)),
    "d64_bf16": ("standard", dict(B=2, H=2, T=700, d=64, C=8, tau=1.4215)),
    "d128_fp32": ("tiny", dict(B=1, H=2, T=300, d=128, C=6, tau=1.4142)),
    # more streams than CTA pairs fit on the device: one scan CTA per stream
    "many_streams_bf16": ("regime", dict(B=3, H=27, T=300, C=3, tau=1.2)),
    # more streams than SMs: the scan cannot keep every stream resident, so the
    # forward pass takes the per-round schedule whatever DLA_SCHEDULE says
    "streams_beyond_sms_bf16": ("regime", dict(B=4, H=40, T=200, C=3, tau=1.2)),
}


@pytest.mark.parametrize("case", list(CASES))
def test_forward_parity(case):
    name, ov = CASES[case]
    w = W.get(name, **ov)
    q, k, v, lam = _safe(w)
    g = run_gpu(w, q, k, v, lam)
    r = run_oracle(w, q, k, v, lam)
    rep = {}
    compare(w, g, r, report=rep)
    structural_checks(w, g, w.T)
    assert g["boundary"].sum() > 2
    print(case, rep)


def test_merges_are_exercised():
    """The small cases above do merge (the fixtures are not vacuous)."""
    w = W.get("long", B=1, H=1, T=1200, block=256)
    q, k, v, lam = _safe(w)
    g = run_gpu(w, q, k, v, lam)
    assert (g["merge_log"] >= 0).sum() > 100


def test_lambda_null_is_causal_linear_attention():
    """lambda = NULL (all ones): merges only regroup sums, so o must be causal
    linear attention (Eq. linear_attn_parallel), whatever the decisions."""
    w = W.get("standard", B=1, H=2, T=777)
    q, k, v, _ = W.host_batch(w, T=w.T)
    g = run_gpu(w, q, k, v, None)
    for h in range(w.H):
        Q, K, V = q[0, :, h], k[0, :, h], v[0, :, h]
        O = np.tril(Q @ K.T) @ V
        assert np.abs(g["o"][0, :, h] - O).max() <= TOL["bf16"]


def test_score_mode_literal_equation():
    """score_mode 1 (Eq. importance_score with S_t = S_{t-1} + s_t)."""
    w0 = W.get("tiny", T=400)
    q, k, v, lam = W.host_batch(w0, T=w0.T)
    st = oracle.Stream(w0.C, w0.d, w0.d, 1e300, score_mode=1)
    _, _, _, it = st.run(q[0, :, 0], k[0, :, 0], v[0, :, 0])
    w = dataclasses.replace(w0, tau=float(np.quantile(it[1:], 0.8)))
    q, k, v, lam = _safe(w, score_mode=1)
    g = run_gpu(w, q, k, v, lam, score_mode=1)
    r = run_oracle(w, q, k, v, lam, score_mode=1)
    compare(w, g, r)
    assert g["boundary"].sum() > 10


def test_bf16_output_dtype():
    w = W.get("standard", B=1, H=2, T=300)
    q, k, v, lam = _safe(w)
    g = run_gpu(w, q, k, v, lam, out_dtype=torch.bfloat16)
    r = run_oracle(w, q, k, v, lam)
    compare(w, g, r, tol=TOL["bf16"] + 2.0 ** -8 * np.abs(r["o"]).max())


@pytest.mark.parametrize("T", [1, 2, 63, 64, 65, 129])
def test_edge_lengths(T):
    w = W.get("tiny", T=T, C=3)
    q, k, v, lam = _safe(w)
    g = run_gpu(w, q, k, v, lam)
    r = run_oracle(w, q, k, v, lam)
    compare(w, g, r)
    assert g["boundary"][0, 0, 0] == 1


@pytest.mark.parametrize("T", [1, 2, 127, 128, 129, 255, 383])
def test_edge_lengths_tensor_core_path(T):
    """bf16, d = 128 (the scan on CTA pairs, the tensor-core read-out): a
    single token, one interval exactly, one token past it, odd interval counts
    and a ragged last interval, whose output rows past T the read-out's TMA
    store must clip."""
    w = W.get("regime", B=1, H=2, T=T, C=8, tau=1.2)
    q, k, v, lam = _safe(w)
    g = run_gpu(w, q, k, v, lam)
    r = run_oracle(w, q, k, v, lam)
    compare(w, g, r)
    assert g["boundary"][0, 0, 0] == 1


def test_many_rounds_small_workspace():
    """The smallest workspace forces one read-out interval per round; the
    result must not change."""
    w = W.get("regime", B=1, H=2, T=1100)
    q, k, v, lam = _safe(w)
    p = dla.make_params(w.tau, w.C)
    nb = dla.dla_forward_min_workspace(p, w.B, w.T, w.H, w.d, w.d, dla.DLA_BF16, True)
    g = run_gpu(w, q, k, v, lam, ws_bytes=nb)
    r = run_oracle(w, q, k, v, lam)
    compare(w, g, r)


def test_prefill_continuation_from_cache():
    """forward(T0) then forward(T - T0) from the cache equals forward(T)."""
    w = W.get("regime", B=1, H=2, T=1300)
    q, k, v, lam = _safe(w)
    T0 = 517
    r = run_oracle(w, q, k, v, lam)
    wa = dataclasses.replace(w, T=T0)
    ga = run_gpu(wa, q[:, :T0], k[:, :T0], v[:, :T0], lam[:, :T0])
    wb = dataclasses.replace(w, T=w.T - T0)
    gb = run_gpu(wb, q[:, T0:], k[:, T0:], v[:, T0:], lam[:, T0:], cache=ga["cache"], from_cache=True)
    bnd = np.concatenate([ga["boundary"], gb["boundary"]], axis=2)
    ml = np.concatenate([ga["merge_log"], gb["merge_log"]], axis=2)
    o = np.concatenate([ga["o"], gb["o"]], axis=1)
    g = dict(boundary=bnd, merge_log=ml, o=o, cache=gb["cache"])
    compare(w, g, r)


def test_decode_steps_match_prefill():
    """dla_forward over T0 tokens, then one dla_decode_step per token, equals
    the oracle over all T tokens (Sec. 3.1 inference rule is the same
    recurrence)."""
    w = W.get("decode", B=3, H=2, T=300, decode_steps=90, C=4, tau=1.4142)
    Ttot = w.total_tokens
    q, k, v, lam = _safe(w, T=Ttot)
    r = run_oracle(w, q, k, v, lam)
    wp = dataclasses.replace(w, decode_steps=0)
    gp = run_gpu(wp, q[:, :w.T], k[:, :w.T], v[:, :w.T], lam[:, :w.T], want_o=False)
    cache = gp["cache"]
    dev = torch.device("cuda:0")
    p = dla.make_params(w.tau, w.C, w.eps, w.rms_eps)
    o_all = np.zeros((w.B, w.decode_steps, w.H, w.d))
    b_all = np.zeros((w.B, w.H, w.decode_steps), np.uint8)
    m_all = np.zeros((w.B, w.H, w.decode_steps), np.int32)
    for s in range(w.decode_steps):
        t = w.T + s
        qt, kt, vt, lt = upload(w, q[:, t], k[:, t], v[:, t], lam[:, t])
        o = torch.empty((w.B, w.H, w.d), dtype=torch.float32, device=dev)
        bb = torch.empty((w.B, w.H), dtype=torch.uint8, device=dev)
        mi = torch.empty((w.B, w.H), dtype=torch.int32, device=dev)
        dla.dla_decode_step(p, cache, qt.contiguous(), kt.contiguous(), vt.contiguous(), lt.contiguous(), o, bb, mi)
        o_all[:, s] = o.double().cpu().numpy()
        b_all[:, :, s] = bb.cpu().numpy()
        m_all[:, :, s] = mi.cpu().numpy()
    torch.cuda.synchronize()
    np.testing.assert_array_equal(gp["boundary"], r["boundary"][:, :, :w.T])
    np.testing.assert_array_equal(b_all, r["boundary"][:, :, w.T:])
    np.testing.assert_array_equal(m_all, r["merge_log"][:, :, w.T:])
    assert np.abs(o_all - r["o"][:, w.T:]).max() <= TOL["bf16"]
    g = dict(boundary=r["boundary"], merge_log=r["merge_log"], o=None, cache=cache)
    compare(w, g, r)
    assert b_all.sum() > 0 and (m_all >= 0).sum() > 0


@pytest.mark.parametrize("sched", ["rounds", "serial"])
@pytest.mark.parametrize("case", ["standard_bf16", "regime_bf16", "long_churn_bf16"])
def test_forward_parity_other_schedules(case, sched, monkeypatch):
    """The rounds schedule (scan and read-out alternating round by round) and
    the serial one (pre-pass, scan, read-out one after another) give the
    oracle's results too."""
    monkeypatch.setenv("DLA_SCHEDULE", sched)
    name, ov = CASES[case]
    w = W.get(name, **ov)
    q, k, v, lam = _safe(w)
    g = run_gpu(w, q, k, v, lam)
    r = run_oracle(w, q, k, v, lam)
    compare(w, g, r)
    structural_checks(w, g, w.T)


def test_concurrent_schedule_first_call_of_a_process():
    """The first forward pass of a process under the concurrent schedule loads
    every kernel before the read-out starts waiting for the scan (a lazily
    loaded scan would otherwise stall behind the waiting read-out)."""
    import os
    import subprocess
    import sys
    code = (
        "import numpy as np, torch\n"
        "from paper_2606_10650_gb300 import dla, workloads as W\n"
        "w = W.get('standard', B=1, H=2, T=700)\n"
        "q, k, v, lam = W.host_batch(w, T=w.T)\n"
        "dev = torch.device('cuda:0')\n"
        "qt, kt, vt = (W.to_device(x, w.dtype, dev) for x in (q, k, v))\n"
        "o = torch.empty(qt.shape, dtype=torch.float32, device=dev)\n"
        "cache = dla.Cache(1, 2, w.C, 128, device=dev)\n"
        "p = dla.make_params(w.tau, w.C, w.eps, w.rms_eps)\n"
        "ws = dla.dla_forward(p, qt, kt, vt, None, o, cache, None, None)\n"
        "torch.cuda.synchronize()\n"
        "print('STATUS', dla.workspace_status(ws))\n")
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    env = dict(os.environ, PYTHONPATH=root)
    env.pop("DLA_SCHEDULE", None)  # the default schedule is the concurrent one
    out = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True, timeout=300)
    assert out.returncode == 0, out.stderr[-2000:]
    assert "STATUS 0" in out.stdout, out.stdout[-2000:]


@pytest.mark.parametrize("sched", ["concurrent", "rounds"])
@pytest.mark.parametrize("case", ["regime_bf16", "standard_bf16", "d128_fp32"])
def test_forward_host_buffers(case, sched, monkeypatch):
    """dla_forward_host: q, k, v, lambda and o in page-locked host memory.  On
    the concurrent schedule (bf16, d = 128) the inputs stream in piece by piece
    beside the scan, which forms its Gram entries itself; elsewhere they are
    copied first.  The oracle's results either way."""
    monkeypatch.setenv("DLA_SCHEDULE", sched)
    name, ov = CASES[case]
    w = W.get(name, **ov)
    q, k, v, lam = _safe(w)
    qt, kt, vt, lt = upload(w, q, k, v, lam)
    qh, kh, vh, lh = (x.cpu().pin_memory() for x in (qt, kt, vt, lt))
    B, T, H, d = kh.shape
    dev = torch.device("cuda:0")
    cache = dla.Cache(B, H, w.C, d, device=dev)
    p = dla.make_params(w.tau, w.C, w.eps, w.rms_eps)
    oh = torch.full((B, T, H, d), float("nan"), dtype=torch.float32).pin_memory()
    bnd = torch.full((B, H, T), 7, dtype=torch.uint8, device=dev)
    ml = torch.full((B, H, T), -7, dtype=torch.int32, device=dev)
    ws = dla.dla_forward_host(p, qh, kh, vh, lh, oh, cache, bnd, ml, device=dev)
    torch.cuda.synchronize()
    assert dla.workspace_status(ws) == 0, "device status word reports a failure"
    g = dict(o=oh.double().numpy(), boundary=bnd.cpu().numpy(), merge_log=ml.cpu().numpy(), cache=cache)
    r = run_oracle(w, q, k, v, lam)
    compare(w, g, r)
    structural_checks(w, g, w.T)


def test_dla_i_without_capacity_bound():
    """DLA(I) (Table 5: dynamic merging without the capacity bound) on the GPU:
    with C = 64 above each stream's number of segments nothing merges, and the
    oracle without a capacity bound (C = T + 1) gives the same decisions and
    outputs."""
    w = W.get("regime", B=1, H=2, T=1500, C=64)
    q, k, v, lam = _safe(w)
    g = run_gpu(w, q, k, v, lam)
    assert (g["merge_log"] == -1).all() and g["boundary"].sum() > 4
    lam_o = np.zeros(lam.shape[:3] + (w.T + 1,))
    lam_o[..., :w.C] = lam
    r = oracle.forward(q, k, v, lam_o, tau=w.tau, C=w.T + 1, eps=w.eps, rms_eps=w.rms_eps)
    compare(w, g, r, check_cache=False)
    structural_checks(w, g, w.T)


@pytest.mark.timeout(900)
@pytest.mark.parametrize("sched", ["concurrent", "rounds"])
def test_dla_i_beyond_64_segments(sched, monkeypatch):
    """DLA(I) (Table 5: dynamic merging without the capacity bound) at the regime
    workload's length, where streams open up to about 80 segments: with C = 128
    (the instances beyond 64, which hold no capacity merge) nothing merges, and
    decisions, caches and outputs equal the oracle's.  Outputs are compared on
    every 16th token (the oracle's read-out of up to 80 states at every token
    takes much longer than the rest)."""
    monkeypatch.setenv("DLA_SCHEDULE", sched)
    w = W.get("regime", B=1, H=5, C=128)
    q, k, v, lam = _safe(w)
    g = run_gpu(w, q, k, v, lam)
    want = np.zeros(w.T, bool)
    want[::16] = True
    want[-1] = True
    r = oracle.forward(q, k, v, lam, tau=w.tau, C=w.C, eps=w.eps, rms_eps=w.rms_eps, want_o=want)
    rep = {}
    compare(w, g, r, report=rep)
    structural_checks(w, g, w.T)
    assert (g["merge_log"] == -1).all()
    ex = g["cache"].export()
    assert ex["m"].max() > 64, ex["m"]
    print("segments", ex["m"].tolist(), rep)


def test_dla_i_segments_past_the_capacity_are_reported():
    """A capacity above 64 with a stream whose segments pass it (the DLA(I)
    instances hold no capacity merge): the call reports status 6 and the next
    call on the stream is correct."""
    w = W.get("regime", B=1, H=5, T=16384, C=65)
    q, k, v, lam = W.host_batch(w, T=w.T)
    qt, kt, vt, lt = upload(w, q, k, v, lam)
    dev = torch.device("cuda:0")
    p = dla.make_params(w.tau, w.C, w.eps, w.rms_eps)
    o = torch.zeros((w.B, w.T, w.H, w.d), dtype=torch.float32, device=dev)
    dla.dla_forward(p, qt, kt, vt, lt, o, dla.Cache(w.B, w.H, w.C, w.d, device=dev))
    assert dla.dla_sync_status() == 6
    w2 = W.get("regime", B=1, H=2, T=2000, C=96)
    q2, k2, v2, l2 = _safe(w2)
    g = run_gpu(w2, q2, k2, v2, l2)
    compare(w2, g, run_oracle(w2, q2, k2, v2, l2))


RAGGED = {
    # name: (workload, overrides, per-row lengths)
    "regime_bf16": ("regime", dict(B=3, H=2, T=1300), [1300, 517, 1]),
    "standard_bf16": ("standard", dict(B=3, H=2, T=700), [0, 700, 333]),
    "d64_bf16": ("standard", dict(B=2, H=2, T=700, d=64, C=8, tau=1.4215), [257, 700]),
    "d128_fp32": ("tiny", dict(B=2, H=2, T=300, d=128, C=6, tau=1.4142), [300, 129]),
}


@pytest.mark.parametrize("sched", ["concurrent", "rounds"])
@pytest.mark.parametrize("case", list(RAGGED))
def test_ragged_rows(case, sched, monkeypatch):
    """Ragged batches in the padded layout (dla_params.seq_lens): row b runs
    over its first seq_lens[b] tokens exactly as a call on those tokens alone
    (the oracle per row); padding tokens get boundary 0 and merge_log -1, and
    their output rows are not written."""
    monkeypatch.setenv("DLA_SCHEDULE", sched)
    name, ov, lens = RAGGED[case]
    w = W.get(name, **ov)
    q, k, v, lam = _safe(w)
    dev = torch.device("cuda:0")
    qt, kt, vt, lt = upload(w, q, k, v, lam)
    B, T, H, d = kt.shape
    sl = torch.tensor(lens, dtype=torch.int32, device=dev)
    cache = dla.Cache(B, H, w.C, d, device=dev)
    p = dla.make_params(w.tau, w.C, w.eps, w.rms_eps, seq_lens=sl)
    o = torch.full((B, T, H, d), float("nan"), dtype=torch.float32, device=dev)
    bnd = torch.full((B, H, T), 7, dtype=torch.uint8, device=dev)
    ml = torch.full((B, H, T), -7, dtype=torch.int32, device=dev)
    ws = dla.dla_forward(p, qt, kt, vt, lt, o, cache, bnd, ml)
    torch.cuda.synchronize()
    assert dla.workspace_status(ws) == 0, "device status word reports a failure"
    g = dict(o=o.double().cpu().numpy(), boundary=bnd.cpu().numpy(), merge_log=ml.cpu().numpy(), cache=cache)
    _check_ragged(w, q, k, v, lam, lens, g, cache)


def _check_ragged(w, q, k, v, lam, lens, g, cache):
    """Each row against the oracle on its own tokens; padding untouched."""
    B, T, H, d = k.shape
    r = dict(o=np.full((B, T, H, d), np.nan), boundary=np.zeros((B, H, T), np.uint8),
             merge_log=np.full((B, H, T), -1, np.int32), caches={})
    live = []
    for b, n in enumerate(lens):
        if n == 0:
            continue
        rb = oracle.forward(q[b:b + 1, :n], k[b:b + 1, :n], v[b:b + 1, :n], lam[b:b + 1, :n], tau=w.tau, C=w.C,
                            eps=w.eps, rms_eps=w.rms_eps)
        r["o"][b, :n] = rb["o"][0]
        r["boundary"][b, :, :n] = rb["boundary"][0]
        r["merge_log"][b, :, :n] = rb["merge_log"][0]
        for h in range(H):
            r["caches"][(b, h)] = rb["caches"][(0, h)]
            live.append((b, h))
    compare(w, g, r, streams=live)
    ex = cache.export()
    for b, n in enumerate(lens):
        assert np.isnan(g["o"][b, n:]).all(), f"row {b}: padding output written"
        np.testing.assert_array_equal(g["boundary"][b, :, n:], 0)
        np.testing.assert_array_equal(g["merge_log"][b, :, n:], -1)
        if n == 0:
            assert (ex["m"][b] == 0).all()


PACKED = {
    # name: (workload, overrides, per-row lengths); max_seqlen = T
    "regime_bf16": ("regime", dict(B=4, H=2, T=1300), [1300, 517, 1, 640]),
    "standard_bf16": ("standard", dict(B=4, H=2, T=700), [0, 700, 333, 64]),
    "d64_bf16": ("standard", dict(B=3, H=2, T=700, d=64, C=8, tau=1.4215), [257, 0, 700]),
    "d128_fp32": ("tiny", dict(B=2, H=2, T=300, d=128, C=6, tau=1.4142), [129, 300]),
}


def _pack(x, lens):
    """Rows x[b, :lens[b]] one after another: [sum(lens), ...]."""
    return np.ascontiguousarray(np.concatenate([x[b, :n] for b, n in enumerate(lens)], axis=0))


@pytest.mark.parametrize("sched", ["concurrent", "rounds", "serial"])
@pytest.mark.parametrize("case", list(PACKED))
def test_packed_rows(case, sched, monkeypatch):
    """Packed batches (dla_forward_varlen): the rows of different lengths lie one
    after another in q, k, v, lambda and o ([total_tokens, H, ...], offsets
    cu_seqlens); each row gives the oracle's results on its own tokens, the
    trace is padded per stream, and every value equals the padded layout's
    (dla_params.seq_lens) on the same rows."""
    monkeypatch.setenv("DLA_SCHEDULE", sched)
    name, ov, lens = PACKED[case]
    w = W.get(name, **ov)
    q, k, v, lam = _safe(w)
    dev = torch.device("cuda:0")
    B, T, H = w.B, w.T, w.H
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    total = int(cu[-1])
    qt, kt, vt, lt = upload(w, _pack(q, lens), _pack(k, lens), _pack(v, lens), _pack(lam, lens))
    d = kt.shape[-1]
    cache = dla.Cache(B, H, w.C, d, device=dev)
    p = dla.make_params(w.tau, w.C, w.eps, w.rms_eps)
    o = torch.full((total, H, d), float("nan"), dtype=torch.float32, device=dev)
    bnd = torch.full((B, H, T), 7, dtype=torch.uint8, device=dev)
    ml = torch.full((B, H, T), -7, dtype=torch.int32, device=dev)
    cut = torch.from_numpy(cu).to(dev)
    dla.dla_forward_varlen(p, cut, T, qt, kt, vt, lt, o, cache, bnd, ml)
    assert dla.dla_sync_status() == 0, "device status reports a failure"
    og = o.double().cpu().numpy()
    assert not np.isnan(og).any(), "an output row of the packed batch was not written"
    o_rows = np.full((B, T, H, d), np.nan)
    for b, n in enumerate(lens):
        o_rows[b, :n] = og[cu[b]:cu[b + 1]]
    g = dict(o=o_rows, boundary=bnd.cpu().numpy(), merge_log=ml.cpu().numpy(), cache=cache)
    r = dict(o=np.full((B, T, H, d), np.nan), boundary=np.zeros((B, H, T), np.uint8),
             merge_log=np.full((B, H, T), -1, np.int32), caches={})
    live = []
    for b, n in enumerate(lens):
        if n == 0:
            continue
        rb = oracle.forward(q[b:b + 1, :n], k[b:b + 1, :n], v[b:b + 1, :n], lam[b:b + 1, :n], tau=w.tau, C=w.C,
                            eps=w.eps, rms_eps=w.rms_eps)
        r["o"][b, :n] = rb["o"][0]
        r["boundary"][b, :, :n] = rb["boundary"][0]
        r["merge_log"][b, :, :n] = rb["merge_log"][0]
        for h in range(H):
            r["caches"][(b, h)] = rb["caches"][(0, h)]
            live.append((b, h))
    compare(w, g, r, streams=live)
    ex = cache.export()
    for b, n in enumerate(lens):
        np.testing.assert_array_equal(g["boundary"][b, :, n:], 0)
        np.testing.assert_array_equal(g["merge_log"][b, :, n:], -1)
        if n == 0:
            assert (ex["m"][b] == 0).all()
    # the padded layout with the same row lengths: the same values, bit for bit
    qp, kp, vp, lp = upload(w, q, k, v, lam)
    cache2 = dla.Cache(B, H, w.C, d, device=dev)
    sl = torch.tensor(lens, dtype=torch.int32, device=dev)  # must outlive the call
    p2 = dla.make_params(w.tau, w.C, w.eps, w.rms_eps, seq_lens=sl)
    o2 = torch.full((B, T, H, d), float("nan"), dtype=torch.float32, device=dev)
    bnd2 = torch.empty((B, H, T), dtype=torch.uint8, device=dev)
    ml2 = torch.empty((B, H, T), dtype=torch.int32, device=dev)
    dla.dla_forward(p2, qp, kp, vp, lp, o2, cache2, bnd2, ml2)
    assert dla.dla_sync_status() == 0
    o2n = o2.double().cpu().numpy()
    for b, n in enumerate(lens):
        np.testing.assert_array_equal(o_rows[b, :n], o2n[b, :n])
    np.testing.assert_array_equal(g["boundary"], bnd2.cpu().numpy())
    np.testing.assert_array_equal(g["merge_log"], ml2.cpu().numpy())
    ex2 = cache2.export()
    for key in ("m", "n"):
        np.testing.assert_array_equal(ex[key], ex2[key])


def test_packed_offsets_out_of_range_are_reported(monkeypatch):
    """Offsets that decrease, pass total_tokens or give a row longer than
    max_seqlen are found on the device: those rows are clamped into range
    (nothing is read past the packed tensors) and the call's status is 6."""
    w = W.get("standard", B=3, H=2, T=256)
    q, k, v, lam = _safe(w)
    dev = torch.device("cuda:0")
    total = 300
    qt, kt, vt, lt = upload(w, _pack(q, [256, 44]), _pack(k, [256, 44]), _pack(v, [256, 44]), _pack(lam, [256, 44]))
    d = kt.shape[-1]
    p = dla.make_params(w.tau, w.C, w.eps, w.rms_eps)
    for cu in ([0, 280, 300, 300], [0, 200, 150, 300], [0, 100, 300, 400]):
        o = torch.zeros((total, w.H, d), dtype=torch.float32, device=dev)
        cache = dla.Cache(w.B, w.H, w.C, d, device=dev)
        dla.dla_forward_varlen(p, torch.tensor(cu, dtype=torch.int32, device=dev), w.T, qt, kt, vt, lt, o, cache)
        assert dla.dla_sync_status() == 6, cu
        assert torch.isfinite(o).all()
    # a correct call on the same stream afterwards
    o = torch.zeros((total, w.H, d), dtype=torch.float32, device=dev)
    dla.dla_forward_varlen(p, torch.tensor([0, 256, 300, 300], dtype=torch.int32, device=dev), w.T, qt, kt, vt, lt,
                           o, dla.Cache(w.B, w.H, w.C, d, device=dev))
    assert dla.dla_sync_status() == 0


@pytest.mark.parametrize("sched", ["concurrent", "rounds", "serial"])
@pytest.mark.parametrize("case", ["standard_bf16", "regime_bf16", "long_churn_bf16", "many_streams_bf16"])
def test_forward_parity_tcgen05_scan(case, sched, monkeypatch):
    """DLA_SCAN=tc: the scan with the open state in tensor memory and its state
    builds and y contractions on tcgen05 (the opt-in scan) gives the oracle's
    results on every schedule."""
    monkeypatch.setenv("DLA_SCAN", "tc")
    monkeypatch.setenv("DLA_SCHEDULE", sched)
    name, ov = CASES[case]
    w = W.get(name, **ov)
    q, k, v, lam = _safe(w)
    g = run_gpu(w, q, k, v, lam)
    r = run_oracle(w, q, k, v, lam)
    compare(w, g, r)
    structural_checks(w, g, w.T)


def test_tcgen05_scan_small_workspace(monkeypatch):
    """DLA_SCAN=tc with the smallest workspace: one read-out interval per round,
    pools reset every round."""
    monkeypatch.setenv("DLA_SCAN", "tc")
    w = W.get("regime", B=1, H=2, T=1100)
    q, k, v, lam = _safe(w)
    p = dla.make_params(w.tau, w.C)
    nb = dla.dla_forward_min_workspace(p, w.B, w.T, w.H, w.d, w.d, dla.DLA_BF16, True)
    g = run_gpu(w, q, k, v, lam, ws_bytes=nb)
    r = run_oracle(w, q, k, v, lam)
    compare(w, g, r)
