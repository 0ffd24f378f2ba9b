"""Helpers of the GPU parity tests: run the CUDA path through the C ABI and the
fp64 oracle on the same seeded inputs and compare them.

Bar: boundary flags, merge indices, live-state counts,
token counts and logical slot order bit-exact; outputs and states within
max-abs 2e-2 for bf16 inputs and 1e-4 for fp32 inputs; summed scores Ibar
within a relative error well below the tie margin of the input generator.
"""
from __future__ import annotations

import numpy as np
import torch

import oracle
from paper_2606_10650_gb300 import dla
from paper_2606_10650_gb300 import workloads as W

TOL = {"bf16": 2e-2, "f32": 1e-4}
IBAR_RTOL = 1e-6  # tenth of the 1e-5 tie margin of the safe-input generator


def device():
    return torch.device("cuda:0")


def upload(w, q, k, v, lam):
    dev = device()
    qt = W.to_device(q, w.dtype, dev)
    kt = W.to_device(k, w.dtype, dev)
    vt = W.to_device(v, w.dtype, dev)
    lt = None if lam is None else torch.from_numpy(np.ascontiguousarray(lam, dtype=np.float32)).to(dev)
    return qt, kt, vt, lt


def run_gpu(w, q, k, v, lam, *, want_o=True, score_mode=0, out_dtype=torch.float32, ws_bytes=None,
            cache=None, from_cache=False, tensors=None):
    """dla_forward through the C ABI; returns numpy results and the cache."""
    dev = device()
    qt, kt, vt, lt = tensors if tensors is not None else upload(w, q, k, v, lam)
    B, T, H, d = kt.shape
    if cache is None:
        cache = dla.Cache(B, H, w.C, d, device=dev)
    od = dla.DLA_BF16 if out_dtype == torch.bfloat16 else dla.DLA_F32
    p = dla.make_params(w.tau, w.C, w.eps, w.rms_eps, score_mode, od, int(from_cache))
    o = torch.full((B, T, H, d), float("nan"), dtype=out_dtype, device=dev) if want_o else None
    bnd = torch.full((B, H, T), 7, dtype=torch.uint8, device=dev)
    ml = torch.full((B, H, T), -7, dtype=torch.int32, device=dev)
    ws = None
    if ws_bytes is not None:
        buf = torch.empty(ws_bytes + 256, dtype=torch.uint8, device=dev)
        ws = (buf, (buf.data_ptr() + 255) // 256 * 256, ws_bytes)
    ws = dla.dla_forward(p, qt if want_o else None, kt, vt, lt, o, cache, bnd, ml, workspace=ws)
    torch.cuda.synchronize()
    assert dla.workspace_status(ws) == 0, "device status word reports a failure"
    return dict(o=None if o is None else o.double().cpu().numpy(), boundary=bnd.cpu().numpy(),
                merge_log=ml.cpu().numpy(), cache=cache)


def run_oracle(w, q, k, v, lam, *, want_o=None, streams=None, score_mode=0):
    return oracle.forward(q, k, v, lam, tau=w.tau, C=w.C, eps=w.eps, rms_eps=w.rms_eps, score_mode=score_mode,
                          want_o=want_o, streams=streams)


def compare(w, g, r, streams=None, tol=None, check_cache=True, report=None):
    """Bit-exact decisions, outputs/states within tolerance (numpy inputs)."""
    tol = TOL[w.dtype] if tol is None else tol
    B, H = g["boundary"].shape[:2]
    streams = [(b, h) for b in range(B) for h in range(H)] if streams is None else streams
    ex = g["cache"].export() if check_cache else None
    worst_o = worst_s = worst_ib = 0.0
    for (b, h) in streams:
        np.testing.assert_array_equal(g["boundary"][b, h], r["boundary"][b, h], err_msg=f"boundary ({b},{h})")
        np.testing.assert_array_equal(g["merge_log"][b, h], r["merge_log"][b, h], err_msg=f"merge_log ({b},{h})")
        if g["o"] is not None:
            ro = r["o"][b, :, h]
            mask = ~np.isnan(ro[:, 0])
            err = np.abs(g["o"][b, :, h][mask] - ro[mask])
            e = float(err.max()) if err.size else 0.0
            worst_o = max(worst_o, e)
            assert e <= tol, f"output ({b},{h}) max-abs {e} > {tol}"
        if check_cache:
            rc = r["caches"][(b, h)]
            m = rc["m"]
            assert int(ex["m"][b, h]) == m
            np.testing.assert_array_equal(ex["n"][b, h, :m].numpy(), rc["n"])
            gs = ex["states"][b, h, :m].double().numpy()
            es = float(np.abs(gs - rc["states"]).max())
            worst_s = max(worst_s, es)
            assert es <= tol, f"states ({b},{h}) max-abs {es} > {tol}"
            ib = ex["ibar"][b, h, :m].numpy()
            rel = float(np.max(np.abs(ib - rc["ibar"]) / np.maximum(np.abs(rc["ibar"]), 1e-30)))
            worst_ib = max(worst_ib, rel)
            assert rel <= IBAR_RTOL, f"Ibar ({b},{h}) rel err {rel}"
            slot = ex["slot"][b, h, :m].numpy()
            assert sorted(slot.tolist()) == list(range(m)), "slot map must permute 0..m-1"
    if report is not None:
        report.update(o=worst_o, states=worst_s, ibar_rel=worst_ib)
    return worst_o, worst_s, worst_ib


def structural_checks(w, g, T):
    """Properties that hold for every stream at any size: m <= C, sum n = T,
    slot map is a permutation, boundaries - merges = m, merges only at
    boundaries, merge indices within 0..C-2."""
    ex = g["cache"].export()
    bnd, ml = g["boundary"], g["merge_log"]
    B, H = bnd.shape[:2]
    for b in range(B):
        for h in range(H):
            m = int(ex["m"][b, h])
            assert 1 <= m <= w.C
            assert int(ex["n"][b, h, :m].sum()) == T
            assert sorted(ex["slot"][b, h, :m].tolist()) == list(range(m))
            nb = int(bnd[b, h].sum())
            nm = int((ml[b, h] >= 0).sum())
            assert nb - nm == m
            assert np.all(bnd[b, h][ml[b, h] >= 0] == 1)
            assert ml[b, h].max() <= w.C - 2 and ml[b, h].min() >= -1
