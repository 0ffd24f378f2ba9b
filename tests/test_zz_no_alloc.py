"""dla_forward_noalloc: the forward pass for callers that cannot allocate
device memory (for example an engine plugin that is handed no workspace, or
code running while another thread captures a CUDA graph in global mode).  It
uses the library's static 64 MiB device scratch instead of a caller
workspace.  This file is collected last on purpose.

Checked through the C ABI against dla_forward (the entry point with a caller
workspace) on the same inputs, for two calls in a row with different inputs,
so that scratch left over from the first call cannot leak into the second."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2606_10650_gb300 import dla
from paper_2606_10650_gb300 import workloads as W
from parity_util import TOL

pytestmark = pytest.mark.gpu


def _inputs(seed, dev, T=900):
    w = W.get("regime", B=1, H=2, T=T)
    q, k, v, lam = W.host_batch(w, seed=seed, T=w.T)
    t = [W.to_device(x, w.dtype, dev) for x in (q, k, v)]
    t.append(torch.from_numpy(lam.astype(np.float32)).to(dev))
    return w, t


def _run(entry, w, t, dev):
    q, k, v, lam = t
    B, T, H, d = k.shape
    p = dla.make_params(w.tau, w.C, w.eps, w.rms_eps)
    cache = dla.Cache(B, H, w.C, d, device=dev)
    o = torch.full((B, T, H, d), float("nan"), device=dev)
    bnd = torch.zeros((B, H, T), dtype=torch.uint8, device=dev)
    ml = torch.zeros((B, H, T), dtype=torch.int32, device=dev)
    if entry == "noalloc":
        dla.dla_forward_noalloc(p, q, k, v, lam, o, cache, bnd, ml)
    else:
        dla.dla_forward(p, q, k, v, lam, o, cache, bnd, ml)
    # the call's device status (its workspace word is inside the library's
    # static array, so it is read through the stream's status word)
    assert dla.dla_sync_status() == 0
    return o.cpu(), bnd.cpu(), ml.cpu(), cache.export()


def test_noalloc_matches_dla_forward_two_calls_in_a_row():
    dev = torch.device("cuda:0")
    for seed in (11, 12):  # two calls in a row, different inputs
        w, t = _inputs(seed, dev)
        o_ref, b_ref, m_ref, c_ref = _run("workspace", w, t, dev)
        o, b, m, c = _run("noalloc", w, t, dev)
        assert torch.equal(b, b_ref) and torch.equal(m, m_ref)
        assert torch.isfinite(o).all()
        assert (o - o_ref).abs().max().item() <= TOL[w.dtype]
        assert torch.equal(c["m"], c_ref["m"]) and torch.equal(c["n"], c_ref["n"])
        assert (c["states"] - c_ref["states"]).abs().max().item() <= TOL[w.dtype]


def test_noalloc_with_a_plan_limited_by_its_scratch():
    """A sequence whose preferred workspace exceeds the 64 MiB scratch (but whose
    smallest one fits) runs with fewer rounds of snapshots; results equal
    dla_forward's with its preferred workspace."""
    dev = torch.device("cuda:0")
    w, t = _inputs(13, dev, T=6000)
    p = dla.make_params(w.tau, w.C, w.eps, w.rms_eps)
    B, T, H, d = t[1].shape
    assert dla.dla_forward_workspace(p, B, T, H, d, d, dla.DLA_BF16, True) > (64 << 20)
    assert dla.dla_forward_min_workspace(p, B, T, H, d, d, dla.DLA_BF16, True) <= (64 << 20)
    o_ref, b_ref, m_ref, c_ref = _run("workspace", w, t, dev)
    o, b, m, c = _run("noalloc", w, t, dev)
    assert torch.equal(b, b_ref) and torch.equal(m, m_ref)
    assert (o - o_ref).abs().max().item() <= TOL[w.dtype]
    assert torch.equal(c["m"], c_ref["m"]) and torch.equal(c["n"], c_ref["n"])


def test_noalloc_replayed_from_a_captured_graph():
    """dla_forward_noalloc captured in a CUDA graph (after a first call on the
    thread, which creates the library's internal streams and events), then the
    graph replayed on other inputs copied into the captured buffers: trace,
    cache and outputs equal dla_forward's on those inputs, and the capture
    stream's status word reads 0."""
    dev = torch.device("cuda:0")
    w, t1 = _inputs(21, dev)
    _, t2 = _inputs(22, dev)
    q, k, v, lam = (x.clone() for x in t1)
    B, T, H, d = k.shape
    p = dla.make_params(w.tau, w.C, w.eps, w.rms_eps)
    cache = dla.Cache(B, H, w.C, d, device=dev)
    o = torch.full((B, T, H, d), float("nan"), device=dev)
    bnd = torch.zeros((B, H, T), dtype=torch.uint8, device=dev)
    ml = torch.zeros((B, H, T), dtype=torch.int32, device=dev)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        dla.dla_forward_noalloc(p, q, k, v, lam, o, cache, bnd, ml, stream=s)
    assert dla.dla_sync_status(s) == 0
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        dla.dla_forward_noalloc(p, q, k, v, lam, o, cache, bnd, ml, stream=s)
    for dst, src in zip((q, k, v, lam), t2):
        dst.copy_(src)
    o.fill_(float("nan"))
    torch.cuda.synchronize()
    g.replay()
    torch.cuda.synchronize()
    assert dla.dla_sync_status(s) == 0
    o_ref, b_ref, m_ref, c_ref = _run("workspace", w, t2, dev)
    assert torch.equal(bnd.cpu(), b_ref) and torch.equal(ml.cpu(), m_ref)
    assert torch.isfinite(o).all()
    assert (o.cpu() - o_ref).abs().max().item() <= TOL[w.dtype]
    c = cache.export()
    assert torch.equal(c["m"], c_ref["m"]) and torch.equal(c["n"], c_ref["n"])


def test_noalloc_rejects_calls_beyond_its_scratch():
    """Without a caller cache the cache itself must live in the scratch; for a
    large batch that exceeds the 64 MiB limit and the call is refused with a
    message naming it, before anything is launched."""
    L = dla.lib()
    p = dla.make_params(1.3, 64)
    fake = ctypes.c_void_p(1 << 24)
    st = L.dla_forward_noalloc(ctypes.byref(p), dla.DLA_BF16, 8, 4096, 32, 128, 128, fake, fake, fake, None, fake,
                               None, None, None, None)
    assert st == 3
    assert b"static scratch" in L.dla_last_error()
