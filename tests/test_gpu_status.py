"""Failure detection on the GPU without a GPU fault: device-side failures come
back through the stream's status word (dla_sync_status), every wait in the
kernels is bounded, and the library stays usable after a failed call.

The failures are made on the host: a debugging knob shortens the kernels' wait
limit to a few milliseconds, and another makes dla_forward_host report only its
first input piece as arrived, so the scan's bounded wait for a later piece runs
out (status 5, DLA_ERR_TIMEOUT).  A cache whose live count is out of range is
clamped by the decode kernel's own check and reported (status 6,
DLA_ERR_DEVICE_CHECK).  Nothing here traps, faults or hangs a kernel."""
import numpy as np
import pytest
import torch

from paper_2606_10650_gb300 import dla
from paper_2606_10650_gb300 import workloads as W
from parity_util import compare, run_oracle, structural_checks, upload
from safe_inputs import safe_batch

pytestmark = pytest.mark.gpu


def _host_forward(w, q, k, v, lam):
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
    return ws, dict(o=oh, boundary=bnd, merge_log=ml, cache=cache)


def test_sync_status_is_ok_after_good_calls():
    w = W.get("standard", B=1, H=2, T=300)
    q, k, v, lam, _ = safe_batch(w)
    assert dla.dla_sync_status() == 0  # nothing pending
    ws, _ = _host_forward(w, q, k, v, lam)
    assert dla.dla_sync_status() == 0
    assert dla.workspace_status(ws) == 0


@pytest.mark.timeout(300)
def test_bounded_wait_runs_out_and_the_next_call_is_correct(monkeypatch):
    """The scan waits (bounded) for input pieces that are never reported: the
    call ends with status 5 on its stream and in its workspace, no kernel hangs,
    and the following normal call on the same inputs matches the oracle."""
    w = W.get("regime", B=1, H=2, T=2500)
    q, k, v, lam, _ = safe_batch(w)
    monkeypatch.delenv("DLA_SCHEDULE", raising=False)  # the concurrent schedule streams the inputs
    monkeypatch.setenv("DLA_DEBUG_WAIT_MS", "20")
    monkeypatch.setenv("DLA_DEBUG_WITHHOLD_PIECES", "1")
    ws, _ = _host_forward(w, q, k, v, lam)
    st = dla.dla_sync_status()
    assert st == 5, f"expected DLA_ERR_TIMEOUT, got {st}"
    assert dla.workspace_status(ws) == 5
    assert dla.dla_sync_status() == 0  # read and cleared
    monkeypatch.delenv("DLA_DEBUG_WAIT_MS")
    monkeypatch.delenv("DLA_DEBUG_WITHHOLD_PIECES")
    ws, g = _host_forward(w, q, k, v, lam)
    assert dla.dla_sync_status() == 0
    assert dla.workspace_status(ws) == 0
    g = dict(o=g["o"].double().numpy(), boundary=g["boundary"].cpu().numpy(), merge_log=g["merge_log"].cpu().numpy(),
             cache=g["cache"])
    r = run_oracle(w, q, k, v, lam)
    compare(w, g, r)
    structural_checks(w, g, w.T)


def test_decode_reports_an_inconsistent_cache(monkeypatch):
    """A live count beyond the capacity is clamped by the decode kernel and
    reported as DLA_ERR_DEVICE_CHECK through the stream's status word."""
    dev = torch.device("cuda:0")
    B, H, C, d = 2, 2, 4, 128
    cache = dla.Cache(B, H, C, d, device=dev)
    dla.dla_init_cache(cache)
    cache.view("states").zero_()
    m = cache.view("m")
    m.fill_(2)
    m[1, 0] = C + 5  # out of range
    cache.view("n").fill_(1)
    cache.view("ibar").fill_(1.0)
    p = dla.make_params(1.4, C)
    x = (torch.randn((B, H, d), device=dev) / np.sqrt(d)).to(torch.bfloat16)
    o = torch.empty((B, H, d), dtype=torch.float32, device=dev)
    dla.dla_decode_step(p, cache, x, x.clone(), x.clone(), None, o)
    assert dla.dla_sync_status() == 6
    m[1, 0] = 2
    dla.dla_decode_step(p, cache, x, x.clone(), x.clone(), None, o)
    assert dla.dla_sync_status() == 0
