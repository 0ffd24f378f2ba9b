"""Host-side checks of the C ABI: the library builds, loads and exports every
entry point include/dla.h declares, and argument errors come back as status
codes before anything touches a GPU (no compute calls here)."""
import ctypes
import os
import re

import pytest

import __graft_entry__
from paper_2606_10650_gb300 import dla

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    __graft_entry__.build()
    return dla.lib()


def _declared():
    src = open(os.path.join(ROOT, "include", "dla.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(dla_[a-z0-9_]+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = _declared()
    for n in ["dla_forward", "dla_decode_step", "dla_init_cache", "dla_forward_workspace", "dla_cache_bytes"]:
        assert n in names


def test_library_exports_every_declared_symbol(L):
    for n in _declared():
        assert hasattr(L, n), n
    assert set(_declared()) == set(dla.EXPORTED)
    assert L.dla_version() == 4


def _fake(addr=1 << 20):
    return ctypes.c_void_p(addr)


def _fwd(L, p, dt=dla.DLA_BF16, B=1, T=64, H=2, d=128, k=True, ws_bytes=1 << 40, ws=True, o=True):
    return L.dla_forward(ctypes.byref(p), dt, B, T, H, d, d, _fake(), _fake() if k else None, _fake(), None,
                         _fake() if o else None, None, None, None, _fake(1 << 24) if ws else None, ws_bytes, None)


def test_argument_errors_return_status_codes(L):
    p = dla.make_params(0.6, 8)
    assert _fwd(L, dla.make_params(0.6, 1)) == 1          # C < 2: Algorithm 2 needs a pair
    assert _fwd(L, dla.make_params(0.6, 257)) == 2        # beyond the built capacity
    assert _fwd(L, dla.make_params(0.6, 65), dt=dla.DLA_F32) == 2  # DLA(I) capacities: bf16 only
    assert _fwd(L, dla.make_params(0.6, 65), d=64) == 2           # ... and d = 128
    assert _fwd(L, dla.make_params(float("nan"), 8)) == 1
    assert _fwd(L, dla.make_params(0.6, 8, score_mode=3)) == 1
    assert _fwd(L, p, d=96) == 2
    assert _fwd(L, p, k=False) == 1
    assert _fwd(L, p, B=0) == 1
    assert _fwd(L, p, ws=False) == 3
    assert _fwd(L, p, ws_bytes=1024) == 3
    assert b"workspace" in L.dla_last_error()
    assert L.dla_status_string(3) == b"DLA_ERR_WORKSPACE"


def test_workspace_sizes_are_monotone(L):
    p = dla.make_params(0.6, 32)
    full = L.dla_forward_workspace(ctypes.byref(p), 2, 16384, 16, 128, 128, 0, 1)
    mini = L.dla_forward_min_workspace(ctypes.byref(p), 2, 16384, 16, 128, 128, 0, 1)
    none = L.dla_forward_workspace(ctypes.byref(p), 2, 16384, 16, 128, 128, 0, 0)
    assert 0 < none < mini <= full


def test_cache_carve_layout(L):
    nb = L.dla_cache_bytes(2, 3, 4, 64, 64)
    assert nb >= 2 * 3 * 4 * 64 * 64 * 4
    c = dla.dla_cache()
    assert L.dla_cache_carve(_fake(1 << 30), nb, 2, 3, 4, 64, 64, ctypes.byref(c)) == 0
    assert c.states == 1 << 30 and c.C == 4
    assert all(getattr(c, f) % 256 == 0 for f in ("states", "slot", "n", "ibar", "m"))
    assert L.dla_cache_carve(_fake(1 << 30), nb - 1, 2, 3, 4, 64, 64, ctypes.byref(c)) == 3


def test_host_buffer_entry_point_errors_and_workspace(L):
    p = dla.make_params(0.6, 32)
    fw = L.dla_forward_workspace(ctypes.byref(p), 2, 16384, 16, 128, 128, 0, 1)
    hw = L.dla_forward_host_workspace(ctypes.byref(p), 2, 16384, 16, 128, 128, 0, 1)
    io = 4 * 2 * 16384 * 16 * 128 * 2 + 2 * 16384 * 16 * 32 * 4  # q, k, v (bf16), o (fp32), lambda
    assert hw >= fw + io
    assert L.dla_forward_host_workspace(ctypes.byref(p), 0, 16, 1, 128, 128, 0, 1) == 0

    def fh(k=True, ws=True, ws_bytes=1 << 40):
        return L.dla_forward_host(ctypes.byref(p), 0, 1, 64, 2, 128, 128, _fake(), _fake() if k else None, _fake(),
                                  None, _fake(), None, None, None, _fake(1 << 24) if ws else None, ws_bytes, None)
    assert fh(k=False) == 1
    assert fh(ws=False) == 3
    assert fh(ws_bytes=1024) == 3
    assert b"workspace" in L.dla_last_error()
    # per-row lengths take device-resident inputs (the host copies move whole rows)
    q = dla.make_params(0.6, 32)
    q.seq_lens = 1 << 20
    st = L.dla_forward_host(ctypes.byref(q), 0, 1, 64, 2, 128, 128, _fake(), _fake(), _fake(), None, _fake(), None,
                            None, None, _fake(1 << 24), 1 << 40, None)
    assert st == 2 and b"seq_lens" in L.dla_last_error()


def test_params_layout_and_seq_lens_checks(L):
    p = dla.dla_params()
    p.seq_lens = 12345
    L.dla_default_params(ctypes.byref(p))
    assert p.tau == 0.6 and p.capacity == 30 and p.from_cache == 0 and not p.seq_lens
    q = dla.make_params(0.6, 8)
    q.seq_lens = (1 << 20) + 2  # not 4-byte aligned
    assert _fwd(L, q) == 1
    assert b"seq_lens" in L.dla_last_error()


def test_packed_batch_argument_errors(L):
    p = dla.make_params(0.6, 8)

    def fv(q=p, cu=True, total=100, ws_bytes=1 << 40, cu_addr=1 << 22):
        return L.dla_forward_varlen(ctypes.byref(q), dla.DLA_BF16, 2, 64, total, _fake(cu_addr) if cu else None, 2,
                                    128, 128, _fake(), _fake(), _fake(), None, _fake(), None, None, None,
                                    _fake(1 << 24), ws_bytes, None)
    assert fv(cu=False) == 1
    assert b"cu_seqlens" in L.dla_last_error()
    assert fv(cu_addr=(1 << 22) + 2) == 1          # offsets not 4-byte aligned
    assert fv(total=-1) == 2
    assert fv(total=1 << 31) == 2
    r = dla.make_params(0.6, 8)
    r.seq_lens = 1 << 21
    assert fv(q=r) == 1                             # lengths come from the offsets only
    assert b"seq_lens" in L.dla_last_error()
    assert fv(ws_bytes=1024) == 3


def test_backward_argument_errors(L):
    p = dla.make_params(0.6, 8)
    nb = L.dla_backward_workspace(ctypes.byref(p), 1, 64, 2, 128, 128, dla.DLA_BF16)
    assert nb >= 256 + 2 * 64 * 4 + 2 * 65 * 64 * 4
    assert L.dla_backward_workspace(ctypes.byref(p), 1, 64, 2, 128, 128, dla.DLA_F32) == 0

    def fb(q=p, dt=dla.DLA_BF16, d=128, k=True, ws_bytes=1 << 30, go=True):
        f = _fake
        return L.dla_backward(ctypes.byref(q), dt, 1, 64, 2, d, d, f(), f() if k else None, f(), None, f(), f(),
                              f() if go else None, f(), f(), f(), None, f(1 << 24), ws_bytes, None)
    assert fb(dt=dla.DLA_F32) == 2
    assert fb(d=96) == 2
    assert fb(k=False) == 1
    assert fb(go=False) == 1
    assert fb(ws_bytes=1024) == 3
    assert fb(q=dla.make_params(0.6, 8, from_cache=1)) == 2
    assert b"from_cache" in L.dla_last_error()


def test_kernel_kinds_match_the_header():
    """dla_timing_read fills DLA_K_COUNT entries; the binding names each kind."""
    src = open(os.path.join(ROOT, "include", "dla.h")).read()
    count = int(re.search(r"DLA_K_COUNT\s*=\s*(\d+)", src).group(1))
    assert count == len(dla.KERNELS)
    for i, name in enumerate(dla.KERNELS):
        assert re.search(rf"DLA_K_{name.upper()}\s*=\s*{i}\b", src) or (name == "readout" and "DLA_K_READOUT = 1" in src)
