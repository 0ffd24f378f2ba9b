"""Thin ctypes binding of libdla.so (include/dla.h), same entry-point names.

Argument marshalling only: torch tensors are passed as raw device pointers and
the current CUDA stream; every step of the computation runs in the library's
CUDA kernels.  There is no CPU fallback: without the built library every call
raises.
"""
from __future__ import annotations

import ctypes
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libdla.so")

DLA_BF16, DLA_F32 = 0, 1
STATUS = {0: "DLA_OK", 1: "DLA_ERR_INVALID_ARG", 2: "DLA_ERR_UNSUPPORTED", 3: "DLA_ERR_WORKSPACE",
          4: "DLA_ERR_CUDA", 5: "DLA_ERR_TIMEOUT", 6: "DLA_ERR_DEVICE_CHECK"}

EXPORTED = ["dla_default_params", "dla_cache_bytes", "dla_cache_carve", "dla_init_cache",
            "dla_forward_workspace", "dla_forward_min_workspace", "dla_forward", "dla_decode_step",
            "dla_last_error", "dla_status_string", "dla_version", "dla_timing_enable", "dla_timing_read", "dla_forward_noalloc",
            "dla_forward_host_workspace", "dla_forward_host", "dla_sync_status", "dla_forward_varlen",
            "dla_backward_workspace", "dla_backward"]
KERNELS = ["scan", "readout", "decode", "init", "gram", "gate", "status", "backward"]


class DLAError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__(f"{STATUS.get(status, status)}: {msg}")
        self.status = status


class dla_params(ctypes.Structure):
    _fields_ = [("tau", ctypes.c_double), ("eps", ctypes.c_double), ("rms_eps", ctypes.c_double),
                ("capacity", ctypes.c_int), ("score_mode", ctypes.c_int), ("out_dtype", ctypes.c_int),
                ("from_cache", ctypes.c_int), ("seq_lens", ctypes.c_void_p)]


class dla_cache(ctypes.Structure):
    _fields_ = [("states", ctypes.c_void_p), ("slot", ctypes.c_void_p), ("n", ctypes.c_void_p),
                ("ibar", ctypes.c_void_p), ("m", ctypes.c_void_p), ("B", ctypes.c_int), ("H", ctypes.c_int),
                ("C", ctypes.c_int), ("dk", ctypes.c_int), ("dv", ctypes.c_int)]


_LIB = None


def lib():
    """Load libdla.so (built by paper_2606_10650_gb300.build); raises if absent."""
    global _LIB
    if _LIB is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"libdla.so not built ({LIB_PATH}); run __graft_entry__.build()")
        L = ctypes.CDLL(LIB_PATH)
        vp, ci, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t
        P = ctypes.POINTER(dla_params)
        Cp = ctypes.POINTER(dla_cache)
        L.dla_default_params.argtypes = [P]
        L.dla_cache_bytes.restype = sz
        L.dla_cache_bytes.argtypes = [ci] * 5
        L.dla_cache_carve.argtypes = [vp, sz, ci, ci, ci, ci, ci, Cp]
        L.dla_init_cache.argtypes = [Cp, vp]
        L.dla_forward_workspace.restype = sz
        L.dla_forward_workspace.argtypes = [P, ci, ci, ci, ci, ci, ci, ci]
        L.dla_forward_min_workspace.restype = sz
        L.dla_forward_min_workspace.argtypes = [P, ci, ci, ci, ci, ci, ci, ci]
        L.dla_forward.argtypes = [P, ci, ci, ci, ci, ci, ci, vp, vp, vp, vp, vp, Cp, vp, vp, vp, sz, vp]
        L.dla_decode_step.argtypes = [P, Cp, ci, vp, vp, vp, vp, vp, vp, vp, vp]
        L.dla_last_error.restype = ctypes.c_char_p
        L.dla_status_string.restype = ctypes.c_char_p
        L.dla_status_string.argtypes = [ci]
        L.dla_version.restype = ci
        L.dla_forward_noalloc.argtypes = [P, ci, ci, ci, ci, ci, ci, vp, vp, vp, vp, vp, Cp, vp, vp, vp]
        L.dla_forward_host_workspace.restype = sz
        L.dla_forward_host_workspace.argtypes = [P, ci, ci, ci, ci, ci, ci, ci]
        L.dla_forward_host.argtypes = [P, ci, ci, ci, ci, ci, ci, vp, vp, vp, vp, vp, Cp, vp, vp, vp, sz, vp]
        L.dla_sync_status.argtypes = [vp]
        L.dla_backward_workspace.restype = sz
        L.dla_backward_workspace.argtypes = [P, ci, ci, ci, ci, ci, ci]
        L.dla_backward.argtypes = [P, ci, ci, ci, ci, ci, ci, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp]
        L.dla_forward_varlen.argtypes = [P, ci, ci, ci, ctypes.c_longlong, vp, ci, ci, ci, vp, vp, vp, vp, vp, Cp, vp,
                                         vp, vp, sz, vp]
        L.dla_timing_enable.argtypes = [ci]
        L.dla_timing_read.argtypes = [ctypes.POINTER(ci), ctypes.POINTER(ctypes.c_double), ci]
        _LIB = L
    return _LIB


def _check(status):
    if status != 0:
        raise DLAError(status, lib().dla_last_error().decode())


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _dtype_code(t):
    if t.dtype == torch.bfloat16:
        return DLA_BF16
    if t.dtype == torch.float32:
        return DLA_F32
    raise TypeError(f"unsupported input dtype {t.dtype} (bf16 or fp32)")


def make_params(tau, capacity, eps=1e-6, rms_eps=1e-6, score_mode=0, out_dtype=DLA_F32, from_cache=0,
                seq_lens=None):
    """seq_lens: None, or an int32 CUDA tensor [B] of per-row lengths (ragged
    batches in the padded layout; it must outlive the calls that use the params)."""
    return dla_params(float(tau), float(eps), float(rms_eps), int(capacity), int(score_mode), int(out_dtype),
                      int(from_cache), None if seq_lens is None else seq_lens.data_ptr())


def dla_default_params():
    p = dla_params()
    lib().dla_default_params(ctypes.byref(p))
    return p


def dla_timing_enable(enable=True):
    _check(lib().dla_timing_enable(int(bool(enable))))


def dla_timing_read(reset=True):
    """{kernel kind: (launches, summed ms)} of the launches recorded since the
    last reset (see dla_timing_enable)."""
    k = len(KERNELS)
    n = (ctypes.c_int * k)()
    ms = (ctypes.c_double * k)()
    _check(lib().dla_timing_read(n, ms, int(bool(reset))))
    return {KERNELS[i]: (n[i], ms[i]) for i in range(k)}


def dla_cache_bytes(B, H, C, dk, dv):
    return lib().dla_cache_bytes(B, H, C, dk, dv)


def dla_forward_workspace(params, B, T, H, dk, dv, in_dtype, with_output=True):
    return lib().dla_forward_workspace(ctypes.byref(params), B, T, H, dk, dv, in_dtype, int(bool(with_output)))


def dla_forward_host_workspace(params, B, T, H, dk, dv, in_dtype, with_output=True):
    return lib().dla_forward_host_workspace(ctypes.byref(params), B, T, H, dk, dv, in_dtype, int(bool(with_output)))


def dla_forward_min_workspace(params, B, T, H, dk, dv, in_dtype, with_output=True):
    return lib().dla_forward_min_workspace(ctypes.byref(params), B, T, H, dk, dv, in_dtype, int(bool(with_output)))


class Cache:
    """A device cache for B x H streams carved from one torch allocation."""

    def __init__(self, B, H, C, d, device="cuda", buffer=None):
        self.B, self.H, self.C, self.d = B, H, C, d
        nbytes = dla_cache_bytes(B, H, C, d, d)
        self.buf = buffer if buffer is not None else torch.empty(nbytes + 256, dtype=torch.uint8, device=device)
        base = (self.buf.data_ptr() + 255) // 256 * 256
        self.c = dla_cache()
        _check(lib().dla_cache_carve(ctypes.c_void_p(base), nbytes, B, H, C, d, d, ctypes.byref(self.c)))
        self._base = base

    def sub(self, b0, nb):
        """A cache object over batch rows [b0, b0 + nb) of this cache (no copy)."""
        c = dla_cache()
        B, H, C, d = self.B, self.H, self.C, self.d
        c.states = self.c.states + b0 * H * C * d * d * 4
        c.slot = self.c.slot + b0 * H * C * 4
        c.n = self.c.n + b0 * H * C * 4
        c.ibar = self.c.ibar + b0 * H * C * 8
        c.m = self.c.m + b0 * H * 4
        c.B, c.H, c.C, c.dk, c.dv = nb, H, C, d, d
        view = object.__new__(Cache)
        view.B, view.H, view.C, view.d, view.buf, view.c, view._base = nb, H, C, d, self.buf, c, None
        return view

    def view(self, name):
        """torch view of one cache array (states [B,H,C,d,d], slot/n [B,H,C],
        ibar [B,H,C] float64, m [B,H])."""
        B, H, C, d = self.B, self.H, self.C, self.d
        spec = {"states": (torch.float32, (B, H, C, d, d)), "slot": (torch.int32, (B, H, C)),
                "n": (torch.int32, (B, H, C)), "ibar": (torch.float64, (B, H, C)), "m": (torch.int32, (B, H))}
        dt, shape = spec[name]
        off = getattr(self.c, name) - self.buf.data_ptr()
        numel = 1
        for s in shape:
            numel *= s
        nbytes = numel * torch.tensor([], dtype=dt).element_size()
        return self.buf[off: off + nbytes].view(dt).view(shape)

    def export(self):
        """Host copy in logical order: states [B,H,C,d,d] (slots >= m zero),
        n, ibar, m."""
        m = self.view("m").cpu()
        slot = self.view("slot").cpu().long()
        states = self.view("states").cpu()
        n = self.view("n").cpu()
        ibar = self.view("ibar").cpu()
        B, H, C = self.B, self.H, self.C
        lg = torch.zeros_like(states)
        for b in range(B):
            for h in range(H):
                mm = int(m[b, h])
                if mm:
                    lg[b, h, :mm] = states[b, h, slot[b, h, :mm]]
        return dict(states=lg, n=n, ibar=ibar, m=m, slot=slot)


def dla_init_cache(cache: Cache, stream=None):
    _check(lib().dla_init_cache(ctypes.byref(cache.c), _stream(stream)))


def _aligned_workspace(nbytes, device):
    buf = torch.empty(nbytes + 256, dtype=torch.uint8, device=device)
    base = (buf.data_ptr() + 255) // 256 * 256
    return buf, base


def dla_forward(params, q, k, v, lam=None, o=None, cache=None, boundary=None, merge_log=None,
                workspace=None, stream=None):
    """Raw call of dla_forward.  q, k, v: [B, T, H, d] contiguous CUDA tensors
    (bf16 or fp32); lam [B, T, H, C] fp32 or None; o [B, T, H, d] (fp32 or bf16
    as params.out_dtype) or None; cache: Cache or None; boundary [B, H, T]
    uint8, merge_log [B, H, T] int32 or None; workspace: (tensor, base_ptr,
    nbytes) or None (allocated here)."""
    B, T, H, d = k.shape
    dt = _dtype_code(k)
    for t in (q, k, v, lam, o, boundary, merge_log):
        if t is not None and not t.is_contiguous():
            raise ValueError("tensors must be contiguous")
    if workspace is None:
        nb = dla_forward_workspace(params, B, T, H, d, d, dt, o is not None)
        buf, base = _aligned_workspace(nb, k.device)
        workspace = (buf, base, nb)
    _, base, nb = workspace
    st = lib().dla_forward(ctypes.byref(params), dt, B, T, H, d, d, _ptr(q), _ptr(k), _ptr(v), _ptr(lam), _ptr(o),
                           ctypes.byref(cache.c) if cache is not None else None, _ptr(boundary), _ptr(merge_log),
                           ctypes.c_void_p(base), nb, _stream(stream))
    _check(st)
    return workspace


def dla_forward_varlen(params, cu_seqlens, max_seqlen, q, k, v, lam=None, o=None, cache=None, boundary=None,
                       merge_log=None, workspace=None, stream=None):
    """Raw call of dla_forward_varlen (a packed batch).  cu_seqlens: int32 CUDA
    tensor [B + 1]; q, k, v: [total_tokens, H, d] contiguous CUDA tensors (bf16
    or fp32); lam [total_tokens, H, C] fp32 or None; o [total_tokens, H, d] or
    None; boundary [B, H, max_seqlen] uint8, merge_log [B, H, max_seqlen] int32
    or None; workspace as for dla_forward (sized with T = max_seqlen)."""
    Ttot, H, d = k.shape
    B = cu_seqlens.numel() - 1
    dt = _dtype_code(k)
    if cu_seqlens.dtype != torch.int32:
        raise ValueError("cu_seqlens must be int32")
    for t in (q, k, v, lam, o, boundary, merge_log, cu_seqlens):
        if t is not None and not t.is_contiguous():
            raise ValueError("tensors must be contiguous")
    if workspace is None:
        nb = dla_forward_workspace(params, B, max_seqlen, H, d, d, dt, o is not None)
        buf, base = _aligned_workspace(nb, k.device)
        workspace = (buf, base, nb)
    _, base, nb = workspace
    st = lib().dla_forward_varlen(ctypes.byref(params), dt, B, int(max_seqlen), int(Ttot), _ptr(cu_seqlens), H, d, d,
                                  _ptr(q), _ptr(k), _ptr(v), _ptr(lam), _ptr(o),
                                  ctypes.byref(cache.c) if cache is not None else None, _ptr(boundary),
                                  _ptr(merge_log), ctypes.c_void_p(base), nb, _stream(stream))
    _check(st)
    return workspace


def dla_backward(params, q, k, v, lam, boundary, merge_log, grad_o, grad_q, grad_k, grad_v, grad_lam=None,
                 workspace=None, stream=None):
    """Raw call of dla_backward: q, k, v [B, T, H, d] bf16; lam [B, T, H, C] fp32
    or None; boundary [B, H, T] uint8 and merge_log [B, H, T] int32 from the
    forward call; grad_o and the outputs grad_q, grad_k, grad_v [B, T, H, d]
    fp32; grad_lam [B, T, H, C] fp32 or None (all contiguous CUDA tensors)."""
    B, T, H, d = k.shape
    dt = _dtype_code(k)
    for t in (q, k, v, lam, boundary, merge_log, grad_o, grad_q, grad_k, grad_v, grad_lam):
        if t is not None and not t.is_contiguous():
            raise ValueError("tensors must be contiguous")
    if workspace is None:
        nb = lib().dla_backward_workspace(ctypes.byref(params), B, T, H, d, d, dt)
        if nb == 0:
            raise DLAError(1, "dla_backward_workspace: unsupported arguments")
        buf, base = _aligned_workspace(nb, k.device)
        workspace = (buf, base, nb)
    _, base, nb = workspace
    st = lib().dla_backward(ctypes.byref(params), dt, B, T, H, d, d, _ptr(q), _ptr(k), _ptr(v), _ptr(lam),
                            _ptr(boundary), _ptr(merge_log), _ptr(grad_o), _ptr(grad_q), _ptr(grad_k), _ptr(grad_v),
                            _ptr(grad_lam), ctypes.c_void_p(base), nb, _stream(stream))
    _check(st)
    return workspace


def backward(q, k, v, lam, boundary, merge_log, grad_o, *, capacity, want_lam=True, stream=None):
    """Convenience gradients of the read-out (decisions of the forward call held
    fixed): allocates the outputs with torch.  Returns dict(dq, dk, dv, dlam)."""
    B, T, H, d = k.shape
    dev = k.device
    p = make_params(0.0, capacity)
    dq, dk, dv = (torch.empty((B, T, H, d), dtype=torch.float32, device=dev) for _ in range(3))
    dlam = torch.empty((B, T, H, capacity), dtype=torch.float32, device=dev) if want_lam else None
    dla_backward(p, q, k, v, lam, boundary, merge_log, grad_o, dq, dk, dv, dlam, stream=stream)
    return dict(dq=dq, dk=dk, dv=dv, dlam=dlam)


def dla_forward_noalloc(params, q, k, v, lam=None, o=None, cache=None, boundary=None, merge_log=None, stream=None):
    """dla_forward without a workspace argument, for callers that cannot
    allocate: the library's 64 MiB static device scratch is used instead (see
    include/dla.h).  Same tensor conventions as dla_forward."""
    B, T, H, d = k.shape
    st = lib().dla_forward_noalloc(ctypes.byref(params), _dtype_code(k), B, T, H, d, d, _ptr(q), _ptr(k), _ptr(v),
                                   _ptr(lam), _ptr(o), ctypes.byref(cache.c) if cache is not None else None,
                                   _ptr(boundary), _ptr(merge_log), _stream(stream))
    _check(st)


def dla_forward_host(params, q, k, v, lam=None, o=None, cache=None, boundary=None, merge_log=None,
                     workspace=None, device=None, stream=None):
    """Raw call of dla_forward_host: q, k, v, lam, o are contiguous CPU tensors
    (page-locked for asynchronous copies), same shapes and dtypes as for
    dla_forward; cache, boundary, merge_log are device tensors or None;
    workspace: (tensor, base_ptr, nbytes) on `device` or None (allocated here).
    Only enqueues: o is filled once the stream has run the call."""
    B, T, H, d = k.shape
    dt = _dtype_code(k)
    for t in (q, k, v, lam, o):
        if t is not None and (not t.is_contiguous() or t.is_cuda):
            raise ValueError("q, k, v, lam, o must be contiguous host tensors")
    if workspace is None:
        dev = torch.device(device) if device is not None else torch.device("cuda", torch.cuda.current_device())
        nb = dla_forward_host_workspace(params, B, T, H, d, d, dt, o is not None)
        buf, base = _aligned_workspace(nb, dev)
        workspace = (buf, base, nb)
    _, base, nb = workspace
    st = lib().dla_forward_host(ctypes.byref(params), dt, B, T, H, d, d, _ptr(q), _ptr(k), _ptr(v), _ptr(lam),
                                _ptr(o), ctypes.byref(cache.c) if cache is not None else None, _ptr(boundary),
                                _ptr(merge_log), ctypes.c_void_p(base), nb, _stream(stream))
    _check(st)
    return workspace


def dla_sync_status(stream=None):
    """Waits for the stream and returns the device status of the library's
    calls on it since the last read (0 ok, 5 a bounded wait gave up, 6 a device
    check failed), clearing it.  Returns the code; does not raise for 5 or 6."""
    st = lib().dla_sync_status(_stream(stream))
    if st not in (0, 5, 6):
        _check(st)
    return st


def workspace_status(workspace):
    """Device status word of the last dla_forward on this workspace (call after
    synchronising): 0 ok, 5 timeout, 6 device check."""
    buf, base, _ = workspace
    off = base - buf.data_ptr()
    return int(buf[off: off + 4].view(torch.int32).item())


def dla_decode_step(params, cache: Cache, q, k, v, lam=None, o=None, boundary=None, merge_idx=None, stream=None):
    """Raw call of dla_decode_step.  q, k, v: [B, H, d]; lam [B, H, C] or None;
    o [B, H, d]; boundary [B, H] uint8; merge_idx [B, H] int32."""
    dt = _dtype_code(k)
    st = lib().dla_decode_step(ctypes.byref(params), ctypes.byref(cache.c), dt, _ptr(q), _ptr(k), _ptr(v), _ptr(lam),
                               _ptr(o), _ptr(boundary), _ptr(merge_idx), _stream(stream))
    _check(st)


def forward(q, k, v, lam=None, *, tau, capacity, eps=1e-6, rms_eps=1e-6, score_mode=0, out_dtype=torch.float32,
            want_o=True, cache=None, from_cache=False, stream=None):
    """Convenience prefill: allocates o, the trace and the workspace with
    torch and calls dla_forward.  Returns dict(o, boundary, merge_log)."""
    B, T, H, d = k.shape
    od = DLA_BF16 if out_dtype == torch.bfloat16 else DLA_F32
    p = make_params(tau, capacity, eps, rms_eps, score_mode, od, int(bool(from_cache)))
    dev = k.device
    o = torch.empty((B, T, H, d), dtype=out_dtype, device=dev) if want_o else None
    bnd = torch.empty((B, H, T), dtype=torch.uint8, device=dev)
    ml = torch.empty((B, H, T), dtype=torch.int32, device=dev)
    dla_forward(p, q, k, v, lam, o, cache, bnd, ml, stream=stream)
    return dict(o=o, boundary=bnd, merge_log=ml)
