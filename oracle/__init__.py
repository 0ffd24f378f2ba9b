"""fp64 CPU oracle of Dynamic Linear Attention (arXiv 2606.10650).

TEST INFRASTRUCTURE ONLY.  Imported by ``tests/``, by
``__graft_entry__.smoke()`` and by the CPU-baseline / reference leg of
``bench.py``; nothing in the ``paper_2606_10650_gb300`` package imports it,
and this package imports nothing from there.

The arithmetic lives in ``dla_oracle.c`` (plain C, fp64, explicit matrices);
this module only compiles it with gcc, loads it with ctypes and marshals
numpy arrays.  Every function cites the passage it follows in the C file.

Orientation: states are ``[d_v, d_k]`` matrices ``S = sum_s v_s k_s^T``
(Sec. 2 recurrent form and Eq. capacity_bounded_output), outputs
``o_t = sum_i lambda_{t,i} S_i q_t``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from concurrent.futures import ThreadPoolExecutor

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "dla_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_SO = os.path.join(_BUILD, "liboracle.so")
_LIB = None
_LOCK = threading.Lock()

_D = ctypes.POINTER(ctypes.c_double)
_I = ctypes.POINTER(ctypes.c_int)
_LL = ctypes.POINTER(ctypes.c_longlong)
_U8 = ctypes.POINTER(ctypes.c_ubyte)


def build(force: bool = False) -> str:
    """Compile the oracle into oracle/_build/liboracle.so (gcc, no FMA contraction)."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_SO) or os.path.getmtime(_SO) < os.path.getmtime(_SRC):
        tmp = _SO + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-fPIC", "-shared", "-ffp-contract=off",
                               "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _SO)
    return _SO


def lib():
    global _LIB
    with _LOCK:
        if _LIB is None:
            L = ctypes.CDLL(build())
            L.orc_new.restype = ctypes.c_void_p
            L.orc_new.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_double,
                                  ctypes.c_double, ctypes.c_double, ctypes.c_int]
            L.orc_free.argtypes = [ctypes.c_void_p]
            L.orc_copy.argtypes = [ctypes.c_void_p, ctypes.c_void_p]
            L.orc_step.argtypes = [ctypes.c_void_p, _D, _D, _D, _I, _I]
            L.orc_probe.argtypes = [ctypes.c_void_p, _D, _D, _D]
            L.orc_readout.argtypes = [ctypes.c_void_p, _D, _D, _D]
            L.orc_forward.argtypes = [ctypes.c_void_p, ctypes.c_longlong, _D, _D, _D,
                                      ctypes.c_longlong, _D, ctypes.c_longlong, _U8, _D,
                                      ctypes.c_longlong, _U8, _I, _D]
            L.orc_export.argtypes = [ctypes.c_void_p, _D, _LL, _D, _LL, _LL, _I, _LL]
            L.orc_get_m.argtypes = [ctypes.c_void_p]
            L.orc_get_m.restype = ctypes.c_int
            L.orc_get_t.argtypes = [ctypes.c_void_p]
            L.orc_get_t.restype = ctypes.c_longlong
            _LIB = L
    return _LIB


def _p(a, typ=_D):
    return None if a is None else a.ctypes.data_as(typ)


def _f64(a):
    return np.ascontiguousarray(a, dtype=np.float64)


class Stream:
    """One (batch, head) stream: the state cache M of Algorithm 2 plus the
    open state of Algorithm 1, advanced one token at a time."""

    def __init__(self, C, dk, dv, tau, eps=1e-6, rms_eps=1e-6, score_mode=0, _handle=None):
        self.C, self.dk, self.dv = int(C), int(dk), int(dv)
        self.tau, self.eps, self.rms_eps, self.score_mode = float(tau), float(eps), float(rms_eps), int(score_mode)
        L = lib()
        self._h = _handle or L.orc_new(self.C, self.dk, self.dv, self.tau, self.eps,
                                       self.rms_eps, self.score_mode)
        if not self._h:
            raise ValueError("oracle: invalid stream parameters (need C >= 2)")

    def __del__(self):
        h = getattr(self, "_h", None)
        if h and _LIB is not None:
            _LIB.orc_free(h)
            self._h = None

    def copy(self) -> "Stream":
        s = Stream(self.C, self.dk, self.dv, self.tau, self.eps, self.rms_eps, self.score_mode)
        lib().orc_copy(s._h, self._h)
        return s

    @property
    def m(self) -> int:
        return lib().orc_get_m(self._h)

    @property
    def t(self) -> int:
        return lib().orc_get_t(self._h)

    def step(self, k, v):
        """Score, boundary, merge and update for one token (Alg. 1 + Alg. 2)."""
        k, v = _f64(k), _f64(v)
        I = ctypes.c_double()
        b = ctypes.c_int()
        j = ctypes.c_int()
        lib().orc_step(self._h, _p(k), _p(v), ctypes.byref(I), ctypes.byref(b), ctypes.byref(j))
        return I.value, b.value, j.value

    def probe(self, k, v) -> dict:
        """The decision ``step`` would take, with its margins; no state change."""
        k, v = _f64(k), _f64(v)
        out = np.zeros(9)
        lib().orc_probe(self._h, _p(k), _p(v), _p(out))
        return dict(I=out[0], boundary=int(out[1]), merge=int(out[2]), best=out[3],
                    runner_up=out[4], thr_margin=out[5], tie_gap=out[6], rollback_to=int(out[7]),
                    rollback_last=int(out[8]))

    def readout(self, q, lam=None) -> np.ndarray:
        """o = sum_i lambda_i S_i q over the current cache (Eq. capacity_bounded_output)."""
        q = _f64(q)
        lam = None if lam is None else _f64(lam)
        o = np.zeros(self.dv)
        lib().orc_readout(self._h, _p(q), _p(lam), _p(o))
        return o

    def export(self) -> dict:
        m = self.m
        states = np.zeros((max(m, 1), self.dv, self.dk))
        n = np.zeros(max(m, 1), np.int64)
        ibar = np.zeros(max(m, 1))
        first = np.zeros(max(m, 1), np.int64)
        last = np.zeros(max(m, 1), np.int64)
        mm = ctypes.c_int()
        tt = ctypes.c_longlong()
        lib().orc_export(self._h, _p(states), _p(n, _LL), _p(ibar), _p(first, _LL), _p(last, _LL),
                         ctypes.byref(mm), ctypes.byref(tt))
        return dict(states=states[:m], n=n[:m], ibar=ibar[:m], first=first[:m], last=last[:m],
                    m=m, t=tt.value)

    def run(self, q, k, v, lam=None, want_o=None, o_out=None):
        """Advance over T tokens of one stream.

        q, k, v: [T, d] (any row stride), lam: [T, C] or None, want_o: bool [T]
        or None (all).  Returns (o [T, dv] or None, boundary u8 [T], merge_log
        int32 [T], itrace f64 [T])."""
        k = _f64(k); v = _f64(v)
        q = _f64(q) if q is not None else np.zeros_like(k)
        T = k.shape[0]
        assert k.shape == (T, self.dk) and v.shape == (T, self.dv) and q.shape == (T, self.dk)
        if self.dk != self.dv:
            raise ValueError("oracle.run expects d_k == d_v (shared row stride)")
        lamv = None if lam is None else _f64(lam)
        if lamv is not None:
            assert lamv.shape == (T, self.C)
        wo = None if want_o is None else np.ascontiguousarray(want_o, dtype=np.uint8)
        compute_o = (want_o is None) or bool(np.any(want_o))
        o = None
        if compute_o:
            o = o_out if o_out is not None else np.zeros((T, self.dv))
        bnd = np.zeros(T, np.uint8)
        ml = np.zeros(T, np.int32)
        it = np.zeros(T)
        lib().orc_forward(self._h, T, _p(q), _p(k), _p(v), self.dk,
                          _p(lamv), self.C, _p(wo, _U8), _p(o), self.dv,
                          _p(bnd, _U8), _p(ml, _I), _p(it))
        return o, bnd, ml, it


def _threads(n):
    return max(1, min(n, int(os.environ.get("DLA_ORACLE_THREADS", os.cpu_count() or 1))))


def forward(q, k, v, lam, *, tau, C, eps=1e-6, rms_eps=1e-6, score_mode=0,
            want_o=None, streams=None, threads=None):
    """Oracle prefill over a [B, T, H, d] batch.

    q, k, v: float arrays [B, T, H, d] (exact input values); lam [B, T, H, C] or
    None; want_o: bool [T] (same tokens for every stream) or None (all);
    streams: iterable of (b, h) to run (default all).  Streams run on a thread
    pool (the C code releases the GIL).  Returns dict with o [B, T, H, dv]
    (NaN where not computed / not run), boundary [B, H, T] u8, merge_log
    [B, H, T] int32, itrace [B, H, T] f64 and caches {(b, h): export dict}.
    """
    q = np.asarray(q); k = np.asarray(k); v = np.asarray(v)
    B, T, H, dk = k.shape
    dv = v.shape[-1]
    if streams is None:
        streams = [(b, h) for b in range(B) for h in range(H)]
    streams = list(streams)
    o = np.full((B, T, H, dv), np.nan)
    bnd = np.zeros((B, H, T), np.uint8)
    ml = np.full((B, H, T), -2, np.int32)
    it = np.zeros((B, H, T))
    caches = {}

    def one(bh):
        b, h = bh
        st = Stream(C, dk, dv, tau, eps, rms_eps, score_mode)
        lam_bh = None if lam is None else lam[b, :, h, :]
        ob, bb, mb, ib = st.run(q[b, :, h, :], k[b, :, h, :], v[b, :, h, :], lam_bh, want_o)
        if ob is not None:
            o[b, :, h, :] = ob if want_o is None else np.where(np.asarray(want_o)[:, None], ob, np.nan)
        bnd[b, h] = bb; ml[b, h] = mb; it[b, h] = ib
        caches[(b, h)] = st.export()

    n = _threads(len(streams) if threads is None else threads)
    if n == 1:
        for bh in streams:
            one(bh)
    else:
        with ThreadPoolExecutor(n) as ex:
            list(ex.map(one, streams))
    return dict(o=o, boundary=bnd, merge_log=ml, itrace=it, caches=caches)
