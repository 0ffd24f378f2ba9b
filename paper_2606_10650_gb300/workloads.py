"""Seeded synthetic workloads for the DLA forward path.

This module only draws random numbers and shapes them into q, k, v and
lambda tensors; it holds none of the method's arithmetic (no score, no
boundary, no merge, no read-out).  Both the CUDA path and the fp64 oracle
consume what it produces.

The paper measures on language data and trained backbones (Sec. 4) that are
not available here; these generators stand in for them with the shapes the
paper's long-context setting implies (16K training context, Sec. 4.1;
capacity 16-64 around the paper's default 30) and with piecewise-stationary
key/value streams, the non-stationary setting of the Corollary in Sec. 3.1.

Workloads (names used across tests and the benchmark):
  tiny      B=1  H=2  T=512    d=64  C=8   fp32  i.i.d. N(0,1), k rows unit norm
  standard  B=4  H=16 T=4096   d=128 C=16  bf16  i.i.d. N(0,1)/sqrt(128), k unit
  regime    B=2  H=16 T=16384  d=128 C=32  bf16  regime shifts, Geometric(mean 256)
  long      B=1  H=32 T=65536  d=128 C=64  bf16  alternating 8K i.i.d. / regime blocks
  decode    B=256 H=32 d=128 C=64 bf16 inputs, fp32 cache: 8K-token i.i.d. prefill,
            then single-token steps of N(0,1)/sqrt(128) q, k, v

tau (and kappa, the value scale of regime spans) are constants calibrated by
``tests/golden/calibrate_workloads.py`` with the oracle's decision pass; a
CPU test re-runs that script and checks it reproduces them.

Every stream (b, h) draws from its own generator keyed by (seed, b, h), so a
single stream can be regenerated on the host without generating the batch;
a rejected token t is redrawn from a generator keyed by (seed, b, h, t,
attempt).
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

try:  # torch is only needed for bf16 rounding and device-side generation
    import torch
except Exception:  # pragma: no cover
    torch = None


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    B: int
    H: int
    T: int
    d: int
    C: int
    dtype: str          # "f32" or "bf16": input dtype of q, k, v
    kind: str           # "iid", "regime", "mixed"
    tau: float          # boundary threshold (calibrated)
    kappa: float = 1.0  # value scale of regime spans (calibrated)
    qk_scale: float = 1.0  # std of the i.i.d. Gaussian draws (before k normalisation)
    seg_mean: float = 256.0  # mean regime length (Geometric)
    noise: float = 0.1  # per-component noise std of regime spans
    block: int = 8192   # block length of the mixed workload
    seed: int = 0
    decode_steps: int = 0
    lam_lo: float = 0.5
    lam_hi: float = 1.5
    eps: float = 1e-6
    rms_eps: float = 1e-6

    @property
    def total_tokens(self) -> int:
        return self.T + self.decode_steps


# Calibrated constants (tests/golden/calibrate_workloads.py writes these).
WORKLOADS = {
    "tiny": Workload("tiny", 1, 2, 512, 64, 8, "f32", "iid", tau=1.41446883, qk_scale=1.0, seed=1),
    "standard": Workload("standard", 4, 16, 4096, 128, 16, "bf16", "iid", tau=1.42122581,
                         qk_scale=1.0 / math.sqrt(128), seed=2),
    "regime": Workload("regime", 2, 16, 16384, 128, 32, "bf16", "regime", tau=1.31297564, kappa=0.140930239,
                       qk_scale=1.0 / math.sqrt(128), seed=3),
    "long": Workload("long", 1, 32, 65536, 128, 64, "bf16", "mixed", tau=1.31297564, kappa=0.140930239,
                     qk_scale=1.0 / math.sqrt(128), seed=4),
    "decode": Workload("decode", 256, 32, 8192, 128, 64, "bf16", "iid", tau=1.42087254,
                       qk_scale=1.0 / math.sqrt(128), seed=5, decode_steps=1024),
}


def get(name: str, **overrides) -> Workload:
    w = WORKLOADS[name]
    return dataclasses.replace(w, **overrides) if overrides else w


# ---------------------------------------------------------------- rounding

def round_to(x: np.ndarray, dtype: str) -> np.ndarray:
    """Round float64 values to the input dtype and return them as float64
    (the exact values the device will see)."""
    if dtype == "f32":
        return x.astype(np.float32).astype(np.float64)
    if dtype == "bf16":
        t = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).to(torch.bfloat16)
        return t.to(torch.float64).numpy()
    raise ValueError(dtype)


def _unit_rows(x: np.ndarray) -> np.ndarray:
    return x / np.linalg.norm(x, axis=-1, keepdims=True)


# ---------------------------------------------------------------- streams

class StreamGen:
    """Token source of one (b, h) stream of a workload (host, float64)."""

    def __init__(self, w: Workload, b: int, h: int, seed: int | None = None):
        self.w, self.b, self.h = w, b, h
        self.seed = w.seed if seed is None else seed
        Ttot = w.total_tokens
        rng = np.random.default_rng(np.random.SeedSequence([self.seed, b, h, 11]))
        d = w.d
        # regime structure: a new regime starts at t with probability 1/seg_mean
        # (Geometric segment lengths, support >= 1); token 0 starts regime 0.
        if w.kind in ("regime", "mixed"):
            flags = rng.random(Ttot) < (1.0 / w.seg_mean)
            flags[0] = True
            self.seg = np.cumsum(flags) - 1
            nseg = int(self.seg[-1]) + 1
            self.mu_k = _unit_rows(rng.standard_normal((nseg, d)))
            self.mu_v = _unit_rows(rng.standard_normal((nseg, d)))
        else:
            self.seg = None
        self._rng = rng

    def _is_regime(self, t: np.ndarray) -> np.ndarray:
        w = self.w
        if w.kind == "regime":
            return np.ones(t.shape, bool)
        if w.kind == "mixed":
            return (t // w.block) % 2 == 1
        return np.zeros(t.shape, bool)

    def _draw_kv(self, rng, t: np.ndarray):
        w, d = self.w, self.w.d
        n = t.shape[0]
        zk = rng.standard_normal((n, d))
        zv = rng.standard_normal((n, d))
        k = _unit_rows(zk)
        v = zv * w.qk_scale
        reg = self._is_regime(t)
        if reg.any():
            s = self.seg[t[reg]]
            k[reg] = _unit_rows(self.mu_k[s] + w.noise * zk[reg])
            v[reg] = w.kappa * (self.mu_v[s] + w.noise * zv[reg])
        dec = t >= w.T
        if dec.any():  # decode steps: plain N(0,1)/sqrt(128) q, k, v (no normalisation)
            k[dec] = zk[dec] * w.qk_scale
        return k, v

    def tokens(self):
        """q, k, v [T_total, d] float64, already rounded to the input dtype."""
        w = self.w
        t = np.arange(w.total_tokens)
        q = self._rng.standard_normal((w.total_tokens, w.d)) * w.qk_scale
        k, v = self._draw_kv(self._rng, t)
        return round_to(q, w.dtype), round_to(k, w.dtype), round_to(v, w.dtype)

    def redraw(self, t: int, attempt: int):
        """A fresh (k, v) for token t (attempt >= 1), same regime as before."""
        rng = np.random.default_rng(np.random.SeedSequence([self.seed, self.b, self.h, t, attempt, 23]))
        k, v = self._draw_kv(rng, np.array([t]))
        return round_to(k[0], self.w.dtype), round_to(v[0], self.w.dtype)

    def lam(self):
        """lambda [T_total, C] float32 values (as float64), U(lam_lo, lam_hi)."""
        w = self.w
        rng = np.random.default_rng(np.random.SeedSequence([self.seed, self.b, self.h, 31]))
        lam = rng.uniform(w.lam_lo, w.lam_hi, size=(w.total_tokens, w.C))
        return lam.astype(np.float32).astype(np.float64)


def host_batch(w: Workload, with_lam: bool = True, seed: int | None = None, T: int | None = None):
    """Whole [B, T, H, d] batch on the host (float64 exact values).
    Returns q, k, v, lam (lam None if not requested)."""
    T = w.total_tokens if T is None else T
    q = np.empty((w.B, T, w.H, w.d))
    k = np.empty_like(q)
    v = np.empty_like(q)
    lam = np.empty((w.B, T, w.H, w.C)) if with_lam else None
    for b in range(w.B):
        for h in range(w.H):
            g = StreamGen(w, b, h, seed)
            qq, kk, vv = g.tokens()
            q[b, :, h], k[b, :, h], v[b, :, h] = qq[:T], kk[:T], vv[:T]
            if with_lam:
                lam[b, :, h] = g.lam()[:T]
    return q, k, v, lam


def _stream_job(job):
    """Worker of host_batch_parallel: one (b, h) stream as float32 arrays."""
    w, b, h, seed, T = job
    g = StreamGen(w, b, h, seed)
    qq, kk, vv = g.tokens()
    return b, h, qq[:T].astype(np.float32), kk[:T].astype(np.float32), vv[:T].astype(np.float32), \
        g.lam()[:T].astype(np.float32)


def host_batch_parallel(w: Workload, seed: int | None = None, T: int | None = None, procs: int | None = None):
    """host_batch drawn by a pool of spawned processes, one stream per task,
    returned as float32 arrays (exact: the values are bf16 or fp32 numbers).
    The same values as host_batch."""
    import multiprocessing as mp
    import os
    T = w.total_tokens if T is None else T
    q = np.empty((w.B, T, w.H, w.d), np.float32)
    k = np.empty_like(q)
    v = np.empty_like(q)
    lam = np.empty((w.B, T, w.H, w.C), np.float32)
    jobs = [(w, b, h, seed, T) for b in range(w.B) for h in range(w.H)]
    n = procs or min(len(jobs), os.cpu_count() or 1)
    with mp.get_context("spawn").Pool(n) as pool:
        for b, h, qq, kk, vv, ll in pool.imap_unordered(_stream_job, jobs):
            q[b, :, h], k[b, :, h], v[b, :, h], lam[b, :, h] = qq, kk, vv, ll
    return q, k, v, lam


def to_device(x: np.ndarray, dtype: str, device):
    """Upload exact values as the device input dtype."""
    tdt = torch.float32 if dtype == "f32" else torch.bfloat16
    return torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).to(device=device).to(tdt)


# ---------------------------------------------------------------- device-side bulk draws

def device_iid_batch(w: Workload, B: int, T: int, seed: int, device, with_lam=True):
    """i.i.d. workload drawn directly on the device (for batches too large to
    draw on the host): q, v ~ N(0, qk_scale^2), k unit rows (or plain Gaussian
    for decode steps, ``T`` tokens treated as decode steps when
    ``decode=True`` in :func:`device_decode_steps`)."""
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    dt = torch.float32 if w.dtype == "f32" else torch.bfloat16
    shape = (B, T, w.H, w.d)
    q = (torch.randn(shape, generator=g, device=device) * w.qk_scale).to(dt)
    k = torch.randn(shape, generator=g, device=device)
    k = (k / k.norm(dim=-1, keepdim=True)).to(dt)
    v = (torch.randn(shape, generator=g, device=device) * w.qk_scale).to(dt)
    lam = None
    if with_lam:
        lam = torch.empty((B, T, w.H, w.C), device=device).uniform_(w.lam_lo, w.lam_hi, generator=g)
    return q, k, v, lam


def device_decode_steps(w: Workload, steps: int, seed: int, device, with_lam=True):
    """Decode-step tokens [steps, B, H, d] (N(0,1)/sqrt(128), bf16) and lambda
    [steps, B, H, C] drawn on the device."""
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    dt = torch.float32 if w.dtype == "f32" else torch.bfloat16
    shape = (steps, w.B, w.H, w.d)
    q = (torch.randn(shape, generator=g, device=device) * w.qk_scale).to(dt)
    k = (torch.randn(shape, generator=g, device=device) * w.qk_scale).to(dt)
    v = (torch.randn(shape, generator=g, device=device) * w.qk_scale).to(dt)
    lam = None
    if with_lam:
        lam = torch.empty((steps, w.B, w.H, w.C), device=device).uniform_(w.lam_lo, w.lam_hi, generator=g)
    return q, k, v, lam
