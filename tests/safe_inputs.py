"""Decision-safe inputs: seeded streams whose every discrete decision has a
margin, so that an fp32 device path and the fp64 oracle must agree bit for bit.

Test infrastructure (uses the oracle).  For one (b, h) stream it walks the
tokens of :class:`paper_2606_10650_gb300.workloads.StreamGen` through the
oracle and

  G1  redraws token t while its score lies within ``THR_MARGIN`` (relative)
      of tau;
  G2  when token t would merge and the best and runner-up adjacent-pair
      densities lie within ``TIE_MARGIN`` (relative) of each other, rolls back
      to the last token of the newest state among the two pairs (changing
      that token's score changes the state's summed score, the shortest
      rollback that moves one of the tied densities), redraws it and replays
      from a checkpoint (G3).

Redraws come from generators keyed by (seed, b, h, t, attempt), so the result
is reproducible.  THR_MARGIN is 1e-3 relative.  TIE_MARGIN is 1e-5 relative:
a 1e-3 tie margin admits almost no streams (the pair densities of a full cache
of i.i.d. tokens crowd into a band about 1e-3 wide), while the device's summed
scores differ from the oracle's by at most ~2.5e-8 relative, so 1e-5 keeps a
safety factor of 400.
"""
from __future__ import annotations

import dataclasses

import numpy as np

import oracle
from paper_2606_10650_gb300 import workloads as W

THR_MARGIN = 1e-3
TIE_MARGIN = 1e-5


class RejectionFailed(RuntimeError):
    pass


def safe_stream(w: W.Workload, b: int, h: int, T: int | None = None, seed: int | None = None,
                thr: float = THR_MARGIN, tie: float = TIE_MARGIN, score_mode: int = 0,
                max_rollbacks: int = 100000, max_attempts: int = 64):
    g = W.StreamGen(w, b, h, seed)
    q, k, v = g.tokens()
    lam = g.lam()
    T = w.total_tokens if T is None else int(T)
    q, k, v, lam = q[:T].copy(), k[:T].copy(), v[:T].copy(), lam[:T].copy()
    attempts = np.zeros(T, np.int64)
    # checkpoints: every FINE tokens, the last NFINE of them kept, plus every COARSE tokens
    FINE, NFINE, COARSE = 16, 32, 1024
    st = oracle.Stream(w.C, w.d, w.d, w.tau, w.eps, w.rms_eps, score_mode)
    ckpts = {0: st.copy()}
    redraws = rollbacks = 0

    def redraw(t):
        attempts[t] += 1
        k[t], v[t] = g.redraw(t, int(attempts[t]))

    def restore(t0):
        nonlocal st
        c = max(c for c in ckpts if c <= t0)
        for kk in [kk for kk in ckpts if kk > c]:
            del ckpts[kk]
        st = ckpts[c].copy()
        for s in range(c, t0):
            st.step(k[s], v[s])

    t = 0
    while t < T:
        r = st.probe(k[t], v[t])
        if r["thr_margin"] < thr:
            if attempts[t] >= max_attempts and t > 0:
                rollbacks += 1
                redraw(t - 1)
                restore(t - 1)
                t -= 1
            else:
                redraw(t)
                redraws += 1
            continue
        if r["merge"] >= 0 and r["tie_gap"] < tie:
            rollbacks += 1
            if rollbacks > max_rollbacks:
                raise RejectionFailed(f"{w.name} stream ({b},{h}): too many rollbacks")
            t0 = r["rollback_last"]
            redraw(t0)
            restore(t0)
            t = t0
            continue
        st.step(k[t], v[t])
        t += 1
        if t % FINE == 0:
            ckpts[t] = st.copy()
            old = t - FINE * NFINE
            if old > 0 and old % COARSE != 0:
                ckpts.pop(old, None)
    return dict(q=q, k=k, v=v, lam=lam, redraws=redraws, rollbacks=rollbacks)


def safe_batch(w: W.Workload, T: int | None = None, streams=None, seed: int | None = None, threads=None):
    """Host batch [B, T, H, d] where the listed streams (default: all) are
    decision-safe and the others are the plain seeded draws."""
    from concurrent.futures import ThreadPoolExecutor
    T = w.total_tokens if T is None else int(T)
    q, k, v, lam = W.host_batch(w, seed=seed, T=T)
    streams = [(b, h) for b in range(w.B) for h in range(w.H)] if streams is None else list(streams)
    stats = {}

    def one(bh):
        b, h = bh
        r = safe_stream(w, b, h, T=T, seed=seed)
        q[b, :, h], k[b, :, h], v[b, :, h], lam[b, :, h] = r["q"], r["k"], r["v"], r["lam"]
        stats[bh] = (r["redraws"], r["rollbacks"])

    n = threads or min(8, len(streams))
    with ThreadPoolExecutor(max(1, n)) as ex:
        list(ex.map(one, streams))
    return q, k, v, lam, stats


def shrink(w: W.Workload, **kw) -> W.Workload:
    return dataclasses.replace(w, **kw)


def _safe_and_oracle(job):
    """Worker of safe_oracle_streams (a separate process): one decision-safe
    stream and the oracle's results on it."""
    w, b, h, T, seed, score_mode, want_o = job
    r = safe_stream(w, b, h, T=T, seed=seed, score_mode=score_mode)
    st = oracle.Stream(w.C, w.d, w.d, w.tau, w.eps, w.rms_eps, score_mode)
    o, bnd, ml, _ = st.run(r["q"], r["k"], r["v"], r["lam"], want_o=want_o)
    ex = st.export()
    f32 = lambda x: x.astype(np.float32)  # exact: the inputs are bf16 / fp32 values
    return dict(b=b, h=h, q=f32(r["q"]), k=f32(r["k"]), v=f32(r["v"]), lam=f32(r["lam"]), bnd=bnd, ml=ml,
                o=None if o is None else (o if want_o is None else o[np.asarray(want_o, bool)]),
                cache=dict(states=ex["states"], n=ex["n"], ibar=ex["ibar"], m=ex["m"]),
                rollbacks=r["rollbacks"], redraws=r["redraws"])


def safe_oracle_streams(w: W.Workload, T: int | None = None, streams=None, seed: int | None = None,
                        score_mode: int = 0, want_o=None, procs: int | None = None):
    """Decision-safe inputs and the oracle's results for the listed streams of
    a batch (default all), one stream per worker process (spawned, so that it
    is safe after CUDA was initialised in this process).

    Returns (q, k, v, lam) host arrays [B, T, H, *] (float64 values; streams
    not listed keep the plain seeded draws) and the oracle's results in the
    layout of ``oracle.forward``: o [B, T, H, d] (NaN where not computed),
    boundary, merge_log and caches."""
    import multiprocessing as mp
    import os
    T = w.total_tokens if T is None else int(T)
    streams = [(b, h) for b in range(w.B) for h in range(w.H)] if streams is None else list(streams)
    q, k, v, lam = W.host_batch(w, seed=seed, T=T)
    o = np.full(q.shape, np.nan)
    bnd = np.zeros((w.B, w.H, T), np.uint8)
    ml = np.full((w.B, w.H, T), -2, np.int32)
    caches = {}
    n = procs or min(len(streams), os.cpu_count() or 1)
    jobs = [(w, b, h, T, seed, score_mode, want_o) for (b, h) in streams]
    with mp.get_context("spawn").Pool(n) as pool:
        for res in pool.imap_unordered(_safe_and_oracle, jobs):
            b, h = res["b"], res["h"]
            q[b, :, h], k[b, :, h], v[b, :, h], lam[b, :, h] = res["q"], res["k"], res["v"], res["lam"]
            bnd[b, h], ml[b, h] = res["bnd"], res["ml"]
            if res["o"] is not None:
                if want_o is None:
                    o[b, :, h] = res["o"]
                else:
                    o[b, np.asarray(want_o, bool), h] = res["o"]
            caches[(b, h)] = res["cache"]
    return (q, k, v, lam), dict(o=o, boundary=bnd, merge_log=ml, caches=caches)
