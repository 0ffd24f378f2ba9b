"""Decision-safe inputs: seeded streams whose every discrete decision has a
margin, so that an fp32 device path and the fp64 oracle must agree bit for bit.

Test infrastructure (uses the oracle).  For one (b, h) stream it walks the
tokens of :class:`paper_2606_10650_gb300.workloads.StreamGen` through the
oracle and

  G1  redraws token t while its score lies within ``THR_MARGIN`` (relative)
      of tau;
  G2  when token t would merge and the best and runner-up adjacent-pair
      densities lie within ``TIE_MARGIN`` (relative) of each other, rolls back
      to the first token of the newest state among the two pairs, redraws that
      token and replays from a checkpoint (G3).

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
                max_rollbacks: int = 20000, max_attempts: int = 64):
    g = W.StreamGen(w, b, h, seed)
    q, k, v = g.tokens()
    lam = g.lam()
    T = w.total_tokens if T is None else int(T)
    q, k, v, lam = q[:T].copy(), k[:T].copy(), v[:T].copy(), lam[:T].copy()
    attempts = np.zeros(T, np.int64)
    ck_every = max(256, T // 32)
    st = oracle.Stream(w.C, w.d, w.d, w.tau, w.eps, w.rms_eps, score_mode)
    ckpts = {0: st.copy()}
    redraws = rollbacks = 0

    def redraw(t):
        attempts[t] += 1
        k[t], v[t] = g.redraw(t, int(attempts[t]))

    def restore(t0):
        nonlocal st, ckpts
        c = max(c for c in ckpts if c <= t0)
        ckpts = {kk: vv for kk, vv in ckpts.items() if kk <= c}
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
            t0 = r["rollback_to"]
            redraw(t0)
            restore(t0)
            t = t0
            continue
        st.step(k[t], v[t])
        t += 1
        if t % ck_every == 0:
            ckpts[t] = st.copy()
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
