"""Calibrate the boundary threshold tau (and the regime value scale kappa) of
each synthetic workload with the fp64 oracle's decision pass.

Run:  python tests/golden/calibrate_workloads.py   (prints the constants)

It calls only ``oracle`` and the seeded generators of
``paper_2606_10650_gb300.workloads``; the constants it prints are the ones
hard-coded in that module, and ``tests/test_workloads.py`` re-runs it and
checks they match.

Rules (each on warm-up seeds disjoint from the test / bench seeds):
  tiny      tau = median of I_t (t >= 1) of a pass whose threshold never fires
  standard  tau such that 1 token in 64 opens a boundary (fixed point of the
            (1 - 1/64) score quantile of the decision pass)
  regime    kappa so that the oracle output RMS is about 1, and tau so that
            1 token in 256 opens a boundary
  long      uses the regime workload's tau and kappa (its regime spans are
            generated the same way; its i.i.d. spans then fire on most tokens)
  decode    as standard, at d = 128, C = 64
"""
import dataclasses
import os
import sys
from concurrent.futures import ThreadPoolExecutor

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import oracle  # noqa: E402
from paper_2606_10650_gb300 import workloads as W  # noqa: E402


def _streams(w, n, T, seed):
    out = []
    for i in range(n):
        g = W.StreamGen(dataclasses.replace(w, T=T, decode_steps=0), 0, i, seed)
        q, k, v = g.tokens()
        out.append((q, k, v, g.lam()))
    return out


def _scores(w, tau, streams, want_o=None):
    def one(s):
        q, k, v, lam = s
        st = oracle.Stream(w.C, w.d, w.d, tau, w.eps, w.rms_eps)
        return st.run(q, k, v, lam, want_o=want_o)

    with ThreadPoolExecutor(len(streams)) as ex:
        res = list(ex.map(one, streams))
    its, bnds, outs = [], [], []
    for o, b, _, it in res:
        its.append(it[1:]); bnds.append(b[1:])
        if o is not None and want_o is not None:
            outs.append(o[np.asarray(want_o, bool)])
    return np.concatenate(its), np.concatenate(bnds), (np.concatenate(outs) if outs else None)


def _rate_tau(w, rate, streams, iters=5):
    it, _, _ = _scores(w, 1e300, streams)
    tau = float(np.quantile(it, 1.0 - rate))
    for _ in range(iters):
        it, _, _ = _scores(w, tau, streams)
        tau = float(np.quantile(it, 1.0 - rate))
    return tau


def calibrate():
    res = {}
    # tiny: median score of a never-firing warm-up pass (warm-up seed 1001)
    w = W.get("tiny")
    it, _, _ = _scores(w, 1e300, _streams(w, 1, w.T, 1001))
    res["tiny"] = dict(tau=float(np.median(it)))
    # standard: 1/64 boundary rate (warm-up seed 2002)
    w = W.get("standard")
    res["standard"] = dict(tau=_rate_tau(w, 1 / 64, _streams(w, 4, 2048, 2002)))
    # regime: kappa for output RMS ~ 1, then tau for a 1/256 rate (warm-up seed 2003)
    w = W.get("regime", kappa=0.1)
    T = 4096
    want = np.zeros(T, bool); want[T // 2::97] = True
    kappa = 0.1
    tau = 1.3
    for _ in range(2):
        w = W.get("regime", kappa=kappa)
        streams = _streams(w, 4, T, 2003)
        tau = _rate_tau(w, 1 / 256, streams, iters=4)
        _, _, o = _scores(dataclasses.replace(w, tau=tau), tau, streams, want)
        rms = float(np.sqrt(np.mean(o ** 2)))
        kappa = kappa / rms
    w = W.get("regime", kappa=kappa)
    tau = _rate_tau(w, 1 / 256, _streams(w, 4, T, 2003), iters=4)
    res["regime"] = dict(tau=tau, kappa=kappa)
    res["long"] = dict(tau=tau, kappa=kappa)
    # decode: 1/64 boundary rate at C = 64 (warm-up seed 2005)
    w = W.get("decode")
    res["decode"] = dict(tau=_rate_tau(w, 1 / 64, _streams(w, 4, 2048, 2005)))
    return res


def rounded(res):
    return {k: {kk: float(f"{vv:.9g}") for kk, vv in v.items()} for k, v in res.items()}


if __name__ == "__main__":
    import json
    print(json.dumps(rounded(calibrate()), indent=1))
