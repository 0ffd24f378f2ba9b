"""Pins of the fp64 oracle against what the paper and the mathematics fix.

None of these re-types the oracle's own formula: each compares it with an
independent fact -- a hand-derived example, a closed form, a textbook routine
(dense causal linear attention), a brute-force recomputation from the
exported cache, or a conservation law -- so that a dropped term, a wrong sign
or index, or a transposed operand in the oracle fails at least one of them.
"""
import json
import math
import os

import numpy as np
import pytest

import oracle

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _rand_stream(rng, T, d, unit_k=True):
    q = rng.standard_normal((T, d))
    k = rng.standard_normal((T, d))
    if unit_k:
        k /= np.linalg.norm(k, axis=1, keepdims=True)
    v = rng.standard_normal((T, d))
    return q, k, v


def _median_tau(q, k, v, d):
    """A threshold near the median score, so that roughly half the tokens open
    a boundary (plenty of boundaries and merges)."""
    st = oracle.Stream(2, d, d, tau=1e300)
    _, _, _, it = st.run(q, k, v)
    return float(np.median(it[1:]))


# ------------------------------------------------------------------ hand example

def test_hand_example_mode0():
    """Algorithm 1 score with RMSNorm, Algorithm 2 merge, Eq. capacity_bounded_output."""
    g = json.load(open(os.path.join(GOLD, "hand_example.json")))
    st = oracle.Stream(2, 2, 2, tau=1.0, eps=0.0, rms_eps=0.0, score_mode=0)
    K = np.array(g["tokens_k"], float)
    V = np.array(g["tokens_v"], float)
    for t in range(4):
        I, b, j = st.step(K[t], V[t])
        assert I == pytest.approx(g["I_mode0"][t], abs=1e-15)
        assert b == g["boundary_mode0"][t]
        assert j == g["merge_mode0"][t]
        if t == 2:
            ex = st.export()
            np.testing.assert_array_equal(ex["states"], np.array(g["after_t2_states"], float))
            np.testing.assert_array_equal(ex["n"], g["after_t2_n"])
            np.testing.assert_allclose(ex["ibar"], g["after_t2_ibar"], rtol=0, atol=1e-15)
            o = st.readout(np.array(g["readout_q"], float), np.array(g["readout_lam"], float))
            np.testing.assert_allclose(o, g["readout_after_t2"], rtol=0, atol=1e-15)


def test_hand_example_mode1():
    """Eq. importance_score read literally: S_t = S_{t-1} + s_t against S_{t-1}."""
    g = json.load(open(os.path.join(GOLD, "hand_example.json")))
    st = oracle.Stream(2, 2, 2, tau=1.0, eps=0.0, rms_eps=0.0, score_mode=1)
    K = np.array(g["tokens_k"], float)
    V = np.array(g["tokens_v"], float)
    st.step(K[0], V[0])
    I, b, j = st.step(K[1], V[1])
    assert I == pytest.approx(g["I1_mode1"], abs=1e-15)
    assert b == 0 and j == -1


def test_hand_example_mode1_at_a_merge():
    """Eq. importance_score read literally, at a token that opens a boundary on a
    full cache (Algorithm 2 merge), values derived by hand."""
    g = json.load(open(os.path.join(GOLD, "hand_example.json")))
    h = g["mode1_merge"]
    st = oracle.Stream(h["C"], 2, 2, tau=h["tau"], eps=0.0, rms_eps=0.0, score_mode=1)
    K = np.array(g["tokens_k"], float)
    V = np.array(g["tokens_v"], float)
    for t in range(3):
        I, b, j = st.step(K[t], V[t])
        assert I == pytest.approx(h["I"][t], abs=1e-15)
        assert b == h["boundary"][t] and j == h["merge"][t]
    ex = st.export()
    np.testing.assert_array_equal(ex["states"], np.array(h["after_t2_states"], float))
    np.testing.assert_array_equal(ex["n"], h["after_t2_n"])
    np.testing.assert_allclose(ex["ibar"], h["after_t2_ibar"], rtol=0, atol=1e-15)


# ------------------------------------------------------------------ closed forms of the score

def _rms(x2, D, e):
    return math.sqrt(x2 / D + e)


@pytest.mark.parametrize("rms_eps,eps", [(1e-6, 1e-6), (0.0, 0.0), (1e-2, 1e-3)])
def test_score_parallel_token_closed_form(rms_eps, eps):
    """Token state parallel to the open state: S = c s.  Then
    N(s) - N(S) = s (1/r_s - c/r_S) and I = ||s|| |1/r_s - c/r_S| / (c ||s|| / r_S + eps),
    r_X = sqrt(||X||^2/D + rms_eps)."""
    rng = np.random.default_rng(3)
    d = 6
    k = rng.standard_normal(d); v = rng.standard_normal(d)
    st = oracle.Stream(4, d, d, tau=1e300, eps=eps, rms_eps=rms_eps)
    c = 3
    for _ in range(c):
        st.step(k, v)
    D = d * d
    a = float(np.dot(k, k) * np.dot(v, v))
    rs, rS = _rms(a, D, rms_eps), _rms(c * c * a, D, rms_eps)
    expect = math.sqrt(a) * abs(1 / rs - c / rS) / (c * math.sqrt(a) / rS + eps)
    assert st.probe(k, v)["I"] == pytest.approx(expect, rel=1e-12, abs=1e-15)


@pytest.mark.parametrize("rms_eps,eps", [(1e-6, 1e-6), (0.5, 0.1)])
def test_score_orthogonal_token_closed_form(rms_eps, eps):
    """k_t orthogonal to every key of the open segment gives <s_t, S> = 0, so
    I = sqrt(a/r_a^2 + g/r_g^2) / (sqrt(g)/r_g + eps) with a = ||k||^2||v||^2, g = ||S||^2."""
    d = 4
    e = np.eye(d)
    st = oracle.Stream(4, d, d, tau=1e300, eps=eps, rms_eps=rms_eps)
    rng = np.random.default_rng(5)
    vs = rng.standard_normal((2, d))
    st.step(e[0], vs[0]); st.step(e[1], vs[1])
    S = np.outer(vs[0], e[0]) + np.outer(vs[1], e[1])
    g = float((S * S).sum())
    kt, vt = 2.0 * e[2], rng.standard_normal(d)
    a = float(np.dot(kt, kt) * np.dot(vt, vt))
    D = d * d
    ra, rg = _rms(a, D, rms_eps), _rms(g, D, rms_eps)
    expect = math.sqrt(a / ra ** 2 + g / rg ** 2) / (math.sqrt(g) / rg + eps)
    assert st.probe(kt, vt)["I"] == pytest.approx(expect, rel=1e-12)


def test_score_is_scale_free_without_rms_eps():
    """With rms_eps = eps = 0 the RMSNorm removes any positive scale of either
    operand, so I depends only on directions (and lies in [0, 2])."""
    rng = np.random.default_rng(9)
    d = 5
    q, k, v = _rand_stream(rng, 12, d)
    st1 = oracle.Stream(3, d, d, tau=1e300, eps=0.0, rms_eps=0.0)
    st2 = oracle.Stream(3, d, d, tau=1e300, eps=0.0, rms_eps=0.0)
    _, _, _, i1 = st1.run(q, k, v)
    _, _, _, i2 = st2.run(q, 7.0 * k, 0.25 * v)
    np.testing.assert_allclose(i1, i2, rtol=1e-12, atol=1e-14)
    assert (i1 >= 0).all() and (i1 <= 2 + 1e-12).all()


# ------------------------------------------------------------------ reductions to textbook forms

@pytest.mark.parametrize("C", [2, 3, 5])
@pytest.mark.parametrize("mode", [0, 1])
def test_lambda_one_is_causal_linear_attention(C, mode):
    """With lambda == 1 merges and shifts only regroup sums, so for any tau and C
    the output is causal linear attention O = (Q K^T o M) V (Eq. linear_attn_parallel)."""
    rng = np.random.default_rng(11 + C)
    T, d = 48, 6
    q, k, v = _rand_stream(rng, T, d)
    tau = _median_tau(q, k, v, d) if mode == 0 else 0.3
    st = oracle.Stream(C, d, d, tau=tau, score_mode=mode)
    o, bnd, ml, _ = st.run(q, k, v)
    assert bnd[1:].sum() >= 4 and (ml >= 0).sum() >= 2, "fixture must exercise boundaries and merges"
    O = np.tril(q @ k.T) @ v
    np.testing.assert_allclose(o, O, rtol=1e-12, atol=1e-12)


def test_tau_inf_single_state_closed_form():
    """A threshold that never fires keeps one state S_t = sum_{s<=t} v_s k_s^T:
    o_t = lambda_{t,0} S_t q_t (Sec. 2 recurrent form scaled by lambda_{t,0})."""
    rng = np.random.default_rng(21)
    T, d, C = 40, 5, 4
    q, k, v = _rand_stream(rng, T, d)
    lam = rng.uniform(0.5, 1.5, size=(T, C))
    st = oracle.Stream(C, d, d, tau=1e300)
    o, bnd, ml, _ = st.run(q, k, v, lam)
    assert bnd.tolist() == [1] + [0] * (T - 1) and (ml == -1).all()
    O = (np.tril(q @ k.T) @ v) * lam[:, :1]
    np.testing.assert_allclose(o, O, rtol=1e-12, atol=1e-12)
    ex = st.export()
    assert ex["m"] == 1 and ex["n"].tolist() == [T]


def test_tau_zero_per_token_states_closed_form():
    """tau = 0 fires on every token (I >= 0); with C >= T nothing merges, each
    token is its own state and o_t = sum_{s<=t} lambda_{t,s} (q_t . k_s) v_s."""
    rng = np.random.default_rng(22)
    T, d = 24, 4
    C = T
    q, k, v = _rand_stream(rng, T, d)
    lam = rng.uniform(0.5, 1.5, size=(T, C))
    st = oracle.Stream(C, d, d, tau=0.0)
    o, bnd, ml, it = st.run(q, k, v, lam)
    assert bnd.all() and (ml == -1).all()
    W = np.tril(lam)  # weight of token s in row t is lambda_{t, s}
    O = ((q @ k.T) * W) @ v
    np.testing.assert_allclose(o, O, rtol=1e-12, atol=1e-12)
    ex = st.export()
    assert (ex["n"] == 1).all()
    np.testing.assert_allclose(ex["ibar"], it, rtol=0, atol=0)


def test_uncapped_dla_i_segment_sums():
    """DLA(I) (Table 5: dynamic merging without the capacity bound): with C above
    the number of segments nothing merges, every segment keeps its own state
    S_i = sum of v_s k_s^T over its tokens, and o_t = sum_i lambda_{t,i} S_i q_t
    over the segments begun at or before t, the open one holding the tokens up
    to t.  Recomputed here from the boundary trace alone."""
    rng = np.random.default_rng(23)
    T, d = 60, 4
    q, k, v = _rand_stream(rng, T, d)
    probe = oracle.Stream(2, d, d, tau=1e300)
    _, _, _, it = probe.run(q, k, v)
    tau = float(np.quantile(it[1:], 0.8))
    C = T + 1
    lam = rng.uniform(0.5, 1.5, size=(T, C))
    st = oracle.Stream(C, d, d, tau=tau)
    o, bnd, ml, _ = st.run(q, k, v, lam)
    assert (ml == -1).all() and 3 < int(bnd.sum()) < T
    starts = [int(s_) for s_ in np.flatnonzero(bnd)]
    ends = starts[1:] + [T]
    O = np.zeros((T, d))
    for t in range(T):
        for i, (s0, s1) in enumerate(zip(starts, ends)):
            if s0 > t:
                break
            S = sum(np.outer(v[s_], k[s_]) for s_ in range(s0, min(s1, t + 1)))
            O[t] += lam[t, i] * (S @ q[t])
    np.testing.assert_allclose(o, O, rtol=1e-12, atol=1e-12)
    ex = st.export()
    assert ex["m"] == len(starts)
    assert ex["n"][:len(starts)].tolist() == [e - s_ for s_, e in zip(starts, ends)]


# ------------------------------------------------------------------ brute force on tiny inputs

@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("C", [2, 3, 4])
@pytest.mark.parametrize("seed", [0, 1, 2])
def test_merge_brute_force(C, seed, mode):
    """Algorithm 2 step by step: before every token recompute from the exported
    cache what must happen (merge iff boundary and |M| = C; i* = argmin of the
    adjacent pair densities, lowest index on ties; S, n, Ibar summed; rest
    shifted; s_t appended) and compare with the oracle's new cache."""
    rng = np.random.default_rng(100 + seed)
    T, d = 64, 3
    q, k, v = _rand_stream(rng, T, d)
    tau = _median_tau(q, k, v, d) if mode == 0 else 0.25
    st = oracle.Stream(C, d, d, tau=tau, score_mode=mode)
    merges = 0
    for t in range(T):
        pre = st.export()
        I, b, j = st.step(k[t], v[t])
        post = st.export()
        s = np.outer(v[t], k[t])
        if pre["m"] == 0:
            assert b == 1 and j == -1 and post["m"] == 1
            continue
        if not b:
            assert j == -1 and post["m"] == pre["m"]
            exp_states = pre["states"].copy(); exp_states[-1] += s
            exp_n = pre["n"].copy(); exp_n[-1] += 1
            exp_ib = pre["ibar"].copy(); exp_ib[-1] += I
        else:
            states, n, ib = list(pre["states"]), list(pre["n"]), list(pre["ibar"])
            if pre["m"] == C:
                dens = [(ib[i] + ib[i + 1]) / (n[i] + n[i + 1]) for i in range(C - 1)]
                jj = min(range(C - 1), key=lambda i: (dens[i], i))
                assert j == jj
                merges += 1
                states[jj] = states[jj] + states[jj + 1]; del states[jj + 1]
                n[jj] += n[jj + 1]; del n[jj + 1]
                ib[jj] += ib[jj + 1]; del ib[jj + 1]
            else:
                assert j == -1
            states.append(s); n.append(1); ib.append(I)
            exp_states, exp_n, exp_ib = np.array(states), np.array(n), np.array(ib)
        np.testing.assert_allclose(post["states"], exp_states, rtol=0, atol=1e-12)
        np.testing.assert_array_equal(post["n"], exp_n)
        np.testing.assert_allclose(post["ibar"], exp_ib, rtol=1e-14, atol=1e-14)
    assert merges >= 5


def test_merge_lowest_index_on_exact_tie():
    """Identical pair densities everywhere: the oldest pair (index 0) is merged."""
    d = 2
    st = oracle.Stream(3, d, d, tau=0.0, eps=0.0, rms_eps=0.0)
    # every token identical -> every score after the first is 0 >= tau=0 -> boundary.
    # Ibar = [0, 0, 0] after three tokens, n = [1, 1, 1]: all densities 0.
    for _ in range(3):
        st.step(np.array([1.0, 0.0]), np.array([0.0, 1.0]))
    I, b, j = st.step(np.array([1.0, 0.0]), np.array([0.0, 1.0]))
    assert b == 1 and j == 0


@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("C", [3, 4, 5])
def test_probe_runner_up_gap_and_rollback_brute_force(C, mode):
    """orc_probe's merge diagnostics, which the decision-safe input generator
    relies on: at every token that merges, recompute from the exported cache
    all C - 1 adjacent pair densities (Algorithm 2's definition), order them by
    (density, index) and check the best pair, the runner-up density, the
    relative gap (runner-up - best) / |best| and the first and last tokens of
    the newest state among the two pairs (from the states' token counts, not
    from the oracle's own token ranges).  The probe must leave the stream unchanged and
    announce the decision the next step takes, with |I - tau| / tau as margin."""
    rng = np.random.default_rng(300 + 7 * C + mode)
    T, d = 96, 3
    q, k, v = _rand_stream(rng, T, d)
    tau = _median_tau(q, k, v, d) if mode == 0 else 0.25
    st = oracle.Stream(C, d, d, tau=tau, score_mode=mode)
    checked = 0
    for t in range(T):
        pre = st.export()
        r = st.probe(k[t], v[t])
        assert st.export()["m"] == pre["m"] and st.t == t
        I, b, j = st.step(k[t], v[t])
        assert (r["boundary"], r["merge"]) == (b, j)
        assert r["I"] == I
        if t > 0:
            assert r["thr_margin"] == pytest.approx(abs(I - tau) / tau, rel=1e-12)
        if j < 0:
            assert r["rollback_to"] == -1 and r["rollback_last"] == -1 and math.isinf(r["tie_gap"])
            continue
        n, ib = pre["n"].astype(np.int64), pre["ibar"]
        dens = [((ib[i] + ib[i + 1]) / (n[i] + n[i + 1]), i) for i in range(C - 1)]
        order = sorted(dens)
        (bd, bi), (sd, si) = order[0], order[1]
        assert j == bi and r["best"] == bd and r["runner_up"] == sd
        assert r["tie_gap"] == pytest.approx((sd - bd) / abs(bd), rel=1e-12, abs=1e-300)
        newest = max(bi, si) + 1
        assert r["rollback_to"] == int(n[:newest].sum())
        assert r["rollback_last"] == int(n[:newest + 1].sum()) - 1
        checked += 1
    assert checked >= 5


# ------------------------------------------------------------------ invariants

@pytest.mark.parametrize("mode", [0, 1])
def test_cache_invariants(mode):
    """m <= C; sum n = t; states tile [0, t) contiguously in order; the sum of
    all states is the prefix sum of the token states; Ibar_i is the sum of the
    scores of the tokens it holds; merge log only where boundary and m was C."""
    rng = np.random.default_rng(7 + mode)
    T, d, C = 160, 4, 5
    q, k, v = _rand_stream(rng, T, d)
    tau = _median_tau(q, k, v, d) if mode == 0 else 0.25
    st = oracle.Stream(C, d, d, tau=tau, score_mode=mode)
    it_all = []
    for t in range(T):
        I, b, j = st.step(k[t], v[t])
        it_all.append(I)
        ex = st.export()
        assert 1 <= ex["m"] <= C
        assert ex["n"].sum() == t + 1
        assert ex["first"][0] == 0 and ex["last"][-1] == t
        assert (ex["first"][1:] == ex["last"][:-1] + 1).all()
        assert (ex["n"] == ex["last"] - ex["first"] + 1).all()
        P = sum(np.outer(v[s], k[s]) for s in range(t + 1))
        np.testing.assert_allclose(ex["states"].sum(0), P, rtol=1e-12, atol=1e-12)
        for i in range(ex["m"]):
            seg = it_all[ex["first"][i]: ex["last"][i] + 1]
            assert ex["ibar"][i] == pytest.approx(sum(seg), rel=1e-12, abs=1e-12)
            S_i = sum(np.outer(v[s], k[s]) for s in range(ex["first"][i], ex["last"][i] + 1))
            np.testing.assert_allclose(ex["states"][i], S_i, rtol=1e-12, atol=1e-12)


def test_forward_matches_incremental_and_decode_split():
    """The batched driver equals token-by-token stepping, and a forward over T0
    tokens followed by single-token steps equals one forward over T (the decode
    step is the same recurrence, Sec. 3.1 inference rule)."""
    rng = np.random.default_rng(31)
    B, T, H, d, C = 1, 50, 2, 4, 4
    q = rng.standard_normal((B, T, H, d)); k = rng.standard_normal((B, T, H, d))
    k /= np.linalg.norm(k, axis=-1, keepdims=True)
    v = rng.standard_normal((B, T, H, d))
    lam = rng.uniform(0.5, 1.5, (B, T, H, C))
    tau = _median_tau(q[0, :, 0], k[0, :, 0], v[0, :, 0], d)
    res = oracle.forward(q, k, v, lam, tau=tau, C=C, threads=2)
    for h in range(H):
        st = oracle.Stream(C, d, d, tau=tau)
        T0 = 30
        o0, b0, m0, _ = st.run(q[0, :T0, h], k[0, :T0, h], v[0, :T0, h], lam[0, :T0, h])
        np.testing.assert_array_equal(res["o"][0, :T0, h], o0)
        for t in range(T0, T):
            I, b, j = st.step(k[0, t, h], v[0, t, h])
            o = st.readout(q[0, t, h], lam[0, t, h])
            assert b == res["boundary"][0, h, t] and j == res["merge_log"][0, h, t]
            np.testing.assert_array_equal(o, res["o"][0, t, h])
