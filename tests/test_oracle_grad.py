"""Pins of the hard-decision gradient oracle (oracle/grad.py) against the
recurrent fp64 oracle: the dense form of the read-out equals the oracle's
outputs, the replayed slots equal the oracle's cache, and the gradients equal
central finite differences of the oracle's forward pass wherever the
perturbation leaves every decision unchanged (the loss is linear in each single
coordinate of q, k, v and lambda once the decisions are fixed, so central
differences are exact up to rounding)."""
import numpy as np
import pytest

import oracle
from oracle import grad

pytestmark = pytest.mark.filterwarnings("ignore")


def _stream(seed, T=28, d=3, C=3):
    rng = np.random.default_rng(seed)
    q = rng.standard_normal((T, d))
    k = rng.standard_normal((T, d))
    k /= np.linalg.norm(k, axis=1, keepdims=True)
    v = rng.standard_normal((T, d))
    lam = rng.uniform(0.5, 1.5, size=(T, C))
    probe = oracle.Stream(2, d, d, tau=1e300)
    _, _, _, it = probe.run(q, k, v)
    tau = float(np.median(it[1:]))  # about half the tokens open a state: plenty of merges at C = 3
    g = rng.standard_normal((T, d))
    return q, k, v, lam, tau, g


def _run(q, k, v, lam, tau, C):
    st = oracle.Stream(C, q.shape[1], v.shape[1], tau=tau)
    o, bnd, ml, _ = st.run(q, k, v, lam)
    return o, bnd, ml, st.export()


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_dense_readout_equals_recurrent_oracle(seed):
    q, k, v, lam, tau, _ = _stream(seed)
    o, bnd, ml, _ = _run(q, k, v, lam, tau, 3)
    assert (ml >= 0).sum() >= 3  # merges are exercised
    W = grad.weights(bnd, ml, lam)
    np.testing.assert_allclose(grad.readout_dense(q, k, v, W), o, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_replayed_slots_match_the_oracle_cache(seed):
    q, k, v, lam, tau, _ = _stream(seed)
    _, bnd, ml, ex = _run(q, k, v, lam, tau, 3)
    slot = grad.token_slots(bnd, ml)
    T = q.shape[0]
    counts = np.bincount(slot[T - 1], minlength=ex["m"])
    assert counts.tolist() == ex["n"][: ex["m"]].tolist()
    # every state after every token holds a contiguous, chronological range of tokens
    for t in range(T):
        assert (np.diff(slot[t, : t + 1]) >= 0).all() and slot[t, t] == slot[t].max()


@pytest.mark.parametrize("seed", [0, 1])
def test_gradients_match_central_differences(seed):
    q, k, v, lam, tau, g = _stream(seed, T=20)
    C = 3
    o, bnd, ml, _ = _run(q, k, v, lam, tau, C)
    gr = grad.readout_grads(q, k, v, lam, bnd, ml, g)
    eps = 1e-5

    def loss(q_, k_, v_, lam_):
        o_, b_, m_, _ = _run(q_, k_, v_, lam_, tau, C)
        return float((g * o_).sum()), np.array_equal(b_, bnd) and np.array_equal(m_, ml)

    checked = 0
    for name, arr, key in (("q", q, "dq"), ("k", k, "dk"), ("v", v, "dv"), ("lam", lam, "dlam")):
        for idx in np.ndindex(arr.shape):
            args = {"q": q, "k": k, "v": v, "lam": lam}
            hi, lo = arr.copy(), arr.copy()
            hi[idx] += eps
            lo[idx] -= eps
            args[name] = hi
            lh, same_h = loss(args["q"], args["k"], args["v"], args["lam"])
            args[name] = lo
            ll, same_l = loss(args["q"], args["k"], args["v"], args["lam"])
            if not (same_h and same_l):
                continue  # a decision flipped: the hard-decision gradient does not describe this step
            fd = (lh - ll) / (2 * eps)
            assert fd == pytest.approx(gr[key][idx], rel=1e-6, abs=1e-8), (name, idx)
            checked += 1
    assert checked >= 0.9 * (q.size + k.size + v.size + lam.size)


@pytest.mark.parametrize("seed", [0, 1, 2])
@pytest.mark.parametrize("with_lam", [True, False])
def test_sampled_gradients_equal_the_dense_ones(seed, with_lam):
    """The row / column evaluation for long sequences (readout_grads_sampled)
    equals the dense gradients at every sampled token, with and without
    lambda, on streams with merges."""
    q, k, v, lam, tau, g = _stream(seed, T=40)
    lam_use = lam if with_lam else None
    _, bnd, ml, _ = _run(q, k, v, lam, tau, 3)
    assert (ml >= 0).sum() > 3
    full = grad.readout_grads(q, k, v, lam_use, bnd, ml, g)
    rows = [0, 1, 7, 20, 39]
    cols = [0, 5, 19, 38, 39]
    s = grad.readout_grads_sampled(q, k, v, lam_use, bnd, ml, g, rows, cols)
    np.testing.assert_allclose(s["dq"], full["dq"][rows], rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(s["dk"], full["dk"][cols], rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(s["dv"], full["dv"][cols], rtol=1e-12, atol=1e-12)
    if with_lam:
        np.testing.assert_allclose(s["dlam"], full["dlam"][rows], rtol=1e-12, atol=1e-12)
    else:
        assert s["dlam"] is None


@pytest.mark.parametrize("seed", [0, 1, 2, 3])
@pytest.mark.parametrize("with_lam", [True, False])
def test_linear_time_gradients_equal_the_dense_ones(seed, with_lam):
    """The two-sweep form (forward states for dq and dlambda, reverse adjoint
    states through the undone merges for dk and dv) equals the dense form on
    streams with merges, with and without lambda."""
    q, k, v, lam, tau, g = _stream(seed, T=40)
    lam_use = lam if with_lam else None
    _, bnd, ml, _ = _run(q, k, v, lam, tau, 3)
    assert (ml >= 0).sum() > 3
    full = grad.readout_grads(q, k, v, lam_use, bnd, ml, g)
    lin = grad.readout_grads_linear(q, k, v, lam_use, bnd, ml, g)
    for key in ("dq", "dk", "dv"):
        np.testing.assert_allclose(lin[key], full[key], rtol=1e-11, atol=1e-11)
    if with_lam:
        np.testing.assert_allclose(lin["dlam"], full["dlam"], rtol=1e-11, atol=1e-11)
