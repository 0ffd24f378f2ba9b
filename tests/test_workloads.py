"""Host-side checks of the seeded workloads and the decision-safe generator."""
import dataclasses
import importlib.util
import os

import numpy as np
import pytest

import oracle
from paper_2606_10650_gb300 import workloads as W
from safe_inputs import THR_MARGIN, TIE_MARGIN, safe_stream

HERE = os.path.dirname(os.path.abspath(__file__))


def test_stream_generator_is_reproducible_and_per_stream():
    w = W.get("standard", T=64)
    a = W.StreamGen(w, 1, 3).tokens()
    b = W.StreamGen(w, 1, 3).tokens()
    c = W.StreamGen(w, 1, 4).tokens()
    for x, y in zip(a, b):
        np.testing.assert_array_equal(x, y)
    assert not np.array_equal(a[1], c[1])
    q, k, v, lam = W.host_batch(dataclasses.replace(w, B=2, H=5))
    np.testing.assert_array_equal(q[1, :, 3], a[0])
    np.testing.assert_array_equal(k[1, :, 3], a[1])


def test_values_are_exact_in_input_dtype():
    import torch
    w = W.get("standard", T=32)
    q, k, v = W.StreamGen(w, 0, 0).tokens()
    for x in (q, k, v):
        t = torch.from_numpy(x.astype(np.float32)).to(torch.bfloat16).double().numpy()
        np.testing.assert_array_equal(t, x)
    w1 = W.get("tiny", T=16)
    q, k, v = W.StreamGen(w1, 0, 0).tokens()
    np.testing.assert_array_equal(q.astype(np.float32).astype(np.float64), q)


def test_regime_workload_shape_of_regimes():
    w = W.get("regime")
    g = W.StreamGen(w, 0, 0)
    lens = np.diff(np.flatnonzero(np.diff(np.r_[-1, g.seg]) != 0))
    assert 150 < lens.mean() < 400  # Geometric(mean 256)


@pytest.mark.parametrize("name,T", [("tiny", 512), ("standard", 1024), ("regime", 2048), ("long", 1024)])
def test_safe_stream_margins_hold_in_a_fresh_oracle_pass(name, T):
    """The accepted tokens keep every score >= 1e-3 (relative) away from tau and
    every merge's best pair >= TIE_MARGIN away from the runner-up, when the
    final stream is replayed from scratch."""
    w = W.get(name)
    if name == "long":  # start inside an i.i.d. block that fires on every token
        w = dataclasses.replace(w, block=512)
    r = safe_stream(w, 0, 1, T=T)
    st = oracle.Stream(w.C, w.d, w.d, w.tau, w.eps, w.rms_eps)
    merges = 0
    for t in range(T):
        p = st.probe(r["k"][t], r["v"][t])
        assert p["thr_margin"] >= THR_MARGIN
        if p["merge"] >= 0:
            merges += 1
            assert p["tie_gap"] >= TIE_MARGIN
        st.step(r["k"][t], r["v"][t])
    if name in ("tiny", "long"):
        assert merges > 10


def test_calibration_script_reproduces_constants():
    spec = importlib.util.spec_from_file_location("calib", os.path.join(HERE, "golden", "calibrate_workloads.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    res = mod.rounded(mod.calibrate())
    for name, consts in res.items():
        w = W.get(name)
        for key, val in consts.items():
            assert getattr(w, key) == pytest.approx(val, rel=1e-8), (name, key)
