"""The oracle reproduces its stored small-case fixtures (regression guard, CPU only)."""
import json
import os

import numpy as np
import pytest

import oracle

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden",
                      "oracle_small_cases.json")
CASES = json.load(open(GOLDEN))["cases"]


@pytest.mark.parametrize("case", CASES, ids=[c["name"] for c in CASES])
def test_oracle_matches_fixture(case):
    q, k, v, g = (np.array(case[n], dtype=np.float64) for n in ("q", "k", "v", "dy"))
    y, lz = oracle.fwd(q, k, v, case["lambda"])
    np.testing.assert_allclose(y, case["Y"], rtol=1e-13, atol=1e-15)
    np.testing.assert_allclose(lz, case["logZ"], rtol=1e-13, atol=1e-15)
    dq, dk, dv, dl = oracle.bwd(q, k, v, g, case["lambda"])
    for name, x in (("dq", dq), ("dk", dk), ("dv", dv)):
        np.testing.assert_allclose(x, case[name], rtol=1e-12, atol=1e-14)
    assert abs(dl - case["dlambda"]) <= 1e-12 * max(1.0, abs(case["dlambda"]))


GOLDEN2 = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden",
                       "linear_layer_small_cases.json")
FIX2 = json.load(open(GOLDEN2))


@pytest.mark.parametrize("case", FIX2["linear"], ids=[c["name"] for c in FIX2["linear"]])
def test_linear_oracle_matches_fixture(case):
    lo = oracle.linear()
    p1, p2, v, a, dy = (np.array(case[n], dtype=np.float64)
                        for n in ("p1", "p2", "v", "alpha", "dy"))
    y, S = lo.fwd(p1, p2, v, a)
    np.testing.assert_allclose(y, case["Y"], rtol=1e-13, atol=1e-15)
    np.testing.assert_allclose(S, case["S"], rtol=1e-13, atol=1e-15)
    for name, x in zip(("dp1", "dp2", "dv", "dalpha"), lo.bwd(p1, p2, v, a, dy)):
        np.testing.assert_allclose(x, case[name], rtol=1e-12, atol=1e-14)


@pytest.mark.parametrize("case", FIX2["layer"], ids=[c["name"] for c in FIX2["layer"]])
def test_layer_oracle_matches_fixture(case):
    from oracle import layer
    arr = {n: np.array(case[n], dtype=np.float64)
           for n in ("p1", "p2", "info", "dq", "dk", "dv", "theta")}
    q, k, v = layer.prep(arr["p1"], arr["p2"], arr["info"], arr["theta"], case["pairing"])
    for name, x in (("q", q), ("k", k), ("v", v)):
        np.testing.assert_allclose(x, case[name], rtol=1e-13, atol=1e-15)
    g = layer.grad(arr["dq"], arr["dk"], arr["dv"], arr["info"], arr["theta"], case["pairing"])
    for name, x in zip(("dp1", "dp2", "dinfo", "dtheta"), g):
        np.testing.assert_allclose(x, case[name], rtol=1e-12, atol=1e-14)
