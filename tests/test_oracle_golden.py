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
