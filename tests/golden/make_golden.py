"""Write tests/golden/oracle_small_cases.json from the fp64 oracle only.

The stored values are regression fixtures of the oracle itself (they are not the
paper's: the paper prints no operator values).  Each case lists its inputs
explicitly, so the fixture is self-contained.  Outputs: Y and logZ of the forward
(Eq. causal-relation, Eq. relation-flow) and dP1, dP2, dI~, dlambda of the backward
(App. A.1.7) for L = sum(Y * G).

Run from the repository root:  python tests/golden/make_golden.py
"""
import json
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)
import oracle  # noqa: E402

CASES = [
    # (name, T, d, lambda, seed)
    ("T1_d3", 1, 3, 0.5, 101),
    ("T2_d2", 2, 2, 0.5, 102),
    ("T5_d4_lam0", 5, 4, 0.0, 103),
    ("T6_d3_negative_lambda", 6, 3, -1.0, 104),
    ("T7_d2_large_lambda", 7, 2, 3.0, 105),
]


def main():
    out = {"source": "fp64 oracle (oracle/relation_oracle.c); tau_S = 2",
           "citation": "Eq. (causal-relation), Eq. (relation-flow), App. A.1.7", "cases": []}
    for name, T, d, lam, seed in CASES:
        rs = np.random.default_rng(seed)
        q, k, v, g = (np.round(rs.standard_normal((T, d)), 3) for _ in range(4))
        y, lz = oracle.fwd(q, k, v, lam)
        dq, dk, dv, dl = oracle.bwd(q, k, v, g, lam)
        out["cases"].append({
            "name": name, "lambda": lam, "q": q.tolist(), "k": k.tolist(), "v": v.tolist(),
            "dy": g.tolist(), "Y": y.tolist(), "logZ": lz.tolist(), "dq": dq.tolist(),
            "dk": dk.tolist(), "dv": dv.tolist(), "dlambda": dl})
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "oracle_small_cases.json")
    with open(path, "w") as f:
        json.dump(out, f, indent=1)
        f.write("\n")
    print("wrote", path)


if __name__ == "__main__":
    main()
