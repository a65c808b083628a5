"""Write tests/golden/oracle_small_cases.json (and linear_layer_small_cases.json) from the
fp64 oracles only.

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
    write_linear_and_layer()


LINEAR_CASES = [
    # (name, T, d, seed): retention alpha in [0.3, 1)
    ("lin_T1_d3", 1, 3, 201),
    ("lin_T5_d4", 5, 4, 202),
    ("lin_T9_d2", 9, 2, 203),
]

LAYER_CASES = [
    # (name, B, T, H, d, pairing, seed)
    ("layer_A_T5_H4_d4", 1, 5, 4, 4, 0, 301),
    ("layer_B_T3_H6_d2", 2, 3, 6, 2, 1, 302),
]


def write_linear_and_layer():
    """Fixtures of the Linear Relation oracle (Sec. 5.2, App. A.4) and of the layer
    transforms (RoPE, Givens mixing; Sec. 3.1-3.2, App. A.2.2, App. B.3)."""
    from oracle import layer
    lo = oracle.linear()
    out = {"source": "fp64 oracles (oracle/linear_oracle.c, oracle/layer.py); tau_S = 2, "
                     "RoPE base 1e4",
           "citation": "Sec. 5.2, App. A.4; Sec. 3.1-3.2, Eq. (givens-rotation), App. B.3",
           "linear": [], "layer": []}
    for name, T, d, seed in LINEAR_CASES:
        rs = np.random.default_rng(seed)
        p1, p2, v, dy = (np.round(rs.standard_normal((T, d)), 3) for _ in range(4))
        a = np.round(rs.uniform(0.3, 1.0, (T, d)), 3)
        y, S = lo.fwd(p1, p2, v, a)
        g1, g2, gv, ga = lo.bwd(p1, p2, v, a, dy)
        out["linear"].append({
            "name": name, "p1": p1.tolist(), "p2": p2.tolist(), "v": v.tolist(),
            "alpha": a.tolist(), "dy": dy.tolist(), "Y": y.tolist(), "S": S.tolist(),
            "dp1": g1.tolist(), "dp2": g2.tolist(), "dv": gv.tolist(), "dalpha": ga.tolist()})
    for name, B, T, H, d, pairing, seed in LAYER_CASES:
        rs = np.random.default_rng(seed)
        p1, p2, info, dq, dk, dv = (np.round(rs.standard_normal((B, T, H, d)), 3)
                                    for _ in range(6))
        theta = np.round(rs.uniform(-3.0, 3.0, H // 2), 3)
        q, k, vv = layer.prep(p1, p2, info, theta, pairing)
        g1, g2, gi, gt = layer.grad(dq, dk, dv, info, theta, pairing)
        out["layer"].append({
            "name": name, "pairing": pairing, "theta": theta.tolist(), "p1": p1.tolist(),
            "p2": p2.tolist(), "info": info.tolist(), "dq": dq.tolist(), "dk": dk.tolist(),
            "dv": dv.tolist(), "q": q.tolist(), "k": k.tolist(), "v": vv.tolist(),
            "dp1": g1.tolist(), "dp2": g2.tolist(), "dinfo": gi.tolist(),
            "dtheta": gt.tolist()})
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)),
                        "linear_layer_small_cases.json")
    with open(path, "w") as f:
        json.dump(out, f, indent=1)
        f.write("\n")
    print("wrote", path)


if __name__ == "__main__":
    main()
