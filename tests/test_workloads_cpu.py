"""The seeded input recipe (paper_2608_20172_gb300/workloads.py): shapes, dtypes, the
value distributions each workload states, determinism, and the flop convention.  CPU
only, on the small workloads or small custom shapes."""
import math

import pytest
import torch

from paper_2608_20172_gb300 import workloads


def test_workload_table():
    W = workloads.WORKLOADS
    assert (W["10M"].B, W["10M"].H, W["10M"].T, W["10M"].d, W["10M"].dtype) == (32, 4, 1024, 64, "bf16")
    assert (W["30M"].B, W["30M"].H, W["30M"].T, W["30M"].d) == (16, 6, 2048, 64)
    assert (W["100M"].B, W["100M"].H, W["100M"].T, W["100M"].d) == (8, 12, 2048, 64)
    assert (W["long"].B, W["long"].H, W["long"].T, W["long"].d) == (2, 16, 16384, 128)
    assert W["long"].qk_std == pytest.approx(math.sqrt(2.0))  # variance 2
    assert W["tiny"].dtype == "fp32" and W["tiny"].qk_std == pytest.approx(1 / math.sqrt(32))
    assert workloads.LAMBDA_INIT == 0.5 and workloads.TAU_S == 2.0


def test_flop_convention():
    w = workloads.WORKLOADS["10M"]
    assert w.flops_fwd() == 2.0 * 32 * 4 * 1024 ** 2 * 64
    assert w.flops_fwd_bwd() == pytest.approx(3.5 * w.flops_fwd())
    assert w.causal_pairs() == 32 * 4 * 1024 * 1025 // 2


def test_inputs_are_seeded_and_shaped():
    w = workloads.custom(2, 3, 40, 16, "bf16")
    a = workloads.make_inputs(w, seed=5)
    b = workloads.make_inputs(w, seed=5)
    c = workloads.make_inputs(w, seed=6)
    for x, y, z in zip(a, b, c):
        assert x.shape == (2, 40, 3, 16) and x.dtype == torch.bfloat16
        assert torch.equal(x, y) and not torch.equal(x, z)
    # the draw order Q, K, V, dO: dO is drawn even when it is not returned
    q2, k2, v2, none = workloads.make_inputs(w, seed=5, with_grad_out=False)
    assert none is None and torch.equal(q2, a[0]) and torch.equal(v2, a[2])


def test_value_distributions():
    w = workloads.custom(4, 4, 512, 64, "fp32", qk_std=math.sqrt(2.0))
    q, k, v, do = workloads.make_inputs(w)
    assert abs(q.var().item() - 2.0) < 0.05 and abs(k.var().item() - 2.0) < 0.05
    assert abs(v.var().item() - 1.0) < 0.03 and abs(do.var().item() - 1.0) < 0.03
    assert abs(q.mean().item()) < 0.02
    t = workloads.WORKLOADS["tiny"]
    tq, _, tv, _ = workloads.make_inputs(t)
    assert abs(tq.std().item() - 1 / math.sqrt(32)) < 0.01 and abs(tv.std().item() - 1.0) < 0.03


def test_linear_inputs():
    w = workloads.custom(2, 4, 64, 32, "bf16")
    p1, p2, v, alpha, dy = workloads.make_linear_inputs(w, seed=0)
    for x in (p1, p2, v, dy):
        assert x.shape == (2, 64, 4, 32) and x.dtype == torch.bfloat16
    assert alpha.dtype == torch.float32 and alpha.shape == p1.shape
    assert (alpha > 0).all() and (alpha <= 1).all()
    # most channels retain between 0.75 and 0.99 per token
    frac = ((alpha > 0.75) & (alpha < 0.99)).float().mean().item()
    assert frac > 0.5
    again = workloads.make_linear_inputs(w, seed=0)
    assert all(torch.equal(x, y) for x, y in zip((p1, p2, v, alpha, dy), again))
