"""The layer's transforms around the operator on the GPU (relation_layer_prep and
relation_layer_grad through the C ABI) against the fp64 oracle (oracle/layer.py), and the
whole layer (prep, Relation forward and backward, grad) against the oracles composed."""
import numpy as np
import pytest
import torch

import oracle
from oracle import layer as lay
from paper_2608_20172_gb300 import binding, workloads
from tests import parity_util as pu

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda:0")


def _inputs(B, T, H, d, dtype, seed):
    g = torch.Generator().manual_seed(seed)
    dt = torch.float32 if dtype == "fp32" else torch.bfloat16
    xs = [torch.randn((B, T, H, d), generator=g).to(dt) for _ in range(3)]
    theta = (torch.rand(H // 2, generator=g) * 6.0 - 3.0).float()
    return xs, theta


def _np(t):
    return t.double().cpu().numpy()


def _check(name, got, ref, dtype, kind):
    return pu.check(name, _np(got), ref, dtype, kind)


SHAPES = [(2, 37, 4, 64), (1, 300, 6, 48), (1, 20, 2, 128), (3, 5, 8, 16)]


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
@pytest.mark.parametrize("pairing", [0, 1])
@pytest.mark.parametrize("B,T,H,d", SHAPES)
def test_prep_matches_oracle(dtype, pairing, B, T, H, d):
    (p1, p2, info), theta = _inputs(B, T, H, d, dtype, 1)
    q, k, v = binding.layer_prep(p1.to(DEV), p2.to(DEV), info.to(DEV), theta.to(DEV), pairing)
    torch.cuda.synchronize()
    rq, rk, rv = lay.prep(_np(p1), _np(p2), _np(info), theta.double().numpy(), pairing)
    _check("q", q, rq, dtype, "out")
    _check("k", k, rk, dtype, "out")
    _check("v", v, rv, dtype, "out")


def test_prep_long_positions_fp32():
    """Positions up to 16383: the angles are reduced in fp64 (an fp32 angle m * w would be
    off by ~1e-3 rad there)."""
    (p1, p2, info), theta = _inputs(1, 16384, 2, 128, "fp32", 2)
    q, k, _ = binding.layer_prep(p1.to(DEV), p2.to(DEV), info.to(DEV), theta.to(DEV), 0)
    torch.cuda.synchronize()
    rq = lay.rope(_np(p1))
    assert float(np.max(np.abs(_np(q) - rq))) <= 2e-5
    assert float(np.max(np.abs(_np(k) - lay.rope(_np(p2))))) <= 2e-5


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
@pytest.mark.parametrize("pairing", [0, 1])
@pytest.mark.parametrize("B,T,H,d", SHAPES)
def test_grad_matches_oracle(dtype, pairing, B, T, H, d):
    (dq, dk, dv), theta = _inputs(B, T, H, d, dtype, 3)
    (info, _, _), _ = _inputs(B, T, H, d, dtype, 4)
    g1, g2, gi, gt = binding.layer_grad(dq.to(DEV), dk.to(DEV), dv.to(DEV), info.to(DEV),
                                        theta.to(DEV), pairing)
    torch.cuda.synchronize()
    r1, r2, ri, rt = lay.grad(_np(dq), _np(dk), _np(dv), _np(info), theta.double().numpy(),
                              pairing)
    _check("dp1", g1, r1, dtype, "grad")
    _check("dp2", g2, r2, dtype, "grad")
    _check("dinfo", gi, ri, dtype, "grad")
    for j in range(len(rt)):
        pu.check_dlambda(float(gt[j].item()), float(rt[j]), dtype)


def test_grad_dtheta_deterministic_and_in_place():
    (dq, dk, dv), theta = _inputs(2, 300, 8, 64, "bf16", 5)
    (info, _, _), _ = _inputs(2, 300, 8, 64, "bf16", 6)
    args = [t.to(DEV) for t in (dq, dk, dv, info)] + [theta.to(DEV)]
    a = binding.layer_grad(*args, 1)
    b = binding.layer_grad(*args, 1)
    torch.cuda.synchronize()
    for x, y in zip(a, b):
        assert torch.equal(x, y)
    # outputs over their inputs
    p1, p2, inf = (t.to(DEV) for t in (dq, dk, dv))
    ref = binding.layer_prep(p1, p2, inf, theta.to(DEV), 0)
    binding.layer_prep(p1, p2, inf, theta.to(DEV), 0, out=(p1, p2, inf))
    torch.cuda.synchronize()
    for x, y in zip(ref, (p1, p2, inf)):
        assert torch.equal(x, y)


@pytest.mark.parametrize("dtype,d,T", [("fp32", 64, 150), ("bf16", 64, 300), ("bf16", 80, 200)])
def test_whole_layer_against_composed_oracles(dtype, d, T):
    """prep -> Relation forward/backward -> grad on the GPU, against oracle/layer.py
    composed with the Relation oracle on sampled heads (and dtheta over all heads)."""
    B, H, lam = 2, 4, workloads.LAMBDA_INIT
    if not pu.kernel_available("auto", dtype, d, "fwd"):
        pytest.skip("no kernel for this head size")
    (p1, p2, info), theta = _inputs(B, T, H, d, dtype, 7)
    g = torch.Generator().manual_seed(8)
    dy = torch.randn((B, T, H, d), generator=g).to(p1.dtype)
    q, k, v = binding.layer_prep(p1.to(DEV), p2.to(DEV), info.to(DEV), theta.to(DEV), 1)
    y, lz = binding.fwd(q, k, v, lam)
    dq, dk, dv, _ = binding.bwd(q, k, v, y, dy.to(DEV), lz, lam)
    g1, g2, gi, gt = binding.layer_grad(dq, dk, dv, info.to(DEV), theta.to(DEV), 1)
    torch.cuda.synchronize()
    th = theta.double().numpy()
    rq, rk, rv = lay.prep(_np(p1), _np(p2), _np(info), th, 1)
    rdq, rdk, rdv = np.zeros_like(rq), np.zeros_like(rq), np.zeros_like(rq)
    for b in range(B):
        for h in range(H):
            yh, _ = oracle.fwd(rq[b, :, h], rk[b, :, h], rv[b, :, h], lam)
            if (b, h) in ((0, 0), (B - 1, H - 1)):
                pu.check(f"Y[{b},{h}]", y[b, :, h].double().cpu().numpy(), yh, dtype, "out")
            a, c, e, _ = oracle.bwd(rq[b, :, h], rk[b, :, h], rv[b, :, h],
                                    dy[b, :, h].double().numpy(), lam)
            rdq[b, :, h], rdk[b, :, h], rdv[b, :, h] = a, c, e
    r1, r2, ri, rt = lay.grad(rdq, rdk, rdv, _np(info), th, 1)
    _check("dp1", g1, r1, dtype, "grad")
    _check("dp2", g2, r2, dtype, "grad")
    _check("dinfo", gi, ri, dtype, "grad")
    for j in range(len(rt)):
        pu.check_dlambda(float(gt[j].item()), float(rt[j]), dtype)
