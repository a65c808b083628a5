"""Seeded synthetic workloads for the causal Relation operator.

This module only draws random numbers and names shapes; it holds none of the
operator's arithmetic.  The test suite, the benchmark and the oracle checks all
take their inputs from here, so the CUDA path and the fp64 oracle always see the
same values.

Recipe: a CPU ``torch.Generator`` seeded with ``seed`` draws, in this order, Q, K, V
and dO as fp32 normals of shape [B, T, H, d_h]; Q and K are then scaled by the
workload's ``qk_std`` (and V by ``v_std``) and every tensor is cast to the run's
dtype.  The oracle receives the cast values widened to fp64.

Workloads (shapes of the paper's ~10M/30M/100M decoder layers, Table 2 and
App. B.1, plus a long-context stress case); all are causal with lambda = 0.5 (the
initial value the paper gives lambda_l, App. A.1.1) and tau_S = 2 (Sec. 3.1):
  tiny : B=1,  H=2,  T=128,   d=32,  fp32, Q,K ~ N(0,1)/sqrt(d), V,dO ~ N(0,1)
  10M  : B=32, H=4,  T=1024,  d=64,  bf16, all N(0,1)
  30M  : B=16, H=6,  T=2048,  d=64,  bf16, all N(0,1)
  100M : B=8,  H=12, T=2048,  d=64,  bf16, all N(0,1)
  long : B=2,  H=16, T=16384, d=128, bf16, Q,K ~ N(0, variance 2), V,dO ~ N(0,1)
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import torch

LAMBDA_INIT = 0.5
TAU_S = 2.0


@dataclass(frozen=True)
class Workload:
    name: str
    B: int
    H: int
    T: int
    d: int
    dtype: str          # "fp32" or "bf16"
    qk_std: float       # standard deviation of Q and K entries
    v_std: float = 1.0  # standard deviation of V entries
    description: str = ""

    @property
    def torch_dtype(self) -> torch.dtype:
        return torch.float32 if self.dtype == "fp32" else torch.bfloat16

    @property
    def tokens(self) -> int:
        return self.B * self.T

    def causal_pairs(self) -> int:
        """Number of (i, j <= i) pairs over all heads."""
        return self.B * self.H * self.T * (self.T + 1) // 2

    def flops_fwd(self) -> float:
        """Causal FLOP count of the forward, FlashAttention convention: 2 B H T^2 d."""
        return 2.0 * self.B * self.H * self.T * self.T * self.d

    def flops_fwd_bwd(self) -> float:
        """Causal FLOP count of forward + backward (backward = 2.5 x forward): 7 B H T^2 d."""
        return 7.0 * self.B * self.H * self.T * self.T * self.d


WORKLOADS = {
    "tiny": Workload("tiny", 1, 2, 128, 32, "fp32", 1.0 / math.sqrt(32),
                     description="Tiny MHR fp32 (B=1,H=2,T=128,d=32)"),
    "10M": Workload("10M", 32, 4, 1024, 64, "bf16", 1.0,
                    description="~10M-scale decoder layer bf16 (B=32,H=4,T=1024,d=64)"),
    "30M": Workload("30M", 16, 6, 2048, 64, "bf16", 1.0,
                    description="~30M-scale decoder layer bf16 (B=16,H=6,T=2048,d=64)"),
    "100M": Workload("100M", 8, 12, 2048, 64, "bf16", 1.0,
                     description="~100M-scale decoder layer bf16 (B=8,H=12,T=2048,d=64)"),
    "long": Workload("long", 2, 16, 16384, 128, "bf16", math.sqrt(2.0),
                     description="long-context stress bf16 (B=2,H=16,T=16384,d=128), Q,K variance 2"),
}


def custom(B: int, H: int, T: int, d: int, dtype: str = "bf16", qk_std: float = 1.0,
           v_std: float = 1.0) -> Workload:
    """An ad-hoc workload with the same recipe (used for ragged and edge-case tests)."""
    return Workload(f"custom_{B}x{H}x{T}x{d}_{dtype}", B, H, T, d, dtype, qk_std, v_std)


def make_linear_inputs(w: Workload, seed: int = 0):
    """Linear Relation inputs on the CPU: p1, p2, v [B, T, H, d] of the workload's dtype
    (p1, p2 ~ N(0, qk_std^2), v ~ N(0, v_std^2)), the retention alpha [B, T, H, d] fp32 and
    dY ~ N(0, 1).  alpha follows a KDA-style draw, alpha = exp(-A softplus(z - 4)) with a
    per-(head, channel) rate A ~ U(1, 16) and z ~ N(0, 1) per token, which puts most
    channels between 0.75 and 0.99."""
    g = torch.Generator().manual_seed(seed + 7919)
    shape = (w.B, w.T, w.H, w.d)
    dt = torch.float32 if w.dtype == "fp32" else torch.bfloat16
    p1 = (torch.randn(shape, generator=g) * w.qk_std).to(dt)
    p2 = (torch.randn(shape, generator=g) * w.qk_std).to(dt)
    v = (torch.randn(shape, generator=g) * w.v_std).to(dt)
    A = torch.rand((1, 1, w.H, w.d), generator=g) * 15.0 + 1.0
    z = torch.randn(shape, generator=g)
    alpha = torch.exp(-A * torch.nn.functional.softplus(z - 4.0)).float()
    dy = torch.randn(shape, generator=g).to(dt)
    return p1, p2, v, alpha, dy


def make_inputs(w: Workload, seed: int = 0, with_grad_out: bool = True):
    """Draw (q, k, v, dout) on the CPU as [B, T, H, d] tensors of the workload's dtype.

    dout is None when ``with_grad_out`` is False (it is still drawn, to keep the
    stream of random numbers identical)."""
    g = torch.Generator(device="cpu")
    g.manual_seed(seed)
    shape = (w.B, w.T, w.H, w.d)
    q = torch.randn(shape, generator=g, dtype=torch.float32)
    k = torch.randn(shape, generator=g, dtype=torch.float32)
    v = torch.randn(shape, generator=g, dtype=torch.float32)
    do = torch.randn(shape, generator=g, dtype=torch.float32)
    if w.qk_std != 1.0:
        q.mul_(w.qk_std)
        k.mul_(w.qk_std)
    if w.v_std != 1.0:
        v.mul_(w.v_std)
    dt = w.torch_dtype
    out = (q.to(dt), k.to(dt), v.to(dt))
    return out + ((do.to(dt) if with_grad_out else None),)
