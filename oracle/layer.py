"""fp64 CPU oracle of the two transforms the paper's layer applies around the operator:
RoPE on the relation coordinates P1, P2 and the Givens mixing of the information states.

TEST INFRASTRUCTURE ONLY (like the rest of this package): only the test suite,
``__graft_entry__.smoke()`` and the benchmark's CPU-baseline leg may use it, and it shares
nothing with the CUDA library.

Definitions followed (plain numpy, fp64, arrays [B, T, H, d] with d the fastest index):

* RoPE (Sec. 3.1 and App. B.3: full-head rotary embedding of P1 and P2, base 10^4, no
  positional scaling; the rotary form itself is RoFormer's).  Channel pairs (2c, 2c + 1),
  c = 0 .. d/2 - 1, of the row at position m are rotated by the angle m * base^(-2c/d):
      x'_{2c}   = x_{2c} cos(a) - x_{2c+1} sin(a)
      x'_{2c+1} = x_{2c} sin(a) + x_{2c+1} cos(a).
  Readings (the paper names neither): interleaved pairs as in RoFormer, and zero-based
  positions restarting at every sequence.  The choice of origin does not change the
  evidence U = Q K^T, which depends on positions only through their differences.
* Givens mixing (Sec. 3.2, Eq. givens-rotation, App. A.2.2).  Heads are paired, and each
  pair (a, b) with angle theta is mixed on every information channel:
      I~_a = cos(theta) I_a - sin(theta) I_b,   I~_b = sin(theta) I_a + cos(theta) I_b.
  Pairing A: (0, 1), (2, 3), ..., (H - 2, H - 1); pairing B: (1, 2), (3, 4), ...,
  (H - 1, 0) (zero-based heads; the paper's one-based sets M_A and M_B).  Pair k takes
  theta[k]; H is even.
* Gradients: the transposed rotations for dP1, dP2 and dI, and
      dtheta_k = sum over (b, t, channels) of
                 dI~_a * (-sin I_a - cos I_b) + dI~_b * (cos I_a - sin I_b).
"""
from __future__ import annotations

import numpy as np

ROPE_BASE = 1.0e4


def rope_angles(T: int, d: int, base: float = ROPE_BASE) -> np.ndarray:
    """[T, d/2] rotation angles m * base^(-2c/d)."""
    m = np.arange(T, dtype=np.float64)[:, None]
    c = np.arange(d // 2, dtype=np.float64)[None, :]
    return m * base ** (-2.0 * c / d)


def rope(x: np.ndarray, base: float = ROPE_BASE, inverse: bool = False) -> np.ndarray:
    """RoPE of x [B, T, H, d] (or its transpose, the rotation by minus the angle)."""
    x = np.asarray(x, dtype=np.float64)
    B, T, H, d = x.shape
    a = rope_angles(T, d, base)[None, :, None, :]
    cs, sn = np.cos(a), np.sin(a)
    if inverse:
        sn = -sn
    xe, xo = x[..., 0::2], x[..., 1::2]
    out = np.empty_like(x)
    out[..., 0::2] = xe * cs - xo * sn
    out[..., 1::2] = xe * sn + xo * cs
    return out


def pairs(H: int, pairing: int):
    """The head pairs (a, b) of pairing A (0) or B (1), in angle order."""
    if H % 2:
        raise ValueError("Givens mixing pairs the heads: H must be even")
    if pairing == 0:
        return [(2 * k, 2 * k + 1) for k in range(H // 2)]
    return [(2 * k + 1, (2 * k + 2) % H) for k in range(H // 2)]


def givens(info: np.ndarray, theta, pairing: int) -> np.ndarray:
    """Mixed information states I~ of info [B, T, H, d]."""
    info = np.asarray(info, dtype=np.float64)
    out = np.empty_like(info)
    for k, (a, b) in enumerate(pairs(info.shape[2], pairing)):
        c, s = np.cos(theta[k]), np.sin(theta[k])
        out[:, :, a] = c * info[:, :, a] - s * info[:, :, b]
        out[:, :, b] = s * info[:, :, a] + c * info[:, :, b]
    return out


def givens_grad(dmix: np.ndarray, info: np.ndarray, theta, pairing: int):
    """(dI, dtheta) from dI~ = dmix."""
    dmix = np.asarray(dmix, dtype=np.float64)
    info = np.asarray(info, dtype=np.float64)
    dinfo = np.empty_like(info)
    dtheta = np.zeros(len(theta))
    for k, (a, b) in enumerate(pairs(info.shape[2], pairing)):
        c, s = np.cos(theta[k]), np.sin(theta[k])
        ga, gb = dmix[:, :, a], dmix[:, :, b]
        dinfo[:, :, a] = c * ga + s * gb
        dinfo[:, :, b] = -s * ga + c * gb
        ia, ib = info[:, :, a], info[:, :, b]
        dtheta[k] = np.sum(ga * (-s * ia - c * ib)) + np.sum(gb * (c * ia - s * ib))
    return dinfo, dtheta


def prep(p1, p2, info, theta, pairing: int, base: float = ROPE_BASE):
    """(Q, K, V) = (RoPE(P1), RoPE(P2), Givens(I)): the operator's inputs."""
    return rope(p1, base), rope(p2, base), givens(info, theta, pairing)


def grad(dq, dk, dv, info, theta, pairing: int, base: float = ROPE_BASE):
    """(dP1, dP2, dI, dtheta) from the operator's (dQ, dK, dV)."""
    dinfo, dtheta = givens_grad(dv, info, theta, pairing)
    return rope(dq, base, inverse=True), rope(dk, base, inverse=True), dinfo, dtheta
