"""fp64 chunked (block-parallel) evaluation of the Linear Relation forward (Sec. 5.2,
App. A.4): the same operator as ``linear_oracle.c``'s recurrence, regrouped so that most
of the work is dense products over blocks of L tokens.

TEST INFRASTRUCTURE ONLY (like the rest of this package).  The paper states the
recurrence only; this regrouping is derived from it (tests pin it to the recurrent
oracle), and gives a reference for the intermediate quantities of a block-parallel
kernel.

Per head, with q'_t = S_t ^p1_t and k'_t = S_t ^p2_t (Ask Self folded into the unit
coordinates, as in the recurrence), I~_t the information and alpha_t the retention,
inside a block of tokens t = 1..L that starts from the state C_0:
    a_t = alpha_1 * ... * alpha_t                       (channel-wise, a_0 = 1)
    C^-_t = Diag(a_t) C_0 + sum_{j<t} Diag(a_t / a_j) k'_j I~_j^T
so that, with Qb_t = a_t * q'_t and Kb_j = k'_j / a_j,
    E_t = C_0^T Qb_t + sum_{j<t} (Qb_t . Kb_j) I~_j          (inter-block + intra-block)
    Y_t = I~_t + E_t
    C_L = Diag(a_L) C_0 + sum_j (a_L * Kb_j) I~_j^T          (the state handed on).
The division by a_j needs retention bounded away from zero over a block (a_L within the
fp64 range); a kernel would form the ratios a_t / a_j in log space or in sub-blocks.
"""
from __future__ import annotations

import numpy as np


def _self_coords(p1, p2, tau_s):
    d = p1.shape[1]
    S = 1.0 / (1.0 + np.exp(-np.sum(p1 * p2, axis=1) / (tau_s * np.sqrt(d))))
    q = S[:, None] * p1 / np.linalg.norm(p1, axis=1, keepdims=True)
    k = S[:, None] * p2 / np.linalg.norm(p2, axis=1, keepdims=True)
    return S, q, k


def linear_fwd_chunked(p1, p2, v, alpha, L: int, tau_s: float = 2.0):
    """Y [T, d] and the final state C [d, d] (rows: coordinate side, columns: information
    side) of one head, evaluated block by block with blocks of L tokens."""
    p1, p2, v, alpha = (np.asarray(x, dtype=np.float64) for x in (p1, p2, v, alpha))
    T, d = p1.shape
    _, q, k = _self_coords(p1, p2, tau_s)
    C = np.zeros((d, d))
    Y = np.empty((T, d))
    for t0 in range(0, T, L):
        sl = slice(t0, min(T, t0 + L))
        a = np.cumprod(alpha[sl], axis=0)          # a_t within the block
        Qb = a * q[sl]
        Kb = k[sl] / a
        A = np.tril(Qb @ Kb.T, -1)                 # strictly earlier tokens of the block
        Y[sl] = v[sl] + Qb @ C + A @ v[sl]         # Answer: I~ + inter + intra
        C = a[-1][:, None] * C + (a[-1] * Kb).T @ v[sl]  # the state handed on
    return Y, C


def linear_bwd_chunked(p1, p2, v, alpha, dy, L: int, tau_s: float = 2.0):
    """(dp1, dp2, dv, dalpha) of L = sum(dy * Y) for the forward above, by reverse mode
    through the block form, last block first, with dC the adjoint of the state a block
    hands on.  Per block (C_0 the entering state, A = tril(Qb Kb^T, -1), Ka = a_L * Kb):
        dI~  = dY + A^T dY + Ka dC
        dA   = tril(dY I~^T, -1)
        dQb  = dA Kb + dY C_0^T,      dKb = dA^T Qb + a_L * (I~ dC^T)
        dC_0 = Qb^T dY + Diag(a_L) dC
        da_t = dQb_t * q'_t - dKb_t * k'_t / a_t^2   (+ for t = L the state's a_L terms)
        dalpha_u = sum_{t >= u} da_t * a_t / alpha_u
    then dq' = a * dQb, dk' = dKb / a, and (dp1, dp2) through S and the normalisation."""
    p1, p2, v, alpha, dy = (np.asarray(x, dtype=np.float64) for x in (p1, p2, v, alpha, dy))
    T, d = p1.shape
    S, q, k = _self_coords(p1, p2, tau_s)
    # forward: the state entering every block
    C = np.zeros((d, d))
    starts = list(range(0, T, L))
    C_in = []
    for t0 in starts:
        sl = slice(t0, min(T, t0 + L))
        a = np.cumprod(alpha[sl], axis=0)
        Kb = k[sl] / a
        C_in.append(C)
        C = a[-1][:, None] * C + (a[-1] * Kb).T @ v[sl]
    dq, dk, dv, dal = (np.zeros((T, d)) for _ in range(4))
    dC = np.zeros((d, d))
    for t0, C0 in zip(reversed(starts), reversed(C_in)):
        sl = slice(t0, min(T, t0 + L))
        a = np.cumprod(alpha[sl], axis=0)
        qs, ks, I, g = q[sl], k[sl], v[sl], dy[sl]
        Qb, Kb = a * qs, ks / a
        A = np.tril(Qb @ Kb.T, -1)
        aL = a[-1]
        Ka = aL * Kb
        dv[sl] = g + A.T @ g + Ka @ dC
        dA = np.tril(g @ I.T, -1)
        dQb = dA @ Kb + g @ C0.T
        dKb = dA.T @ Qb + aL * (I @ dC.T)
        da = dQb * qs - dKb * ks / (a * a)
        # C_L[c, :] = a_L[c] (C_0[c, :] + sum_t Kb_t[c] I~_t): the a_L factor
        da[-1] += np.sum(dC * (C0 + Kb.T @ I), axis=1)
        dal[sl] = np.cumsum((da * a)[::-1], axis=0)[::-1] / alpha[sl]
        dq[sl] = a * dQb
        dk[sl] = dKb / a
        dC = Qb.T @ g + aL[:, None] * dC
    # q' = S ^p1, k' = S ^p2, S = sigmoid(p1 . p2 / (tau_S sqrt d))
    n1 = np.linalg.norm(p1, axis=1, keepdims=True)
    n2 = np.linalg.norm(p2, axis=1, keepdims=True)
    h1, h2 = p1 / n1, p2 / n2
    dS = np.sum(dq * h1, axis=1) + np.sum(dk * h2, axis=1)
    du = (dS * S * (1.0 - S) / (tau_s * np.sqrt(d)))[:, None]
    g1, g2 = S[:, None] * dq, S[:, None] * dk
    dp1 = (g1 - h1 * np.sum(h1 * g1, axis=1, keepdims=True)) / n1 + du * p2
    dp2 = (g2 - h2 * np.sum(h2 * g2, axis=1, keepdims=True)) / n2 + du * p1
    return dp1, dp2, dv, dal
