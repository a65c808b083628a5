"""The block form of the Linear Relation backward that the chunked tcgen05 kernel uses for
the retention gradient where the retention is small (Sec. 5.2, App. A.4; the paper writes
out the forward only), restated in fp64 numpy and checked against the oracle's reverse
mode through the token recurrence.

Per block of LT tokens, channel c, with L_t the running sum of log2 alpha inside the block
(inclusive), L_m its value at the end of the first half and L_end at the block's end:
  Qm_t = q'_t 2^(L_t - L_m),  Km_j = k'_j 2^(L_m - L_j)     (q' = S p1 / |p1|, k' = S p2 / |p2|)
  dC(b - 1) = Diag(2^(L_end(b))) dC(b) + sum_{t in b} (q'_t 2^(L_t)) dY_t^T   (the state's adjoint)
  P_u = 2^(L_m) C_in + sum_{j < u} Km_j v_j^T,   Q_u = 2^(L_end - L_m) dC(b) + sum_{t >= u} Qm_t dY_t^T
  dalpha_u[c] = <P_u[c], Q_u[c]> / alpha_u[c]
C_in is the state entering the block (the oracle's forward states)."""
import numpy as np
import pytest

import oracle

TAU_S = 2.0


def _block_form_dalpha(p1, p2, v, alpha, dy, lt, decay_adjoint=True):
    T, d = p1.shape
    _, _, C = oracle.linear_fwd(p1, p2, v, alpha, want_states=True)  # C[t]: after t tokens
    n1 = np.linalg.norm(p1, axis=1, keepdims=True)
    n2 = np.linalg.norm(p2, axis=1, keepdims=True)
    S = 1.0 / (1.0 + np.exp(-(p1 * p2).sum(1, keepdims=True) / (TAU_S * np.sqrt(d))))
    qp, kp = S * p1 / n1, S * p2 / n2
    la = np.log2(alpha)
    starts = list(range(0, T, lt))
    # running log2 sums per block, the midpoint and end values
    L = {}
    for t0 in starts:
        t1 = min(t0 + lt, T)
        Lb = np.cumsum(la[t0:t1], axis=0)
        half = min(lt // 2, t1 - t0) - 1
        L[t0] = (Lb, Lb[half], Lb[-1])
    # the state's adjoint leaving every block, from the last block back
    dC = {}
    nxt = np.zeros((d, d))
    for t0 in reversed(starts):
        dC[t0] = nxt
        Lb, _, Lend = L[t0]
        t1 = t0 + Lb.shape[0]
        qs = qp[t0:t1] * np.exp2(Lb)
        nxt = (np.exp2(Lend)[:, None] if decay_adjoint else 1.0) * nxt + qs.T @ dy[t0:t1]
    da = np.zeros((T, d))
    for t0 in starts:
        Lb, Lm, Lend = L[t0]
        t1 = t0 + Lb.shape[0]
        qm = qp[t0:t1] * np.exp2(Lb - Lm)
        km = kp[t0:t1] * np.exp2(Lm - Lb)
        for i in range(t1 - t0):
            P = np.exp2(Lm)[:, None] * C[t0] + km[:i].T @ v[t0:t0 + i]
            Q = np.exp2(Lend - Lm)[:, None] * dC[t0] + qm[i:].T @ dy[t0 + i:t1]
            da[t0 + i] = (P * Q).sum(1) / alpha[t0 + i]
    return da


@pytest.mark.parametrize("T,lt", [(300, 64), (129, 128), (64, 16), (1, 8)])
def test_block_form_retention_gradient_matches_the_recurrence(T, lt):
    rng = np.random.default_rng(T + lt)
    d = 6
    p1, p2, v, dy = (rng.standard_normal((T, d)) for _ in range(4))
    alpha = rng.uniform(0.5, 1.0, (T, d))
    # retention down to 1e-7 on some tokens, where the kernel takes this form
    tiny = rng.random((T, d)) < 0.05
    alpha[tiny] = 10.0 ** rng.uniform(-7, -3, tiny.sum())
    ref = oracle.linear_bwd(p1, p2, v, alpha, dy)[3]
    got = _block_form_dalpha(p1, p2, v, alpha, dy, lt)
    scale = np.abs(ref).max()
    assert np.abs(got - ref).max() <= 1e-10 * scale
    # at the small-retention tokens too, entry by entry
    np.testing.assert_allclose(got[tiny], ref[tiny], rtol=1e-8, atol=1e-12 * scale)


def test_block_form_catches_a_wrong_adjoint():
    """The check has teeth: the state's adjoint carried back without the decay through the
    later block (a plausible slip) breaks the agreement with the recurrence."""
    rng = np.random.default_rng(5)
    T, d, lt = 96, 4, 32
    p1, p2, v, dy = (rng.standard_normal((T, d)) for _ in range(4))
    alpha = rng.uniform(0.3, 0.9, (T, d))
    ref = oracle.linear_bwd(p1, p2, v, alpha, dy)[3]
    right = _block_form_dalpha(p1, p2, v, alpha, dy, lt)
    wrong = _block_form_dalpha(p1, p2, v, alpha, dy, lt, decay_adjoint=False)
    scale = np.abs(ref).max()
    assert np.abs(right - ref).max() <= 1e-10 * scale
    assert np.abs(wrong - ref).max() > 1e-3 * scale
