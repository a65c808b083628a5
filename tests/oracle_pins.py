"""Pins of the fp64 oracle to facts the paper and plain mathematics fix.

Each ``pin_*`` function takes an :class:`oracle.Oracle` and raises AssertionError
when the oracle disagrees with the fact it checks.  None of them re-types the
oracle's own formula: they use closed forms of special inputs, identities the
paper proves (with a citation), library routines (torch softmax / logsumexp),
finite differences, and agreement between independently coded paths.

The same functions run against deliberately broken copies of the oracle in
``test_oracle_mutants.py`` to show that plausible mistakes are caught.
"""
from __future__ import annotations

import math

import numpy as np
import torch

TAU = 2.0


def _rand(T, d, seed, scale=1.0):
    rs = np.random.default_rng(seed)
    q = rs.standard_normal((T, d)) * scale
    k = rs.standard_normal((T, d)) * scale
    v = rs.standard_normal((T, d))
    g = rs.standard_normal((T, d))
    return q, k, v, g


def _close(a, b, rtol, atol=0.0, what=""):
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    err = np.max(np.abs(a - b)) if a.size else 0.0
    ref = np.max(np.abs(b)) if b.size else 0.0
    assert err <= atol + rtol * max(ref, 1e-300), f"{what}: max|diff|={err:.3e}, max|ref|={ref:.3e}"


# --- forward ---------------------------------------------------------------

def pin_T1_closed_form(orc):
    """T = 1 (App. A.1.8): no history, so F_11 = 1, Y_1 = I~_1 and the normaliser is
    Z_1 = e^{S_1} with S_1 = sigmoid(q.k / (sqrt(d) tau_S))."""
    q, k, v, _ = _rand(1, 5, 1)
    y, lz = orc.fwd(q, k, v, 0.5)
    u = float(q[0] @ k[0]) / math.sqrt(5)
    s = 1.0 / (1.0 + math.exp(-u / TAU))
    _close(y, v, 1e-15, what="Y_1")
    assert abs(lz[0] - s) < 1e-15, (lz[0], s)


def pin_T2_hand_formula(orc):
    """T = 2 by hand from Eq. (causal-relation): row 2 has R_22 = sigmoid(U_22/2) and
    R_21 = SiLU(U_21) - lambda log 2, so Y_2 = (1-g) v_2 + g v_1 with
    g = e^{R_21} / (e^{R_21} + e^{R_22})."""
    q, k, v, _ = _rand(2, 3, 2)
    lam = 0.7
    y, lz = orc.fwd(q, k, v, lam)
    u21 = float(q[1] @ k[0]) / math.sqrt(3)
    u22 = float(q[1] @ k[1]) / math.sqrt(3)
    r22 = 1.0 / (1.0 + math.exp(-u22 / TAU))
    r21 = u21 / (1.0 + math.exp(-u21)) - lam * math.log(2.0)
    g = math.exp(r21) / (math.exp(r21) + math.exp(r22))
    _close(y[1], (1 - g) * v[1] + g * v[0], 1e-14, what="Y_2")
    assert abs(lz[1] - math.log(math.exp(r21) + math.exp(r22))) < 1e-14


def pin_zero_evidence(orc):
    """P1 = 0 makes every U_ij = 0, so S_i = sigmoid(0) = 1/2 and E_ij = SiLU(0) = 0.
    Row i then has one entry 1/2 and (i-1) entries -lambda log i:
    Z_i = e^{1/2} + (i-1) i^{-lambda}, F_ii = e^{1/2}/Z_i, F_ij = i^{-lambda}/Z_i."""
    T, d, lam = 9, 4, 0.5
    _, k, v, _ = _rand(T, d, 3)
    q = np.zeros((T, d))
    y, lz = orc.fwd(q, k, v, lam)
    for r in range(T):
        i = r + 1
        Z = math.exp(0.5) + (i - 1) * i ** (-lam)
        expect = (math.exp(0.5) * v[r] + i ** (-lam) * v[:r].sum(axis=0)) / Z
        _close(y[r], expect, 1e-14, what=f"Y row {i}")
        assert abs(lz[r] - math.log(Z)) < 1e-14


def pin_materialised_structure(orc):
    """Eq. (causal-relation) / (relation-flow): rows of F sum to 1, F and R vanish /
    are -inf above the diagonal, R_ii lies strictly in (0, 1) (bounded Self)."""
    q, k, v, _ = _rand(12, 6, 4, scale=2.0)
    _, _, R, F = orc.fwd(q, k, v, -0.3, want_matrices=True)
    _close(F.sum(axis=1), np.ones(12), 1e-14, what="row sums")
    upper = np.triu_indices(12, 1)
    assert np.all(F[upper] == 0.0)
    assert np.all(np.isneginf(R[upper]))
    diag = np.diag(R)
    assert np.all(diag > 0.0) and np.all(diag < 1.0)
    # logZ row normaliser against torch's logsumexp of the materialised row
    _, lz = orc.fwd(q, k, v, -0.3)
    _close(lz, torch.logsumexp(torch.from_numpy(R), dim=1).numpy(), 1e-14, what="logZ")


def pin_self_bounded_extremes(orc):
    """S_i in (0, 1) even for huge |U_ii| (Sec. 3.1: the Self map is bounded); with
    |U_ii| >> tau_S the diagonal logit saturates at 0 or 1."""
    T, d = 4, 2
    q = np.array([[30.0, 0.0], [-30.0, 0.0], [1.0, 0.0], [0.0, 0.0]])
    k = np.array([[30.0, 0.0], [30.0, 0.0], [0.0, 0.0], [0.0, 0.0]])
    v = np.eye(T, d)
    _, _, R, _ = orc.fwd(q, k, v, 0.5, want_matrices=True)
    assert abs(R[0, 0] - 1.0) < 1e-12 and abs(R[1, 1]) < 1e-12
    assert R[2, 2] == 0.5 and R[3, 3] == 0.5


def pin_factorized_equals_materialised(orc):
    """App. A.1.6: (1-g) I~_i + g Ibar_i equals the materialised sum_j F_ij I~_j, and
    logZ = log(e^S + e^A) equals log sum_j e^{R_ij} (two independently coded paths)."""
    for (T, d, lam, seed) in [(1, 3, 0.5, 5), (2, 1, 0.5, 6), (7, 4, 0.0, 7), (33, 8, -1.0, 8),
                              (20, 5, 3.0, 9)]:
        q, k, v, _ = _rand(T, d, seed, scale=1.5)
        y, lz = orc.fwd(q, k, v, lam)
        f = orc.fwd_factorized(q, k, v, lam)
        _close(f["Y"], y, 1e-12, what=f"Y T={T}")
        _close(f["logZ"], lz, 1e-12, what=f"logZ T={T}")


def pin_self_exchange_split(orc):
    """Eq. (self-flow-mass): the materialised diagonal F_ii equals sigma(S - A) and the
    materialised historical mass sum_{j<i} F_ij equals g = sigma(A - S); F_ii + g = 1;
    log(g / F_ii) = A - S (Eq. self-history-odds)."""
    T = 15
    q, k, v, _ = _rand(T, 4, 10, scale=1.3)
    lam = 0.4
    _, _, _, F = orc.fwd(q, k, v, lam, want_matrices=True)
    f = orc.fwd_factorized(q, k, v, lam)
    g_mat = np.array([F[r, :r].sum() for r in range(T)])
    _close(np.diag(F), f["Fii"], 1e-13, what="F_ii")
    _close(g_mat, f["g"], 1e-13, what="g")
    _close(f["Fii"] + f["g"], np.ones(T), 1e-15, what="F_ii + g")
    r = np.arange(1, T)
    _close(np.log(f["g"][r] / f["Fii"][r]), f["A"][r] - f["S"][r], 1e-12, what="odds")
    assert f["g"][0] == 0.0 and f["Fii"][0] == 1.0 and np.isneginf(f["A"][0])


def pin_conditional_allocation(orc):
    """Eq. (conditional-exchange-distribution) / (within-history-preference):
    pi^E_ij = F_ij / g_i sums to 1 over j < i and does not depend on lambda, while
    the Self share does."""
    T = 14
    q, k, v, _ = _rand(T, 3, 11)
    _, _, _, F1 = orc.fwd(q, k, v, 0.5, want_matrices=True)
    _, _, _, F2 = orc.fwd(q, k, v, -2.0, want_matrices=True)
    f1 = orc.fwd_factorized(q, k, v, 0.5)
    for r in range(1, T):
        p1 = F1[r, :r] / F1[r, :r].sum()
        p2 = F2[r, :r] / F2[r, :r].sum()
        _close(p1, p2, 1e-13, what=f"pi lambda-invariance row {r}")
        _close(p1, f1["pi"][r, :r], 1e-13, what=f"pi row {r}")
        assert abs(f1["pi"][r, :r].sum() - 1.0) < 1e-14
    assert np.max(np.abs(np.diag(F1) - np.diag(F2))) > 1e-3


def pin_output_on_segment(orc):
    """Eq. (information-space-form): Y_i = I~_i + g_i (Ibar_i - I~_i) with g_i in
    [0, 1]: the output lies on the segment from the Self state to the Exchange
    aggregate, at the fraction g_i of its length."""
    T, d = 11, 6
    q, k, v, _ = _rand(T, d, 12, scale=1.7)
    y, _ = orc.fwd(q, k, v, 0.5)
    f = orc.fwd_factorized(q, k, v, 0.5)
    for r in range(1, T):
        delta = f["Ibar"][r] - v[r]
        t = float((y[r] - v[r]) @ delta) / float(delta @ delta)
        assert -1e-12 <= t <= 1 + 1e-12
        assert abs(t - f["g"][r]) < 1e-11
        _close(y[r], v[r] + t * delta, 1e-12, what=f"segment row {r}")


def pin_scan_tile_invariance(orc):
    """App. A.3.2-A.3.5: the tiled (m, l, z) scan reproduces the materialised row for
    every tile size and tile order."""
    T, d, lam = 37, 5, 0.5
    q, k, v, _ = _rand(T, d, 13, scale=2.0)
    y, lz = orc.fwd(q, k, v, lam)
    for tile in (1, 2, 3, 8, 16, 64):
        for rev in (False, True):
            ys, lzs = orc.fwd_scan(q, k, v, lam, tile, rev)
            _close(ys, y, 1e-12, what=f"scan Y tile={tile} rev={rev}")
            _close(lzs, lz, 1e-12, what=f"scan logZ tile={tile} rev={rev}")


def pin_lambda_plus_limit(orc):
    """lambda -> +inf suppresses every Exchange entry (-lambda log i -> -inf for i >= 2),
    so each row keeps only Self: Y -> I~."""
    q, k, v, _ = _rand(10, 4, 14)
    y, _ = orc.fwd(q, k, v, 60.0)
    _close(y, v, 1e-12, what="lambda=+60")


def pin_lambda_minus_limit(orc):
    """lambda -> -inf makes the Exchange shift dominate Self for i >= 2, so row i becomes
    the strictly causal softmax of SiLU(U_ij) over j < i (torch masked softmax),
    applied to I~; row 1 stays I~_1."""
    T, d = 10, 4
    q, k, v, _ = _rand(T, d, 15)
    y, _ = orc.fwd(q, k, v, -60.0)
    U = torch.from_numpy(q @ k.T / math.sqrt(d))
    E = torch.nn.functional.silu(U)
    mask = torch.ones(T, T, dtype=torch.bool).tril(-1)
    W = torch.softmax(E.masked_fill(~mask, float("-inf"))[1:], dim=1)
    _close(y[1:], (W @ torch.from_numpy(v)).numpy(), 1e-12, what="lambda=-60")
    _close(y[0], v[0], 1e-15, what="row 1")


def pin_lambda_zero_logsumexp(orc):
    """lambda = 0 (the 'no count calibration' ablation, Table 3): logZ_i is torch's
    logsumexp of [SiLU(U_i1), ..., SiLU(U_i,i-1), sigmoid(U_ii / 2)]."""
    T, d = 9, 3
    q, k, v, _ = _rand(T, d, 16)
    _, lz = orc.fwd(q, k, v, 0.0)
    U = torch.from_numpy(q @ k.T / math.sqrt(d))
    for r in range(T):
        row = torch.cat([torch.nn.functional.silu(U[r, :r]), torch.sigmoid(U[r, r:r + 1] / 2)])
        assert abs(lz[r] - float(torch.logsumexp(row, 0))) < 1e-14


def pin_mhr_heads_independent(orc):
    """Sec. 3.2 / App. A.2.1: every head is an independent SER problem; the multi-head
    wrapper equals per-head calls and permuting heads permutes the outputs."""
    B, T, H, d = 2, 9, 3, 4
    rs = np.random.default_rng(17)
    q, k, v = (rs.standard_normal((B, T, H, d)) for _ in range(3))
    y, lz = orc.mhr_fwd(q, k, v, 0.5)
    for b in range(B):
        for h in range(H):
            yh, lzh = orc.fwd(q[b, :, h], k[b, :, h], v[b, :, h], 0.5)
            _close(y[b, :, h], yh, 1e-15, what=f"head {b},{h}")
            _close(lz[b, h], lzh, 1e-15)
    perm = [2, 0, 1]
    yp, _ = orc.mhr_fwd(q[:, :, perm], k[:, :, perm], v[:, :, perm], 0.5)
    _close(yp, y[:, :, perm], 1e-15, what="head permutation")


def pin_causality(orc):
    """Eq. (causal-relation): row i depends only on tokens j <= i, so changing the last
    token leaves every earlier output unchanged."""
    q, k, v, _ = _rand(8, 3, 18)
    y, lz = orc.fwd(q, k, v, 0.5)
    q2, k2, v2 = q.copy(), k.copy(), v.copy()
    q2[-1] += 1.0; k2[-1] -= 2.0; v2[-1] *= 3.0
    y2, lz2 = orc.fwd(q2, k2, v2, 0.5)
    assert np.array_equal(y[:-1], y2[:-1]) and np.array_equal(lz[:-1], lz2[:-1])


def pin_rows_subset(orc):
    """The sampled-row forward returns exactly the rows of the full forward."""
    q, k, v, _ = _rand(19, 3, 19)
    y, lz = orc.fwd(q, k, v, 0.5)
    rows = [0, 5, 18, 7]
    yr, lzr = orc.fwd_rows(q, k, v, rows, 0.5)
    assert np.array_equal(yr, y[rows]) and np.array_equal(lzr, lz[rows])


# --- backward --------------------------------------------------------------

def _loss(orc, q, k, v, g, lam):
    y, _ = orc.fwd(q, k, v, lam)
    return float(np.sum(y * g))


def pin_bwd_finite_differences(orc):
    """Central finite differences (fp64, h = 1e-6) of L = sum(Y * G) with respect to
    every entry of P1, P2, I~ and to lambda match the analytic gradient (App. A.1.7)."""
    for (T, d, lam, seed) in [(6, 3, 0.5, 20), (8, 4, -0.8, 21), (3, 2, 2.0, 22)]:
        q, k, v, g = _rand(T, d, seed, scale=1.2)
        dq, dk, dv, dl = orc.bwd(q, k, v, g, lam)
        h = 1e-6
        for name, x, gx in (("q", q, dq), ("k", k, dk), ("v", v, dv)):
            num = np.zeros_like(x)
            for idx in np.ndindex(x.shape):
                xp = x.copy(); xp[idx] += h
                xm = x.copy(); xm[idx] -= h
                args_p = {"q": q, "k": k, "v": v}; args_p[name] = xp
                args_m = {"q": q, "k": k, "v": v}; args_m[name] = xm
                num[idx] = (_loss(orc, args_p["q"], args_p["k"], args_p["v"], g, lam)
                            - _loss(orc, args_m["q"], args_m["k"], args_m["v"], g, lam)) / (2 * h)
            _close(gx, num, 1e-7, atol=1e-9, what=f"d{name} T={T}")
        numl = (_loss(orc, q, k, v, g, lam + h) - _loss(orc, q, k, v, g, lam - h)) / (2 * h)
        assert abs(dl - numl) <= 1e-7 * max(1.0, abs(numl)), (dl, numl)


def pin_bwd_two_derivations(orc):
    """App. A.1.7 gives two derivations of the same gradient: the generic softmax
    gradient dR = F o (H - sum_k F_ik H_ik) and the Self-Exchange credit
    decomposition through g, pi^E and c_i = G_i . Delta_i.  They agree."""
    for (T, d, lam, seed) in [(1, 2, 0.5, 23), (2, 3, 0.5, 24), (17, 5, 0.5, 25),
                              (30, 4, -1.5, 26), (12, 6, 3.0, 27)]:
        q, k, v, g = _rand(T, d, seed, scale=1.4)
        a = orc.bwd(q, k, v, g, lam)
        b = orc.bwd_credit(q, k, v, g, lam)
        for name, x, y in zip(("dq", "dk", "dv"), a[:3], b[:3]):
            _close(x, y, 1e-11, atol=1e-14, what=f"{name} T={T}")
        assert abs(a[3] - b[3]) <= 1e-11 * max(1.0, abs(a[3])), (a[3], b[3])


def pin_bwd_T1(orc):
    """T = 1: F_11 = 1 whatever P1, P2 are, so dP1 = dP2 = 0, dI~ = G, dlambda = 0."""
    q, k, v, g = _rand(1, 4, 28)
    dq, dk, dv, dl = orc.bwd(q, k, v, g, 0.5)
    assert np.all(dq == 0) and np.all(dk == 0) and dl == 0.0
    _close(dv, g, 1e-15, what="dv")


def pin_bwd_dv_mass(orc):
    """dI~ = F^T G and the rows of F sum to 1, so the column sums of dI~ equal the
    column sums of G (Eq. relation-flow)."""
    q, k, v, g = _rand(16, 5, 29, scale=1.5)
    _, _, dv, _ = orc.bwd(q, k, v, g, 0.5)
    _close(dv.sum(axis=0), g.sum(axis=0), 1e-13, what="sum dv")


def pin_bwd_lambda_plus_limit(orc):
    """lambda -> +inf: Y = I~ (pin_lambda_plus_limit), so dI~ = G, and the P1, P2 and
    lambda gradients vanish."""
    q, k, v, g = _rand(7, 3, 30)
    dq, dk, dv, dl = orc.bwd(q, k, v, g, 60.0)
    _close(dv, g, 1e-12, what="dv")
    assert np.max(np.abs(dq)) < 1e-12 and np.max(np.abs(dk)) < 1e-12 and abs(dl) < 1e-12


def pin_mhr_bwd_sums(orc):
    """lambda is shared by the heads (App. A.1.1), so the multi-head dlambda is the sum
    of the per-head values; the other gradients are per head."""
    B, T, H, d = 2, 7, 2, 3
    rs = np.random.default_rng(31)
    q, k, v, g = (rs.standard_normal((B, T, H, d)) for _ in range(4))
    dq, dk, dv, dl = orc.mhr_bwd(q, k, v, g, 0.5)
    tot = 0.0
    for b in range(B):
        for h in range(H):
            a = orc.bwd(q[b, :, h], k[b, :, h], v[b, :, h], g[b, :, h], 0.5)
            _close(dq[b, :, h], a[0], 1e-15); _close(dk[b, :, h], a[1], 1e-15)
            _close(dv[b, :, h], a[2], 1e-15)
            tot += a[3]
    assert abs(dl - tot) <= 1e-13 * max(1.0, abs(tot))


def pin_bwd_tail_rows(orc):
    """Rows of the softmax-gradient form are independent: restricting the backward to
    rows r >= r0 leaves dq rows >= r0 and dk, dv rows >= r0 unchanged (only rows i >= j
    feed key j, Eq. causal-relation)."""
    q, k, v, g = _rand(13, 4, 32, scale=1.3)
    full = orc.bwd(q, k, v, g, 0.5)
    for r0 in (0, 5, 12):
        dq, dk, dv, _ = orc.bwd_tail(q, k, v, g, 0.5, r0)
        _close(dq[r0:], full[0][r0:], 1e-14); _close(dk[r0:], full[1][r0:], 1e-14)
        _close(dv[r0:], full[2][r0:], 1e-14)
        assert np.all(dq[:r0] == 0)


ALL_PINS = [
    pin_T1_closed_form, pin_T2_hand_formula, pin_zero_evidence, pin_materialised_structure,
    pin_self_bounded_extremes, pin_factorized_equals_materialised, pin_self_exchange_split,
    pin_conditional_allocation, pin_output_on_segment, pin_scan_tile_invariance,
    pin_lambda_plus_limit, pin_lambda_minus_limit, pin_lambda_zero_logsumexp,
    pin_mhr_heads_independent, pin_causality, pin_rows_subset, pin_bwd_finite_differences,
    pin_bwd_two_derivations, pin_bwd_T1, pin_bwd_dv_mass, pin_bwd_lambda_plus_limit,
    pin_mhr_bwd_sums, pin_bwd_tail_rows,
]
