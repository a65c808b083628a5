"""Pins of the Linear Relation oracle (oracle/linear_oracle.c) against what the paper and
the mathematics fix, independently of the oracle's own code (Sec. 5.2, App. A.4), and
planted mistakes in a copy of the oracle that the pins must catch.  CPU only."""
import os
import tempfile

import numpy as np
import pytest

import oracle

TAU = 2.0


def _inputs(T, d, seed, a_lo=0.3, a_hi=1.0):
    rng = np.random.default_rng(seed)
    p1, p2, v = (rng.standard_normal((T, d)) for _ in range(3))
    alpha = rng.uniform(a_lo, a_hi, (T, d))
    return p1, p2, v, alpha


def _self_and_coords(p1, p2):
    d = p1.shape[1]
    S = 1.0 / (1.0 + np.exp(-np.sum(p1 * p2, axis=1) / (TAU * np.sqrt(d))))
    q = p1 / np.linalg.norm(p1, axis=1, keepdims=True)
    k = p2 / np.linalg.norm(p2, axis=1, keepdims=True)
    return S, q, k


def pin_recurrent_equals_unrolled(lo):
    """App. A.4.2 (state recurrence) and App. A.4.5 (expanded historical Exchange) are
    two writings of the same operator."""
    for T, d, seed in [(1, 3, 0), (5, 4, 1), (12, 6, 2), (20, 2, 3)]:
        p1, p2, v, a = _inputs(T, d, seed)
        y, _ = lo.fwd(p1, p2, v, a)
        yu = lo.fwd_unrolled(p1, p2, v, a)
        assert np.abs(y - yu).max() <= 1e-12 * max(1.0, np.abs(yu).max())


def pin_first_token_is_its_information(lo):
    """C_0 = 0, so the first token has no Exchange: Y_1 = I~_1."""
    p1, p2, v, a = _inputs(1, 8, 4)
    y, S = lo.fwd(p1, p2, v, a)
    assert np.array_equal(y, v)
    assert 0.0 < S[0] < 1.0


def pin_no_retention_decay_is_causal_linear_attention(lo):
    """alpha = 1: E_t = S_t sum_{j<t} S_j (^p2_j . ^p1_t) I~_j, a strictly causal linear
    attention with Self weights, computed here with plain matrix products."""
    T, d = 16, 5
    p1, p2, v, _ = _inputs(T, d, 5)
    a = np.ones((T, d))
    S, q, k = _self_and_coords(p1, p2)
    W = np.tril(q @ k.T, -1) * np.outer(S, S)
    y, S_o = lo.fwd(p1, p2, v, a)
    assert np.allclose(S_o, S, rtol=0, atol=1e-15)
    assert np.abs(y - (v + W @ v)).max() <= 1e-12


def pin_vanishing_retention_forgets_history(lo):
    """alpha -> 0 erases C before every read: Y_t = I~_t."""
    p1, p2, v, _ = _inputs(10, 4, 6)
    a = np.full((10, 4), 1e-30)
    y, _ = lo.fwd(p1, p2, v, a)
    assert np.abs(y - v).max() <= 1e-25


def pin_strict_historical_support(lo):
    """App. A.4.3: E_t depends only on tokens before t.  Changing token s's information
    leaves every earlier output unchanged, moves Y_s by exactly the change (the Answer
    term), and reaches later outputs only through the state."""
    T, d, s = 9, 4, 4
    p1, p2, v, a = _inputs(T, d, 7)
    y0, _ = lo.fwd(p1, p2, v, a)
    v1 = v.copy()
    dv = np.linspace(0.1, 0.4, d)
    v1[s] += dv
    y1, _ = lo.fwd(p1, p2, v1, a)
    assert np.array_equal(y1[:s], y0[:s])
    assert np.allclose(y1[s] - y0[s], dv, rtol=0, atol=1e-14)
    assert np.abs(y1[s + 1:] - y0[s + 1:]).max() > 1e-6
    # the same for the relation coordinates of token s: its own output only moves via S_s,
    # which multiplies an Exchange read of the earlier state
    p2b = p2.copy()
    p2b[s] *= 1.7
    y2, _ = lo.fwd(p1, p2b, v, a)
    assert np.array_equal(y2[:s], y0[:s])


def pin_backward_matches_finite_differences(lo):
    """The reverse-mode backward against central differences of L = sum(dy * Y)."""
    for T, d, seed in [(1, 3, 10), (6, 3, 11), (9, 4, 12)]:
        _fd_check(lo, T, d, seed)


def _fd_check(lo, T, d, seed):
    p1, p2, v, a = _inputs(T, d, seed, 0.4, 0.95)
    rng = np.random.default_rng(seed + 100)
    dy = rng.standard_normal((T, d))
    grads = lo.bwd(p1, p2, v, a, dy)
    args = [p1, p2, v, a]
    h = 1e-6
    for which, g in enumerate(grads):
        num = np.empty_like(g)
        for idx in np.ndindex(*g.shape):
            hi = [x.copy() for x in args]
            lw = [x.copy() for x in args]
            hi[which][idx] += h
            lw[which][idx] -= h
            num[idx] = (np.sum(dy * lo_fwd(lo, hi)) - np.sum(dy * lo_fwd(lo, lw))) / (2 * h)
        err = np.abs(g - num).max() / max(1.0, np.abs(num).max())
        assert err <= 1e-7, f"input {which}: relative error {err:.2e}"


def lo_fwd(lo, args):
    return lo.fwd(*args)[0]


LINEAR_PINS = [pin_recurrent_equals_unrolled, pin_first_token_is_its_information,
               pin_no_retention_decay_is_causal_linear_attention,
               pin_vanishing_retention_forgets_history, pin_strict_historical_support,
               pin_backward_matches_finite_differences]


@pytest.mark.parametrize("pin", LINEAR_PINS, ids=[p.__name__ for p in LINEAR_PINS])
def test_linear_oracle_pin(pin):
    pin(oracle.linear())


# Planted mistakes (each keeps every memory access in bounds; the mutants run in-process).
LINEAR_MUTANTS = [
    ("read after the write (current token in its own Exchange)",
     "    /* Ask Others: E_t = S_t (C_t^-)^T ^p1_t;  Answer: Y_t = I~_t + E_t */\n    for (int j = 0; j < d; ++j) {\n      double e = 0.0;",
     "    for (int c = 0; c < d; ++c)\n      for (int j = 0; j < d; ++j) C[(size_t)c * d + j] += s_t * k[c] * I[j];\n    for (int j = 0; j < d; ++j) {\n      double e = 0.0;"),
    ("retention applied to the information side",
     "      for (int j = 0; j < d; ++j) C[(size_t)c * d + j] *= a[c];",
     "      for (int j = 0; j < d; ++j) C[(size_t)c * d + j] *= a[j];"),
    ("read not scaled by S_t", "      y[(size_t)t * d + j] = I[j] + s_t * e;",
     "      y[(size_t)t * d + j] = I[j] + e;"),
    ("write not scaled by S_t",
     "      for (int j = 0; j < d; ++j) C[(size_t)c * d + j] += s_t * k[c] * I[j];\n    if (S)",
     "      for (int j = 0; j < d; ++j) C[(size_t)c * d + j] += k[c] * I[j];\n    if (S)"),
    ("Self temperature dropped", "  *S = lsig(ldot(p1, p2, d) / (tau_s * sqrt((double)d)));",
     "  *S = lsig(ldot(p1, p2, d) / sqrt((double)d));"),
    ("coordinates not normalised", "    q[c] = p1[c] / n1;", "    q[c] = p1[c];"),
    ("read and write coordinates swapped", "      for (int c = 0; c < d; ++c) e += C[(size_t)c * d + j] * q[c];",
     "      for (int c = 0; c < d; ++c) e += C[(size_t)c * d + j] * k[c];"),
    ("dalpha uses the decayed state", "        da += dcm * Cprev[(size_t)c * d + j];",
     "        da += dcm * Cm[(size_t)c * d + j];"),
    ("adjoint state not decayed", "        dC[(size_t)c * d + j] = a[c] * dcm;  /* becomes dL/dC_{t-1} */",
     "        dC[(size_t)c * d + j] = dcm;  /* becomes dL/dC_{t-1} */"),
    ("normalisation gradient drops the projection", "      dp1[(size_t)t * d + c] = du * P2[c] + (dq[c] - q[c] * qdq) / n1;",
     "      dp1[(size_t)t * d + c] = du * P2[c] + dq[c] / n1;"),
    ("information gradient drops the write path", "      dv[(size_t)t * d + j] = G[j] + s_t * kdc;  /* Answer: Y = I + E;  write */",
     "      dv[(size_t)t * d + j] = G[j];"),
]


@pytest.mark.parametrize("mutant", LINEAR_MUTANTS, ids=[m[0] for m in LINEAR_MUTANTS])
def test_linear_mutant_is_caught(mutant):
    name, old, new = mutant
    src = open(oracle.LINEAR_SOURCE).read()
    assert src.count(old) == 1, f"mutation site for '{name}' not unique/not found"
    with tempfile.TemporaryDirectory() as tmp:
        path = os.path.join(tmp, "mutant.c")
        with open(path, "w") as f:
            f.write(src.replace(old, new))
        lo = oracle.LinearOracle(oracle.compile_source(path, os.path.join(tmp, "libmutant.so")))
        caught = []
        for pin in LINEAR_PINS:
            try:
                pin(lo)
            except (AssertionError, ValueError, FloatingPointError):
                caught.append(pin.__name__)
        assert caught, f"no pin catches the planted mistake '{name}'"


# --- the chunked (block-parallel) evaluation, pinned to the recurrence -------------

def pin_chunked_equals_recurrent(ch, lo=None):
    """oracle/linear_chunked.py regroups the recurrence into blocks of L tokens; for every
    block size its Y equals the recurrent oracle's (which covers the state handed from
    block to block whenever T > L)."""
    lo = lo or oracle.linear()
    for T, d, seed in [(1, 3, 40), (7, 4, 41), (20, 6, 42)]:
        p1, p2, v, a = _inputs(T, d, seed, 0.3, 1.0)
        y, _ = lo.fwd(p1, p2, v, a)
        for L in sorted({1, 2, 3, 5, 8, T}):
            yc, _ = ch.linear_fwd_chunked(p1, p2, v, a, L)
            assert np.abs(yc - y).max() <= 1e-12 * max(1.0, np.abs(y).max()), (T, d, L)


def test_chunked_oracle_pin():
    from oracle import linear_chunked
    pin_chunked_equals_recurrent(linear_chunked)


CHUNKED_MUTANTS = [
    ("current token in its own read", "A = np.tril(Qb @ Kb.T, -1)                 # strictly",
     "A = np.tril(Qb @ Kb.T, 0)                 # strictly"),
    ("inter-block term dropped", "Y[sl] = v[sl] + Qb @ C + A @ v[sl]",
     "Y[sl] = v[sl] + A @ v[sl]"),
    ("state not decayed across the block",
     "C = a[-1][:, None] * C + (a[-1] * Kb).T @ v[sl]  # the state handed on",
     "C = C + (a[-1] * Kb).T @ v[sl]  # the state handed on"),
    ("exclusive cumulative retention", "a = np.cumprod(alpha[sl], axis=0)          # a_t",
     "a = np.cumprod(alpha[sl], axis=0) / alpha[sl]  # a_t"),
]


@pytest.mark.parametrize("mutant", CHUNKED_MUTANTS, ids=[m[0] for m in CHUNKED_MUTANTS])
def test_chunked_mutant_is_caught(mutant):
    import importlib.util
    from oracle import linear_chunked
    name, old, new = mutant
    src = open(linear_chunked.__file__).read()
    assert src.count(old) == 1, f"mutation site for '{name}' not unique/not found"
    with tempfile.TemporaryDirectory() as tmp:
        path = os.path.join(tmp, "chunked_mutant.py")
        with open(path, "w") as f:
            f.write(src.replace(old, new))
        spec = importlib.util.spec_from_file_location("chunked_mutant", path)
        mod = importlib.util.module_from_spec(spec)
        spec.loader.exec_module(mod)
        with pytest.raises(AssertionError):
            pin_chunked_equals_recurrent(mod)


def pin_chunked_backward_equals_recurrent(ch, lo=None):
    """The block-form backward equals the recurrent oracle's reverse mode for every block
    size (all four gradients)."""
    lo = lo or oracle.linear()
    rng = np.random.default_rng(43)
    for T, d in [(1, 3), (7, 4), (20, 6)]:
        p1, p2, v, dy = (rng.standard_normal((T, d)) for _ in range(4))
        a = rng.uniform(0.3, 1.0, (T, d))
        ref = lo.bwd(p1, p2, v, a, dy)
        for L in sorted({1, 2, 3, 5, 8, T}):
            got = ch.linear_bwd_chunked(p1, p2, v, a, dy, L)
            for name, x, y in zip(("dp1", "dp2", "dv", "dalpha"), got, ref):
                assert np.abs(x - y).max() <= 1e-11 * max(1.0, np.abs(y).max()), (T, d, L, name)


def test_chunked_backward_pin():
    from oracle import linear_chunked
    pin_chunked_backward_equals_recurrent(linear_chunked)


CHUNKED_BWD_MUTANTS = [
    ("dI~ misses the state's adjoint", "dv[sl] = g + A.T @ g + Ka @ dC", "dv[sl] = g + A.T @ g"),
    ("dC_0 not decayed", "dC = Qb.T @ g + aL[:, None] * dC", "dC = Qb.T @ g + dC"),
    ("a_L factor of the handed-on state dropped",
     "da[-1] += np.sum(dC * (C0 + Kb.T @ I), axis=1)", "da[-1] += np.sum(dC * C0, axis=1)"),
    ("retention gradient not accumulated over later tokens",
     "dal[sl] = np.cumsum((da * a)[::-1], axis=0)[::-1] / alpha[sl]",
     "dal[sl] = da * a / alpha[sl]"),
    ("inter-block read missing from dQb", "dQb = dA @ Kb + g @ C0.T", "dQb = dA @ Kb"),
]


@pytest.mark.parametrize("mutant", CHUNKED_BWD_MUTANTS, ids=[m[0] for m in CHUNKED_BWD_MUTANTS])
def test_chunked_backward_mutant_is_caught(mutant):
    import importlib.util
    from oracle import linear_chunked
    name, old, new = mutant
    src = open(linear_chunked.__file__).read()
    assert src.count(old) == 1, f"mutation site for '{name}' not unique/not found"
    with tempfile.TemporaryDirectory() as tmp:
        path = os.path.join(tmp, "chunked_bwd_mutant.py")
        with open(path, "w") as f:
            f.write(src.replace(old, new))
        spec = importlib.util.spec_from_file_location("chunked_bwd_mutant", path)
        mod = importlib.util.module_from_spec(spec)
        spec.loader.exec_module(mod)
        with pytest.raises(AssertionError):
            pin_chunked_backward_equals_recurrent(mod)
