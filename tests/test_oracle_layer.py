"""Pins of the RoPE / Givens oracle (oracle/layer.py) against what the paper and the
mathematics fix, independently of the oracle's own code (Sec. 3.1-3.2, App. A.2.2,
App. B.3), and planted mistakes in a copy of the oracle that the pins must catch.  CPU
only."""
import importlib.util
import math
import os
import tempfile

import numpy as np
import pytest

from oracle import layer as lay


def _rand(shape, seed):
    return np.random.default_rng(seed).standard_normal(shape)


def _rot(angle):
    return np.array([[math.cos(angle), -math.sin(angle)], [math.sin(angle), math.cos(angle)]])


def pin_rope_position_zero_is_identity(L):
    x = _rand((2, 5, 3, 8), 0)
    assert np.array_equal(L.rope(x)[:, 0], x[:, 0])


def pin_rope_textbook_rotations(L):
    """RoFormer: pair c of the row at position m turns by m * base^(-2c/d).  d = 2: the
    angle is m; d = 4 with base 100: the second pair turns by m / 10."""
    T = 7
    x = _rand((1, T, 1, 2), 1)
    y = L.rope(x, base=100.0)
    for m in range(T):
        assert np.allclose(y[0, m, 0], _rot(m) @ x[0, m, 0], rtol=0, atol=1e-13)
    x4 = _rand((1, T, 1, 4), 2)
    y4 = L.rope(x4, base=100.0)
    for m in range(T):
        assert np.allclose(y4[0, m, 0, 0:2], _rot(m) @ x4[0, m, 0, 0:2], rtol=0, atol=1e-13)
        assert np.allclose(y4[0, m, 0, 2:4], _rot(m / 10.0) @ x4[0, m, 0, 2:4], rtol=0, atol=1e-13)


def pin_rope_keeps_pair_norms(L):
    x = _rand((2, 9, 2, 16), 3)
    y = L.rope(x)
    nx = x[..., 0::2] ** 2 + x[..., 1::2] ** 2
    ny = y[..., 0::2] ** 2 + y[..., 1::2] ** 2
    assert np.allclose(nx, ny, rtol=1e-12, atol=0)


def pin_rope_relative_positions(L):
    """q_m . k_n depends on m - n only: the same vectors at (m, n) and (m + s, n + s)."""
    d, T = 12, 40
    q, k = _rand(d, 4), _rand(d, 5)
    for (m, n, s) in [(3, 1, 7), (10, 10, 20), (25, 2, 9)]:
        def dot(mq, nk):
            Q = np.zeros((1, T, 1, d))
            K = np.zeros((1, T, 1, d))
            Q[0, mq, 0] = q
            K[0, nk, 0] = k
            return float(L.rope(Q)[0, mq, 0] @ L.rope(K)[0, nk, 0])
        assert abs(dot(m, n) - dot(m + s, n + s)) <= 1e-12 * max(1.0, abs(dot(m, n)))


def pin_rope_inverse_and_adjoint(L):
    x, y = _rand((2, 6, 2, 10), 6), _rand((2, 6, 2, 10), 7)
    assert np.allclose(L.rope(L.rope(x), inverse=True), x, rtol=0, atol=1e-13)
    assert abs(np.sum(L.rope(x) * y) - np.sum(x * L.rope(y, inverse=True))) <= 1e-11


def pin_givens_zero_angle_is_identity(L):
    info = _rand((2, 4, 6, 5), 8)
    for pairing in (0, 1):
        assert np.array_equal(L.givens(info, np.zeros(3), pairing), info)


def pin_givens_quarter_turn(L):
    """theta = pi/2 sends (I_a, I_b) to (-I_b, I_a) on every pair."""
    info = _rand((1, 3, 4, 5), 9)
    out = L.givens(info, np.full(2, math.pi / 2), 0)
    for a, b in ((0, 1), (2, 3)):
        assert np.allclose(out[:, :, a], -info[:, :, b], atol=1e-15)
        assert np.allclose(out[:, :, b], info[:, :, a], atol=1e-15)


def pin_givens_pairing_b_wraps(L):
    """Pairing B of 4 heads: pair 0 mixes heads 1 and 2, pair 1 heads 3 and 0 (M_B with
    one-based (2,3), (4,1))."""
    info = _rand((1, 2, 4, 3), 10)
    th = np.array([0.3, -1.1])
    out = L.givens(info, th, 1)
    for (a, b), t in (((1, 2), th[0]), ((3, 0), th[1])):
        for bt in range(2):
            for c in range(3):
                v = _rot(t) @ np.array([info[0, bt, a, c], info[0, bt, b, c]])
                assert np.allclose([out[0, bt, a, c], out[0, bt, b, c]], v, atol=1e-14)


def pin_givens_keeps_pair_energy(L):
    info = _rand((2, 5, 6, 4), 11)
    th = np.array([0.4, 2.0, -0.7])
    for pairing in (0, 1):
        out = L.givens(info, th, pairing)
        for (a, b) in L.pairs(6, pairing):
            e0 = info[:, :, a] ** 2 + info[:, :, b] ** 2
            e1 = out[:, :, a] ** 2 + out[:, :, b] ** 2
            assert np.allclose(e0, e1, rtol=1e-12, atol=0)


def pin_gradients_match_finite_differences(L):
    """L = sum(dQ * Q + dK * K + dV * V) with (Q, K, V) = prep(P1, P2, I, theta)."""
    B, T, H, d = 1, 5, 4, 6
    p1, p2, info = _rand((B, T, H, d), 12), _rand((B, T, H, d), 13), _rand((B, T, H, d), 14)
    dq, dk, dv = _rand((B, T, H, d), 15), _rand((B, T, H, d), 16), _rand((B, T, H, d), 17)
    th = np.array([0.5, -0.9])
    for pairing in (0, 1):
        def loss(a, b, c, t):
            Q, K, V = L.prep(a, b, c, t, pairing)
            return np.sum(dq * Q) + np.sum(dk * K) + np.sum(dv * V)
        g1, g2, gi, gt = L.grad(dq, dk, dv, info, th, pairing)
        h = 1e-6
        rng = np.random.default_rng(18)
        for which, g in ((0, g1), (1, g2), (2, gi)):
            for _ in range(8):
                idx = tuple(int(rng.integers(0, n)) for n in (B, T, H, d))
                args = [p1.copy(), p2.copy(), info.copy()]
                args[which][idx] += h
                up = loss(*args, th)
                args[which][idx] -= 2 * h
                dn = loss(*args, th)
                assert abs((up - dn) / (2 * h) - g[idx]) <= 1e-7 * max(1.0, abs(g[idx]))
        for k in range(len(th)):
            tp, tm = th.copy(), th.copy()
            tp[k] += h
            tm[k] -= h
            num = (loss(p1, p2, info, tp) - loss(p1, p2, info, tm)) / (2 * h)
            assert abs(num - gt[k]) <= 1e-7 * max(1.0, abs(gt[k]))


LAYER_PINS = [pin_rope_position_zero_is_identity, pin_rope_textbook_rotations,
              pin_rope_keeps_pair_norms, pin_rope_relative_positions,
              pin_rope_inverse_and_adjoint, pin_givens_zero_angle_is_identity,
              pin_givens_quarter_turn, pin_givens_pairing_b_wraps,
              pin_givens_keeps_pair_energy, pin_gradients_match_finite_differences]


@pytest.mark.parametrize("pin", LAYER_PINS, ids=[p.__name__ for p in LAYER_PINS])
def test_layer_oracle_pin(pin):
    pin(lay)


LAYER_MUTANTS = [
    ("frequency exponent without the factor 2", "return m * base ** (-2.0 * c / d)",
     "return m * base ** (-1.0 * c / d)"),
    ("rotation sign flipped", "out[..., 0::2] = xe * cs - xo * sn",
     "out[..., 0::2] = xe * cs + xo * sn"),
    ("half-split pairs instead of interleaved", "xe, xo = x[..., 0::2], x[..., 1::2]",
     "xe, xo = x[..., : d // 2], x[..., d // 2:]"),
    ("transpose not inverted", "    if inverse:\n        sn = -sn", "    if inverse:\n        pass"),
    ("pairing B without the wrap", "return [(2 * k + 1, (2 * k + 2) % H) for k in range(H // 2)]",
     "return [(2 * k + 1, min(2 * k + 2, H - 1)) for k in range(H // 2)]"),
    ("Givens sign convention swapped", "out[:, :, a] = c * info[:, :, a] - s * info[:, :, b]",
     "out[:, :, a] = c * info[:, :, a] + s * info[:, :, b]"),
    ("dtheta sign dropped", "np.sum(ga * (-s * ia - c * ib))", "np.sum(ga * (s * ia - c * ib))"),
    ("dI of the second head not transposed", "dinfo[:, :, b] = -s * ga + c * gb",
     "dinfo[:, :, b] = s * ga + c * gb"),
]


@pytest.mark.parametrize("mutant", LAYER_MUTANTS, ids=[m[0] for m in LAYER_MUTANTS])
def test_layer_mutant_is_caught(mutant):
    name, old, new = mutant
    src = open(lay.__file__).read()
    assert src.count(old) == 1, f"mutation site for '{name}' not unique/not found"
    with tempfile.TemporaryDirectory() as tmp:
        path = os.path.join(tmp, "layer_mutant.py")
        with open(path, "w") as f:
            f.write(src.replace(old, new))
        spec = importlib.util.spec_from_file_location("layer_mutant", path)
        mod = importlib.util.module_from_spec(spec)
        spec.loader.exec_module(mod)
        caught = []
        for pin in LAYER_PINS:
            try:
                pin(mod)
            except (AssertionError, ValueError, IndexError, FloatingPointError):
                caught.append(pin.__name__)
        assert caught, f"no pin catches the planted mistake '{name}'"
