"""Pins for the QKV projection + RoPE oracle: textbook properties of a
rotary embedding (identity at position 0, norm-preserving, composes by adding
angles, inner products depend only on relative position, a plain 2-D
rotation when d = 2) and brute-force sums for the projection."""

import math

import numpy as np
import pytest

from oracle import projection as R


def _rng(seed):
    return np.random.default_rng(seed)


def test_position_zero_is_identity():
    x = _rng(1).standard_normal((5, 3, 8))
    assert np.array_equal(R.rope(x, np.zeros(5), 10000.0), x)


def test_rotation_preserves_each_pair_norm():
    x = _rng(2).standard_normal((7, 2, 16))
    y = R.rope(x, np.arange(7) * 13.0, 500000.0)
    h = 8
    assert np.allclose(x[..., :h] ** 2 + x[..., h:] ** 2, y[..., :h] ** 2 + y[..., h:] ** 2,
                       rtol=1e-12, atol=1e-12)


def test_angles_add():
    x = _rng(3).standard_normal((4, 1, 32))
    a = np.array([0.0, 5.0, 1000.0, 131000.0])
    b = np.array([3.0, 7.0, 2.0, 71.0])
    assert np.allclose(R.rope(R.rope(x, a, 500000.0), b, 500000.0), R.rope(x, a + b, 500000.0),
                       atol=1e-9)


def test_inner_products_depend_on_relative_position():
    rng = _rng(4)
    q = rng.standard_normal((1, 1, 64))
    k = rng.standard_normal((1, 1, 64))
    for m, n, t in [(10, 3, 5), (1000, 1000, 77), (5, 900, 1234)]:
        d1 = np.sum(R.rope(q, [m], 10000.0) * R.rope(k, [n], 10000.0))
        d2 = np.sum(R.rope(q, [m + t], 10000.0) * R.rope(k, [n + t], 10000.0))
        assert abs(d1 - d2) < 1e-9


def test_two_dimensional_case_is_a_plain_rotation():
    # d = 2: one pair with frequency theta^0 = 1, so the angle is the position
    x = np.array([[[1.0, 0.0]], [[0.3, -2.0]]])
    pos = np.array([math.pi / 2, 1.0])
    y = R.rope(x, pos, 12345.0)
    assert np.allclose(y[0, 0], [0.0, 1.0], atol=1e-15)
    c, s = math.cos(1.0), math.sin(1.0)
    assert np.allclose(y[1, 0], [0.3 * c + 2.0 * s, -2.0 * c + 0.3 * s], atol=1e-15)


def test_projection_split_matches_brute_force():
    rng = _rng(5)
    n, hidden, hq, hkv, d = 3, 5, 2, 1, 4
    x = rng.standard_normal((n, hidden))
    w = rng.standard_normal(((hq + 2 * hkv) * d, hidden))
    q, k, v = R.qkv_rope(x, w, hq, hkv, d, pos0=0, theta=10000.0)
    # position 0 row: no rotation, plain sums
    for h in range(hq):
        for c in range(d):
            ref = math.fsum(x[0, i] * w[h * d + c, i] for i in range(hidden))
            assert abs(q[0, h, c] - ref) < 1e-12
    for c in range(d):
        ref_k = math.fsum(x[0, i] * w[hq * d + c, i] for i in range(hidden))
        ref_v = math.fsum(x[2, i] * w[(hq + hkv) * d + c, i] for i in range(hidden))
        assert abs(k[0, 0, c] - ref_k) < 1e-12
        assert abs(v[2, 0, c] - ref_v) < 1e-12   # V is never rotated


def test_rows_are_rotated_at_their_global_position():
    rng = _rng(6)
    x = rng.standard_normal((4, 6))
    w = rng.standard_normal((3 * 8, 6))
    q, _, _ = R.qkv_rope(x, w, 1, 1, 8, pos0=100, theta=10000.0)
    plain = (x @ w.T)[:, :8].reshape(4, 1, 8)
    assert np.allclose(q, R.rope(plain, 100 + np.arange(4), 10000.0), atol=1e-12)


def test_four_dims_pin_frequencies_and_pairing():
    # d = 4, theta = 10000: pair (0, 2) turns by pos * 1, pair (1, 3) by
    # pos * 10000^(-2/4) = pos / 100 (rotate-half pairing, not adjacent dims).
    pos = 37.0
    e1 = np.array([[[0.0, 1.0, 0.0, 0.0]]])
    y = R.rope(e1, [pos], 10000.0)
    assert np.allclose(y[0, 0], [0.0, math.cos(pos / 100), 0.0, math.sin(pos / 100)], atol=1e-15)
    e0 = np.array([[[1.0, 0.0, 0.0, 0.0]]])
    y = R.rope(e0, [pos], 10000.0)
    assert np.allclose(y[0, 0], [math.cos(pos), 0.0, math.sin(pos), 0.0], atol=1e-15)
