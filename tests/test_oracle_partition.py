"""Pins for the partition oracle (Sec. 3.2 / Eq. 1, Sec. 4.2).

None of these re-types the oracle's isqrt formula: rounding is checked by
exact rational interval membership and by floating point away from ties, the
cost model by its algebra and by brute-force pair counting, the clamps by
invariants, and the closed form at the boundaries where sqrt(i/M) is rational.
"""

import math
import os
import random
from fractions import Fraction

import pytest

from oracle import partition as P

G = 128


def _brute_round_half_up_sqrt(i, m, units):
    """n with n - 1/2 <= units*sqrt(i/m) < n + 1/2, found by scanning n."""
    x2 = Fraction(units * units * i, m)          # x^2, exact
    for n in range(units + 2):
        lo = Fraction(2 * n - 1, 2)
        hi = Fraction(2 * n + 1, 2)
        lo_ok = lo <= 0 or lo * lo <= x2
        hi_ok = x2 < hi * hi
        if lo_ok and hi_ok:
            return n
    raise AssertionError("no n found")


@pytest.mark.parametrize("units", [1, 2, 3, 5, 8, 13, 32, 64])
def test_rounding_matches_rational_brute_force(units):
    for m in range(1, min(units, 16) + 1):
        for i in range(m):
            assert P._round_half_up_sqrt(i, m, units) == _brute_round_half_up_sqrt(i, m, units)


def test_rounding_matches_float_away_from_ties():
    rnd = random.Random(7)
    for _ in range(3000):
        units = rnd.randint(1, 4096)
        m = rnd.randint(1, 64)
        i = rnd.randint(0, m - 1)
        x = units * math.sqrt(i / m)
        if abs((x % 1.0) - 0.5) < 1e-7:
            continue
        assert P._round_half_up_sqrt(i, m, units) == math.floor(x + 0.5)


def _check_invariants(b, seq_len, m, g):
    assert len(b) == m + 1
    assert b[0] == 0 and b[-1] == seq_len
    for i in range(1, m):
        assert b[i] % g == 0
        assert b[i] - b[i - 1] >= g
    assert b[m] - b[m - 1] >= g


@pytest.mark.parametrize("mode", [P.LBCP, P.UNIFORM])
def test_invariants_small_exhaustive(mode):
    for units in range(1, 65):
        for m in range(1, min(units, 16) + 1):
            for extra in (0, 1, 77):
                s = units * G + extra
                _check_invariants(P.boundaries(s, m, G, mode), s, m, G)


def test_clamp_is_noop_when_rounding_is_already_valid():
    for units in range(4, 200):
        for m in range(1, min(units, 12) + 1):
            raw = [_brute_round_half_up_sqrt(i, m, units) for i in range(m)] + [units]
            if all(raw[i + 1] - raw[i] >= 1 for i in range(m)):
                assert P.boundaries(units * G, m, G) == [G * n for n in raw]


def test_closed_form_at_rational_square_roots():
    # b_i = S * sqrt(i / M) exactly when i/M is a square of a rational.
    s, m = 32768, 16
    b = P.boundaries(s, m, G)
    assert b[1] == s // 4 and b[4] == s // 2 and b[9] == 3 * s // 4 and b[16] == s
    s, m = 131072, 32
    b = P.boundaries(s, m, G)
    assert b[2] == s // 4 and b[8] == s // 2 and b[18] == 3 * s // 4
    s, m = 8192, 4
    b = P.boundaries(s, m, G)
    assert b[1] == s // 2


def test_real_closed_form_balances_cost():
    # With b_i = S sqrt(i/M), c_i (p_i + c_i/2) = S^2 / (2M) for every chunk.
    s, m = 131072.0, 32
    b = [s * math.sqrt(i / m) for i in range(m + 1)]
    costs = [(b[i + 1] - b[i]) * (b[i] + (b[i + 1] - b[i]) / 2) for i in range(m)]
    for c in costs:
        assert c == pytest.approx(s * s / (2 * m), rel=1e-12)


def test_cost_telescopes_for_any_split():
    rnd = random.Random(3)
    for _ in range(200):
        s = rnd.randint(2, 5000)
        cuts = sorted(rnd.sample(range(1, s), k=min(s - 1, rnd.randint(1, 9))))
        b = [0] + cuts + [s]
        c2 = P.chunk_cost_x2(b)
        assert sum(c2) == s * s
        for i in range(len(b) - 1):
            assert c2[i] == b[i + 1] ** 2 - b[i] ** 2


def test_causal_pairs_brute_force():
    rnd = random.Random(5)
    for _ in range(40):
        s = rnd.randint(1, 60)
        cuts = sorted(rnd.sample(range(1, s), k=min(max(s - 1, 0), rnd.randint(0, 5)))) if s > 1 else []
        b = [0] + cuts + [s]
        pairs = P.causal_pairs(b)
        for i in range(len(b) - 1):
            n = sum(1 for t in range(b[i], b[i + 1]) for j in range(s) if j <= t)
            assert pairs[i] == n
        assert sum(pairs) == s * (s + 1) // 2


def test_eq1_cost_form():
    b = [0, 3, 7, 12]
    # c_i * (p_i + c_i) with p_i the prefix: 3*3, 4*7, 5*12
    assert P.eq1_cost(b) == [9, 28, 60]


@pytest.mark.parametrize("s,m", [(32768, 16), (131072, 32), (65536, 8)])
def test_lbcp_spread_far_below_uniform(s, m):
    lb = P.chunk_cost_x2(P.boundaries(s, m, G, P.LBCP))
    un = P.chunk_cost_x2(P.boundaries(s, m, G, P.UNIFORM))
    # uniform: cost_i proportional to 2i+1, spread exactly 2M-1
    assert max(un) == (2 * m - 1) * min(un)
    assert max(lb) / min(lb) < 1.25
    # later chunks are shorter (Sec. 3.2 insight), up to one rounding step
    b = P.boundaries(s, m, G, P.LBCP)
    c = [b[i + 1] - b[i] for i in range(m)]
    for i in range(m - 1):
        assert c[i + 1] <= c[i] + G


def test_uniform_configs_exact():
    assert P.boundaries(1024, 4, G, P.UNIFORM) == [0, 256, 512, 768, 1024]
    assert P.boundaries(8192, 8, G, P.UNIFORM) == [1024 * i for i in range(9)]


def test_invalid_arguments():
    for args in [(0, 1, G), (1024, 0, G), (1024, 9, G), (100, 1, 128), (1024, 2, 0)]:
        with pytest.raises(ValueError):
            P.boundaries(*args)


def _read_golden():
    path = os.path.join(os.path.dirname(__file__), "golden", "partition_boundaries.txt")
    rows = []
    with open(path) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            head, vals = line.split(":")
            s, m, g, mode = (int(x) for x in head.split())
            rows.append(((s, m, g, mode), [int(x) for x in vals.split()]))
    return rows


def test_golden_boundaries():
    rows = _read_golden()
    assert len(rows) >= 8
    for (s, m, g, mode), b in rows:
        assert P.boundaries(s, m, g, mode) == b
