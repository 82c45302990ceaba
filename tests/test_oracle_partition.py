"""Pins for the partition oracle (Sec. 3.2 / Eq. 1, Sec. 4.2).

None of these re-types the oracle's isqrt formula: rounding is checked by
exact rational interval membership and by floating point away from ties, the
cost model by its algebra and by brute-force pair counting, the clamps by
invariants, and the closed form at the boundaries where sqrt(i/M) is rational.
"""

import functools
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


# ---------------------------------------------------------------- Algorithm 1 DP --
def _compositions(total, parts):
    """All ways to write `total` units as `parts` positive sizes."""
    if parts == 1:
        yield (total,)
        return
    for first in range(1, total - parts + 2):
        for rest in _compositions(total - first, parts - 1):
            yield (first,) + rest


@functools.lru_cache(maxsize=None)
def _brute_cost(k, s, model, gemm):
    """Chunk cost from counted (query, key) pairs, independent of the oracle.

    Causal: twice c (p + c/2) = twice the causal pair count minus c (the
    pair count is c p + c (c + 1) / 2).  Eq. 1: twice c (p + c), every key up
    to the chunk end for every query of the chunk.  Plus gemm * c."""
    queries = range(s, s + k)
    if model == P.COST_CAUSAL:
        pairs = sum(1 for t in queries for j in range(s + k) if j <= t)
        attn = 2 * pairs - k
    else:
        attn = 2 * sum(1 for t in queries for j in range(s + k))
    return attn + gemm * k


def _chunk_costs(sizes, model, gemm):
    s, out = 0, []
    for k in sizes:
        out.append(_brute_cost(k, s, model, gemm))
        s += k
    return out


@pytest.mark.parametrize("model", [P.COST_CAUSAL, P.COST_EQ1])
def test_evaluate_chunk_counts_pairs(model):
    for k in range(1, 9):
        for s in range(0, 9):
            for gemm in (0, 5):
                assert P.evaluate_chunk(k, s, model, gemm) == _brute_cost(k, s, model, gemm)


@pytest.mark.parametrize("model", [P.COST_CAUSAL, P.COST_EQ1])
@pytest.mark.parametrize("gemm", [0, 3, 40])
def test_dp_single_stage_minimises_total_cost(model, gemm):
    # N = 1: the objective is t_sum alone, which decomposes over chunks, so the
    # suffix recursion is exact: the DP total equals the brute-force minimum.
    for units in range(1, 11):
        for m in range(1, min(units, 5) + 1):
            b = P.dp_boundaries(units * 128, m, 128, 1, model, gemm)
            sizes = [(b[i + 1] - b[i]) // 128 for i in range(m)]
            best = min(sum(_chunk_costs(c, model, gemm)) for c in _compositions(units, m))
            assert sum(_chunk_costs(sizes, model, gemm)) == best


@pytest.mark.parametrize("model", [P.COST_CAUSAL, P.COST_EQ1])
@pytest.mark.parametrize("gemm", [0, 7])
def test_dp_many_stages_reaches_the_minimax_chunk(model, gemm):
    # (N - 1) larger than any possible t_sum: comparisons are lexicographic in
    # (t_max, t_sum), every kept suffix has the least t_max, and max(t, .) is
    # monotone, so the DP's largest chunk cost is the brute-force minimax.
    for units in range(1, 12):
        for m in range(1, min(units, 5) + 1):
            n_stages = 10 ** 9
            b = P.dp_boundaries(units * 128, m, 128, n_stages, model, gemm)
            sizes = [(b[i + 1] - b[i]) // 128 for i in range(m)]
            best = min(max(_chunk_costs(c, model, gemm)) for c in _compositions(units, m))
            assert max(_chunk_costs(sizes, model, gemm)) == best


def test_dp_invariants_and_remainder():
    for s, m, n in [(1000, 3, 4), (32768, 16, 16), (640, 5, 2), (100000, 9, 16)]:
        b = P.dp_boundaries(s, m, 128 if s != 100000 else 64, n)
        g = 128 if s != 100000 else 64
        _check_invariants(b, s, m, g)


def test_dp_causal_cost_telescopes():
    # with the causal model and no GEMM term every partition has t_sum = U^2
    for units, m in [(7, 3), (12, 4), (20, 6)]:
        b = P.dp_boundaries(units * 128, m, 128, 8)
        sizes = [(b[i + 1] - b[i]) // 128 for i in range(m)]
        assert sum(_chunk_costs(sizes, P.COST_CAUSAL, 0)) == units * units


def test_dp_beats_closed_form_objective_on_workload_shapes():
    for s, m in [(32768, 16), (8192, 8)]:
        dp = P.dp_boundaries(s, m, 128, 16)
        cf = P.boundaries(s, m, 128)
        assert P.dp_objective(dp, 128, 16) <= P.dp_objective(cf, 128, 16)


# ---------------------------------------------------------------------------
# Algorithm 1's exact output under ties (Sec. 4.2, stage 1): the table of a
# case worked by hand from the algorithm's steps (tests/golden/dp_tie_case.txt)
# fixes which of several equal-objective splits the DP keeps.
from tests.golden_utils import dp_boundary_rows, dp_tie_case  # noqa: E402


def test_dp_tables_match_the_hand_worked_tie_case():
    case, states, terminal, bounds = dp_tie_case()
    t_max, t_sum, ss = P.dp_tables(case["units"], case["chunks"], case["stages"],
                                   case["model"], case["gemm"])
    got = {key: (ss[key], t_max[key], t_sum[key]) for key in ss}
    assert got == states
    m_end, s_end, tmax_end, tsum_end = terminal
    assert (t_max[(m_end, s_end)], t_sum[(m_end, s_end)]) == (tmax_end, tsum_end)
    assert set(t_max) == set(states) | {(m_end, s_end)}  # no other state is reached
    assert P.dp_boundaries(case["seq_len"], case["chunks"], case["granularity"], case["stages"],
                           case["model"], case["gemm"]) == bounds


def test_hand_worked_case_has_two_optima_brute_force():
    # independent of the DP: the objective t_sum + (N - 1) t_max over every
    # composition of 6 units into 3 chunks has two minimisers; the golden
    # boundaries are one of them
    case, _, _, bounds = dp_tie_case()
    n = case["stages"]
    objs = {}
    for sizes in _compositions(case["units"], case["chunks"]):
        costs = _chunk_costs(sizes, P.COST_CAUSAL, 0)
        objs[sizes] = sum(costs) + (n - 1) * max(costs)
    best = min(objs.values())
    optima = sorted(s for s, v in objs.items() if v == best)
    assert optima == [(3, 2, 1), (4, 1, 1)]
    g = case["granularity"]
    assert tuple((bounds[i + 1] - bounds[i]) // g for i in range(3)) == (3, 2, 1)


def _mutant_dp(replace_from, replace_to):
    """The oracle's dp_tables with one planted change, compiled on the CPU."""
    import inspect
    src = inspect.getsource(P.dp_tables)
    assert src.count(replace_from) == 1, replace_from
    ns = dict(P.__dict__)
    exec(src.replace(replace_from, replace_to), ns)
    return ns["dp_tables"]


@pytest.mark.parametrize("mutation", [
    ("tsum_new + (N - 1) * tmax_new < t_sum[cur]", "tsum_new + (N - 1) * tmax_new <= t_sum[cur]"),
    ("range(1, S - s - (M - m) + 1)", "range(S - s - (M - m), 0, -1)"),
])
def test_reversed_tie_rule_fails_the_hand_worked_case(mutation):
    # a "<=" comparison or k tried downward keeps the same objective values
    # but a different split, which the golden table catches
    case, states, _, _ = dp_tie_case()
    dp = _mutant_dp(*mutation)
    t_max, t_sum, ss = dp(case["units"], case["chunks"], case["stages"], case["model"],
                          case["gemm"])
    assert (t_max[(1, 0)], t_sum[(1, 0)]) == states[(1, 0)][1:]  # same objective ...
    assert ss[(1, 0)] != states[(1, 0)][0]                      # ... other split


def test_dp_golden_rows_of_the_32k_shape():
    # the rows written by make_golden.py from the oracle alone; re-derived here
    # for the 32768-token shape (the 131072-token rows take minutes in Python)
    rows = [r for r in dp_boundary_rows() if r[0] == 32768]
    assert len(rows) == 3
    for s, m, g, n, model, gemm, b in rows:
        assert P.dp_boundaries(s, m, g, n, model, gemm) == b
        _check_invariants(b, s, m, g)


# ---------------------------------------------------------------------------
# Algorithm 1 stage 1 with EvaluateChunk = the kernel's compute-latency model.
C, T = P.CTA_PS, P.TILE_PS


def test_latency_model_hand_worked_cases():
    # 2 SMs, 1 query head per KV head (one CTA per KV head and row block),
    # 2 KV heads, 256 rows at prefix 0: row block 1 = 2 CTAs of 2 tiles, row
    # block 0 = 2 CTAs of 1 tile; list scheduling puts one of each on each SM
    assert P.chunk_latency_ps(0, 256, 2, 2, 128, 2, 1) == 2 * C + 3 * T
    # 3 SMs: the third SM takes one 1-tile CTA, then the last one (least loaded)
    assert P.chunk_latency_ps(0, 256, 2, 2, 128, 3, 1) == 2 * C + 2 * T
    # d = 64 halves the tile cost
    assert P.chunk_latency_ps(0, 256, 2, 2, 64, 2, 1) == 2 * C + 3 * (T // 2)
    # two splits of a one-block chunk with two key tiles: one tile each on two
    # SMs, plus the merge of 128 rows x 1 head: 3 us + bytes / 5 ps
    moved = 128 * 1 * (2 * (4 * 128 + 4) + 2 * 128 + 4)
    assert P.chunk_latency_ps(128, 128, 1, 1, 128, 2, 2) == C + T + P.COMBINE_FIXED_PS + moved // 5
    # a ragged chunk: 130 rows at prefix 0 = row blocks of 1 and 2 tiles
    assert P.chunk_latency_ps(0, 130, 1, 1, 128, 1, 1) == 2 * C + 3 * T
    # four query heads per KV head = two CTAs per KV head and row block
    assert P.chunk_latency_ps(0, 128, 4, 1, 128, 1, 1) == 2 * (C + T)


def test_latency_model_bounds():
    import random
    rnd = random.Random(4)
    for _ in range(200):
        prefix = rnd.randint(0, 3000)
        length = rnd.randint(1, 2000)
        hkv = rnd.choice([1, 2, 4])
        hq = hkv * rnd.choice([1, 2, 4, 8])
        sms = rnd.choice([1, 3, 8, 152])
        t = P.chunk_latency_ps(prefix, length, hq, hkv, 128, sms, 1)
        q_blocks = (length + 127) // 128
        per_block = hkv * ((hq // hkv + 1) // 2)
        jobs = []
        for qb in range(q_blocks):
            tiles = (min(prefix + 128 * (qb + 1), prefix + length) + 127) // 128
            jobs += [C + T * tiles] * per_block
        assert t >= max(jobs) and t * sms >= sum(jobs)
        assert t <= sum(jobs) // sms + max(jobs)            # list-scheduling bound
        best = P.chunk_latency_best_ps(prefix, length, hq, hkv, 128, sms)
        assert best <= t


def test_latency_dp_window_zero_is_the_closed_form():
    for s, m in [(32768, 16), (8192, 8), (5000, 5)]:
        assert P.dp_latency_boundaries(s, m, 16, 32, 8, 128, 152, 0) == P.boundaries(s, m, 128)


def _lat_costs(sizes, hq, hkv, sms):
    s, out = 0, []
    for k in sizes:
        out.append(P.chunk_latency_best_ps(128 * s, 128 * k, hq, hkv, 128, sms))
        s += k
    return out


@pytest.mark.parametrize("hq,hkv,sms", [(2, 1, 3), (8, 2, 5), (4, 4, 2)])
def test_latency_dp_reaches_the_brute_force_optimum(hq, hkv, sms):
    # windows wider than the prompt: the DP ranges over every split, so with
    # N = 1 it minimises the total and with (N - 1) above any total it reaches
    # the minimax chunk latency (the objective's two extremes)
    for units in range(2, 10):
        for m in range(1, min(units, 4) + 1):
            comps = list(_compositions(units, m))
            b1 = P.dp_latency_boundaries(128 * units, m, 1, hq, hkv, 128, sms, units)
            got = _lat_costs([(b1[i + 1] - b1[i]) // 128 for i in range(m)], hq, hkv, sms)
            assert sum(got) == min(sum(_lat_costs(c, hq, hkv, sms)) for c in comps)
            bn = P.dp_latency_boundaries(128 * units, m, 10 ** 12, hq, hkv, 128, sms, units)
            got = _lat_costs([(bn[i + 1] - bn[i]) // 128 for i in range(m)], hq, hkv, sms)
            assert max(got) == min(max(_lat_costs(c, hq, hkv, sms)) for c in comps)


def test_latency_dp_stays_in_its_window_and_lowers_the_modelled_maximum():
    s, m, w = 32768, 16, 6
    closed = P.boundaries(s, m, 128)
    dp = P.dp_latency_boundaries(s, m, 10 ** 12, 32, 8, 128, 152, w)
    _check_invariants(dp, s, m, 128)
    assert all(abs(a - b) <= 128 * w for a, b in zip(dp, closed))
    lat = lambda b: [P.chunk_latency_best_ps(b[i], b[i + 1] - b[i], 32, 8, 128, 152)
                     for i in range(m)]
    assert max(lat(dp)) <= max(lat(closed))
