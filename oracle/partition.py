"""Chunk-boundary oracle for Latency-Balanced Chunk Partitioning (TEST INFRASTRUCTURE).

Test infrastructure only (see ``oracle/__init__.py``); the product path never
imports this module.

What the paper fixes
--------------------
Sec. 3.2, Eq. 1: the attention cost of chunk ``i`` with length ``c_i`` and
prefix ``p_i = c_1 + ... + c_{i-1}`` grows with ``c_i`` times the number of keys
it sees, while the GEMM part grows with ``c_i`` alone.  Sec. 3.2 (Insight) and
Sec. 4.2: later chunks are made shorter so that chunk costs are balanced;
stage 1 of Algorithm 1 builds a compute-balanced split.

Readings taken here (the paper gives no closed rule):

* cost_i = c_i * (p_i + c_i / 2), the number of (query, key) pairs of a causal
  chunk up to the O(c_i) diagonal term.  Then
  ``2 * cost_i = b_{i+1}^2 - b_i^2`` with ``b_i = p_i`` the chunk start, so the
  total cost telescopes to ``S^2 / 2`` for ANY split and equal costs give the
  closed form ``b_i = S * sqrt(i / M)``.
* Boundaries are multiples of the granularity ``g``: with ``U = S // g``,
  ``n_i = round_half_up(U * sqrt(i / M))`` (computed exactly in integers as the
  largest ``n >= 0`` with ``n == 0`` or ``M * (2n - 1)^2 <= 4 * i * U^2``),
  ``b_i = g * n_i``.
* Clamp in one forward pass so every chunk has at least ``g`` tokens:
  ``b_i = min(max(b_i, b_{i-1} + g), g * (U - (M - i)))``; ``b_0 = 0``,
  ``b_M = S`` (the last chunk absorbs ``S % g``).
* Uniform mode (used for the two small configurations): ``n_i =
  round_half_up(i * U / M)`` with the same clamps.

Everything is exact Python integer arithmetic (``math.isqrt``), so the result
is bit-exact by construction.
"""

from __future__ import annotations

import math
from typing import List

UNIFORM = 0
LBCP = 1


def _check(seq_len: int, num_chunks: int, granularity: int) -> int:
    if seq_len <= 0 or num_chunks < 1 or granularity < 1:
        raise ValueError("seq_len > 0, num_chunks >= 1, granularity >= 1 required")
    if num_chunks * granularity > seq_len:
        raise ValueError("num_chunks * granularity must not exceed seq_len")
    return seq_len // granularity


def _round_half_up_sqrt(i: int, num_chunks: int, units: int) -> int:
    """round_half_up(units * sqrt(i / num_chunks)) exactly.

    round_half_up(x) = n  <=>  n - 1/2 <= x < n + 1/2.  For n >= 1 the left
    side is (2n - 1)^2 <= 4 x^2 = 4 i U^2 / M; the largest odd q = 2n - 1 with
    q^2 <= 4 i U^2 / M is isqrt(floor(4 i U^2 / M)).
    """
    q = math.isqrt((4 * i * units * units) // num_chunks)
    return (q + 1) // 2


def _round_half_up_ratio(i: int, num_chunks: int, units: int) -> int:
    """round_half_up(i * units / num_chunks) exactly."""
    return (2 * i * units + num_chunks) // (2 * num_chunks)


def boundaries(seq_len: int, num_chunks: int, granularity: int = 128,
               mode: int = LBCP) -> List[int]:
    """Chunk boundaries ``[b_0 = 0, b_1, ..., b_M = seq_len]``.

    ``mode`` is ``LBCP`` (equal cost_i, Sec. 3.2 / Sec. 4.2) or ``UNIFORM``.
    """
    units = _check(seq_len, num_chunks, granularity)
    if mode == LBCP:
        raw = [_round_half_up_sqrt(i, num_chunks, units) for i in range(num_chunks)]
    elif mode == UNIFORM:
        raw = [_round_half_up_ratio(i, num_chunks, units) for i in range(num_chunks)]
    else:
        raise ValueError("unknown partition mode")
    out = [0]
    for i in range(1, num_chunks):
        b = granularity * raw[i]
        b = max(b, out[-1] + granularity)
        b = min(b, granularity * (units - (num_chunks - i)))
        out.append(b)
    out.append(seq_len)
    return out


def chunk_cost_x2(bounds: List[int]) -> List[int]:
    """Twice the per-chunk attention cost, ``2 * c_i * (p_i + c_i / 2)``.

    Written with the chunk length and prefix of Eq. 1 (not with the
    telescoped squares) so that the telescoping identity can be tested.
    """
    costs = []
    for i in range(len(bounds) - 1):
        p = bounds[i]
        c = bounds[i + 1] - bounds[i]
        costs.append(c * (2 * p + c))
    return costs


def eq1_cost(bounds: List[int]) -> List[int]:
    """Eq. 1 as printed, ``c_i * (p_i + c_i)`` (used only for comparison)."""
    return [(bounds[i + 1] - bounds[i]) * (bounds[i + 1]) for i in range(len(bounds) - 1)]


def causal_pairs(bounds: List[int]) -> List[int]:
    """Exact number of causal (query, key) pairs per chunk,
    ``c_i * p_i + c_i * (c_i + 1) / 2`` (the attention FLOP count / (4 H d))."""
    out = []
    for i in range(len(bounds) - 1):
        p = bounds[i]
        c = bounds[i + 1] - bounds[i]
        out.append(c * p + c * (c + 1) // 2)
    return out


# ---------------------------------------------------------------------------
# Algorithm 1, stage 1 (Sec. 4.2): the compute-balanced DP initialisation.
#
# Positions and chunk sizes are counted in units of the granularity g
# (U = S // g units; the last chunk absorbs S % g tokens).  EvaluateChunk(k, s)
# is the compute cost of a chunk of k units starting at unit s, doubled so it
# stays an integer:
#   COST_CAUSAL: 2 * k (s + k/2) = k (2 s + k)      (c_i (p_i + c_i / 2))
#   COST_EQ1:    2 * k (s + k)                       (Eq. 1 as printed)
# plus gemm_weight * k for the GEMM term of Eq. 1 (cost proportional to c_i).
# Suffix states (m, s) keep one (t_max, t_sum) pair: the one minimising
# t_sum + (N - 1) t_max over the chunk sizes k tried in increasing order
# (strict improvement, so the smallest k wins ties).

COST_CAUSAL = 0
COST_EQ1 = 1


def evaluate_chunk(k: int, s: int, model: int, gemm_weight: int) -> int:
    if model == COST_CAUSAL:
        attn = k * (2 * s + k)
    elif model == COST_EQ1:
        attn = 2 * k * (s + k)
    else:
        raise ValueError("unknown cost model")
    return attn + gemm_weight * k


def dp_tables(units: int, num_chunks: int, num_stages: int, model: int = COST_CAUSAL,
              gemm_weight: int = 0):
    """The three tables of Algorithm 1's stage-1 DP over ``units`` positions.

    Returns dicts ``t_max``, ``t_sum`` and ``ss`` keyed by ``(m, s)`` (chunk
    index m in 1..M, start position s); a state that no valid suffix reaches
    has no key (its objective counts as +infinity).  The terminal state
    ``(M + 1, units)`` has ``t_max = t_sum = 0``.
    """
    if units < num_chunks or num_chunks < 1:
        raise ValueError("1 <= num_chunks <= units required")
    if num_stages < 1 or gemm_weight < 0:
        raise ValueError("num_stages >= 1 and gemm_weight >= 0 required")
    M, S, N = num_chunks, units, num_stages
    t_max = {(M + 1, S): 0}
    t_sum = {(M + 1, S): 0}
    ss = {}
    for m in range(M, 0, -1):                      # chunk index, last first
        for s in range(S - 1, -1, -1):             # start position, right to left
            for k in range(1, S - s - (M - m) + 1):  # candidate chunk size
                nxt = (m + 1, s + k)
                if nxt not in t_max:
                    continue
                t = evaluate_chunk(k, s, model, gemm_weight)
                tmax_new = max(t_max[nxt], t)
                tsum_new = t_sum[nxt] + t
                cur = (m, s)
                if cur not in t_max or \
                        tsum_new + (N - 1) * tmax_new < t_sum[cur] + (N - 1) * t_max[cur]:
                    t_max[cur], t_sum[cur], ss[cur] = tmax_new, tsum_new, k
    return t_max, t_sum, ss


def dp_boundaries(seq_len: int, num_chunks: int, granularity: int, num_stages: int,
                  model: int = COST_CAUSAL, gemm_weight: int = 0) -> List[int]:
    """Chunk boundaries from stage 1 of Algorithm 1 (exact integers): the
    chunk slice scheme ``ss`` read forward from state (1, 0)."""
    units = _check(seq_len, num_chunks, granularity)
    _, _, ss = dp_tables(units, num_chunks, num_stages, model, gemm_weight)
    out, s = [0], 0
    for m in range(1, num_chunks + 1):
        s += ss[(m, s)]
        out.append(granularity * s)
    out[-1] = seq_len
    return out


def dp_objective(bounds: List[int], granularity: int, num_stages: int,
                 model: int = COST_CAUSAL, gemm_weight: int = 0) -> int:
    """t_sum + (N - 1) t_max of a partition whose interior boundaries are
    multiples of the granularity (units as in dp_boundaries)."""
    units = [b // granularity for b in bounds[:-1]] + [bounds[-1] // granularity]
    costs = [evaluate_chunk(units[i + 1] - units[i], units[i], model, gemm_weight)
             for i in range(len(units) - 1)]
    return sum(costs) + (num_stages - 1) * max(costs)


# ---------------------------------------------------------------------------
# Algorithm 1, stage 1 with EvaluateChunk as a compute-latency model of the
# chunk attention kernel (Sec. 4.2: "EvaluateChunk returns the compute
# latency t").  The model, in integer picoseconds so that it is exact:
#   * a chunk of `length` rows at `prefix` has ceil(length / 128) query row
#     blocks; row block qb sees keys up to min(prefix + 128 (qb + 1),
#     prefix + length), i.e. tiles(qb) = ceil(that / 128) key tiles of 128;
#   * each row block is Hkv * ceil((Hq / Hkv) / 2) CTAs (two query heads per
#     CTA), each split into `splits` contiguous key ranges of
#     floor((j + 1) tiles / splits) - floor(j tiles / splits) tiles;
#   * a CTA costs CTA_PS + TILE_PS * (d / 128) per tile; CTAs are taken
#     heaviest row block first and each goes to a least-loaded SM of `sms`
#     (list scheduling); the chunk's time is the largest SM load;
#   * with splits > 1 the merge adds COMBINE_FIXED_PS + (bytes moved) / 5 ps
#     (bytes = length Hq (splits (4 d + 4) + 2 d + 4)), and the chunk takes the
#     split count 1..4 with the smallest time (more than one only when the
#     chunk has fewer than 8 sms CTAs, and at most the first row block's
#     tile count);
# the constants are the ones the library's split planner uses.

TILE_PS = 1400000
CTA_PS = 4000000
COMBINE_FIXED_PS = 3000000
MAX_SPLITS = 4


def chunk_latency_ps(prefix: int, length: int, n_q_heads: int, n_kv_heads: int, head_dim: int,
                     sms: int, splits: int) -> int:
    """Modelled time of one chunk's attention launch with `splits` key
    ranges (list scheduling of its CTAs over `sms` SMs), picoseconds."""
    import heapq
    group = n_q_heads // n_kv_heads
    per_block = n_kv_heads * ((group + 1) // 2)
    tile_ps = TILE_PS * head_dim // 128
    q_blocks = (length + 127) // 128
    loads = [0] * sms
    for qb in range(q_blocks - 1, -1, -1):
        kv_end = min(prefix + 128 * (qb + 1), prefix + length)
        tiles = (kv_end + 127) // 128
        for _ in range(per_block):
            for j in range(splits):
                nk = (j + 1) * tiles // splits - j * tiles // splits
                least = heapq.heappop(loads)
                heapq.heappush(loads, least + CTA_PS + tile_ps * nk)
    t = max(loads)
    if splits > 1:
        moved = length * n_q_heads * (splits * (4 * head_dim + 4) + 2 * head_dim + 4)
        t += COMBINE_FIXED_PS + moved // 5
    return t


def chunk_latency_best_ps(prefix: int, length: int, n_q_heads: int, n_kv_heads: int,
                          head_dim: int, sms: int) -> int:
    """The model's time with the split count it would choose (see above)."""
    group = n_q_heads // n_kv_heads
    ctas = ((length + 127) // 128) * n_kv_heads * ((group + 1) // 2)
    best = chunk_latency_ps(prefix, length, n_q_heads, n_kv_heads, head_dim, sms, 1)
    if ctas >= 8 * sms:
        return best
    first_tiles = (min(prefix + 128, prefix + length) + 127) // 128
    for sp in range(2, min(MAX_SPLITS, first_tiles) + 1):
        best = min(best, chunk_latency_ps(prefix, length, n_q_heads, n_kv_heads, head_dim, sms,
                                          sp))
    return best


def dp_latency_boundaries(seq_len: int, num_chunks: int, num_stages: int, n_q_heads: int,
                          n_kv_heads: int, head_dim: int, sms: int, window: int) -> List[int]:
    """Algorithm 1's stage-1 DP (loops and strict-improvement rule as in
    dp_tables) with EvaluateChunk = chunk_latency_best_ps, over 128-row units,
    each interior boundary restricted to `window` units either side of the
    closed-form split's (``boundaries(seq_len, num_chunks, 128)``).  The last
    chunk ends at seq_len (absorbing seq_len % 128)."""
    if window < 0:
        raise ValueError("window >= 0 required")
    g = 128
    units = _check(seq_len, num_chunks, g)
    M, U, N = num_chunks, units, num_stages
    if N < 1:
        raise ValueError("num_stages >= 1 required")
    closed = [b // g for b in boundaries(seq_len, num_chunks, g)]
    closed[-1] = U

    def allowed(m):  # unit positions boundary m may take
        if m == 0:
            return [0]
        if m == M:
            return [U]
        lo = max(m, closed[m] - window)
        hi = min(U - (M - m), closed[m] + window)
        return list(range(lo, hi + 1))

    def evaluate(s, k):
        length = seq_len - g * s if s + k == U else g * k
        return chunk_latency_best_ps(g * s, length, n_q_heads, n_kv_heads, head_dim, sms)

    t_max = {(M + 1, U): 0}
    t_sum = {(M + 1, U): 0}
    ss = {}
    for m in range(M, 0, -1):
        ends = set(allowed(m))
        for s in sorted(allowed(m - 1), reverse=True):
            for k in range(1, U - s - (M - m) + 1):
                if s + k not in ends:
                    continue
                nxt = (m + 1, s + k)
                if nxt not in t_max:
                    continue
                t = evaluate(s, k)
                tmax_new = max(t_max[nxt], t)
                tsum_new = t_sum[nxt] + t
                cur = (m, s)
                if cur not in t_max or \
                        tsum_new + (N - 1) * tmax_new < t_sum[cur] + (N - 1) * t_max[cur]:
                    t_max[cur], t_sum[cur], ss[cur] = tmax_new, tsum_new, k
    out, s = [0], 0
    for m in range(1, M + 1):
        s += ss[(m, s)]
        out.append(g * s)
    out[-1] = seq_len
    return out
