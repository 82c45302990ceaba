// lbcp.cpp -- Latency-Balanced Chunk Partitioning boundaries (host, exact).
//
// Sec. 3.2 / Eq. 1: attention cost of chunk i grows with c_i times the keys it
// sees; we balance cost_i = c_i * (p_i + c_i / 2).  Because 2 * cost_i =
// b_{i+1}^2 - b_i^2, equal costs mean b_i = S * sqrt(i / M) (the
// compute-balanced split that seeds Algorithm 1, Sec. 4.2).  The boundaries
// are snapped to a granularity g with integer-only arithmetic so that every
// platform produces the same bits:
//   U = S / g,  n_i = round_half_up(U * sqrt(i / M))
//     = (q + 1) / 2 with q = isqrt(floor(4 i U^2 / M)),
//   b_i = min(max(g n_i, b_{i-1} + g), g (U - (M - i))),  b_0 = 0, b_M = S.
// Uniform mode: n_i = round_half_up(i U / M) = floor((2 i U + M) / (2 M)).
#include <cstdint>
#include <vector>

#include "internal.h"

namespace {

// floor(sqrt(x)) for x < 2^62, exact.
uint64_t isqrt_u64(uint64_t x) {
  // bitwise restoring square root: no floating point involved
  uint64_t rem = x, root = 0, bit = 1ull << 62;
  while (bit > rem) bit >>= 2;
  while (bit != 0) {
    if (rem >= root + bit) {
      rem -= root + bit;
      root = (root >> 1) + bit;
    } else {
      root >>= 1;
    }
    bit >>= 2;
  }
  return root;
}

}  // namespace

extern "C" mocap_status mocap_lbcp_partition(int64_t seq_len, int32_t num_chunks,
                                             int32_t granularity, mocap_part_mode mode,
                                             int64_t *boundaries) {
  if (boundaries == nullptr || seq_len <= 0 || num_chunks < 1 || granularity < 1)
    return MOCAP_EINVAL;
  if (mode != MOCAP_PART_UNIFORM && mode != MOCAP_PART_LBCP) return MOCAP_EINVAL;
  if (static_cast<int64_t>(num_chunks) * granularity > seq_len) return MOCAP_EINVAL;
  const uint64_t units = static_cast<uint64_t>(seq_len / granularity);
  if (units >= (1ull << 30)) return MOCAP_EINVAL;  // keeps 4 U^2 below 2^62
  const uint64_t m = static_cast<uint64_t>(num_chunks);
  const int64_t g = granularity;

  boundaries[0] = 0;
  for (uint64_t i = 1; i < m; ++i) {
    uint64_t n;
    if (mode == MOCAP_PART_LBCP) {
      const unsigned __int128 num = static_cast<unsigned __int128>(4u) * i * units * units;
      const uint64_t x = static_cast<uint64_t>(num / m);  // < 4 U^2 < 2^62
      n = (isqrt_u64(x) + 1) / 2;
    } else {
      n = (2 * i * units + m) / (2 * m);
    }
    int64_t b = g * static_cast<int64_t>(n);
    const int64_t lo = boundaries[i - 1] + g;
    const int64_t hi = g * static_cast<int64_t>(units - (m - i));
    if (b < lo) b = lo;
    if (b > hi) b = hi;
    boundaries[i] = b;
  }
  boundaries[m] = seq_len;
  return MOCAP_OK;
}

// ---------------------------------------------------------------------------
// Stage 1 of Algorithm 1 (Sec. 4.2): dynamic programming over (chunk index m,
// start position s, chunk size k), all counted in units of the granularity.
// Suffix state (m, s) keeps the (t_max, t_sum) of the chunk sizes tried so far
// that minimises t_sum + (N - 1) t_max; k is tried in increasing order and
// only a strict improvement replaces the kept choice.  EvaluateChunk is the
// chunk's compute cost, doubled to stay integral: k (2 s + k) for the causal
// count c (p + c/2), 2 k (s + k) for Eq. 1 as printed, plus gemm_weight * k.
extern "C" mocap_status mocap_lbcp_partition_dp(int64_t seq_len, int32_t num_chunks,
                                                int32_t granularity, int32_t num_stages,
                                                mocap_cost_model model, int64_t gemm_weight,
                                                int64_t *boundaries) {
  if (boundaries == nullptr || seq_len <= 0 || num_chunks < 1 || granularity < 1 ||
      num_stages < 1 || gemm_weight < 0)
    return MOCAP_EINVAL;
  if (model != MOCAP_COST_CAUSAL && model != MOCAP_COST_EQ1) return MOCAP_EINVAL;
  if (static_cast<int64_t>(num_chunks) * granularity > seq_len) return MOCAP_EINVAL;
  const int64_t U = seq_len / granularity;
  const int64_t M = num_chunks;
  if (static_cast<double>(M) * static_cast<double>(U) * static_cast<double>(U) > 4e9)
    return MOCAP_EUNSUPPORTED;  // O(M U^2) host work; use a coarser granularity
  if (gemm_weight > (int64_t(1) << 40)) return MOCAP_EINVAL;
  // Every chunk cost is at most 2 U^2 + gemm_weight U (Eq. 1's form with
  // s + k <= U), so t_sum and t_max are too, and the compared objective
  // t_sum + (N - 1) t_max is at most N (2 U^2 + gemm_weight U).  Refuse
  // arguments for which that bound could leave int64.
  {
    const unsigned __int128 t_bound = static_cast<unsigned __int128>(2) * U * U +
                                      static_cast<unsigned __int128>(gemm_weight) * U;
    if (t_bound * static_cast<unsigned __int128>(num_stages) >=
        (static_cast<unsigned __int128>(1) << 62))
      return MOCAP_EINVAL;
  }
  const int64_t nm1 = num_stages - 1;
  const size_t W = static_cast<size_t>(U + 1);
  auto at = [&](int64_t m, int64_t s) { return static_cast<size_t>(m) * W + static_cast<size_t>(s); };
  std::vector<int64_t> t_max(static_cast<size_t>(M + 2) * W, 0), t_sum(t_max.size(), 0);
  std::vector<uint8_t> set(t_max.size(), 0);
  std::vector<int32_t> ss(t_max.size(), 0);
  set[at(M + 1, U)] = 1;
  for (int64_t m = M; m >= 1; --m) {
    for (int64_t s = U - 1; s >= 0; --s) {
      const size_t cur = at(m, s);
      for (int64_t k = 1; k <= U - s - (M - m); ++k) {
        const size_t nxt = at(m + 1, s + k);
        if (!set[nxt]) continue;
        const int64_t attn = model == MOCAP_COST_CAUSAL ? k * (2 * s + k) : 2 * k * (s + k);
        const int64_t t = attn + gemm_weight * k;
        const int64_t tmax_new = t_max[nxt] > t ? t_max[nxt] : t;
        const int64_t tsum_new = t_sum[nxt] + t;
        if (!set[cur] || tsum_new + nm1 * tmax_new < t_sum[cur] + nm1 * t_max[cur]) {
          t_max[cur] = tmax_new;
          t_sum[cur] = tsum_new;
          ss[cur] = static_cast<int32_t>(k);
          set[cur] = 1;
        }
      }
    }
  }
  if (!set[at(1, 0)]) return MOCAP_EINVAL;
  boundaries[0] = 0;
  int64_t s = 0;
  for (int64_t m = 1; m <= M; ++m) {
    s += ss[at(m, s)];
    boundaries[m] = granularity * s;
  }
  boundaries[M] = seq_len;
  return MOCAP_OK;
}

// Eq. 1 with its GEMM term: a chunk stage costs a * (causal pairs) + b *
// (rows).  In the DP's doubled units of g rows, a chunk of k units at unit s
// has about g^2 k (s + k/2) pairs and g k rows, so its cost is proportional
// to k (2 s + k) + w k with w = 2 b / (g a), rounded to the nearest integer.
extern "C" mocap_status mocap_lbcp_gemm_weight(double attn_s_per_pair, double gemm_s_per_row,
                                               int32_t granularity, int64_t *weight) {
  if (weight == nullptr || granularity < 1) return MOCAP_EINVAL;
  if (!(attn_s_per_pair > 0.0) || !(gemm_s_per_row >= 0.0)) return MOCAP_EINVAL;  // NaN too
  const double w = 2.0 * gemm_s_per_row / (static_cast<double>(granularity) * attn_s_per_pair);
  if (!(w <= static_cast<double>(int64_t(1) << 40))) return MOCAP_EINVAL;  // inf, too large
  *weight = static_cast<int64_t>(w + 0.5);  // w >= 0: round half up
  return MOCAP_OK;
}
