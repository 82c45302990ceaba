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
#include <algorithm>
#include <cstdint>
#include <functional>
#include <unordered_map>
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

// ---------------------------------------------------------------------------
// Stage 1 of Algorithm 1 with EvaluateChunk as a compute-latency model of the
// chunk attention kernel (Sec. 4.2: EvaluateChunk returns the compute
// latency).  The model, in integer picoseconds so that every platform gets
// the same bits: a chunk's CTAs (Hkv * ceil(group / 2) per 128-row block,
// each covering split j of the block's key tiles) are list-scheduled,
// heaviest row block first, each onto a least-loaded SM; a CTA costs
// kCtaPs + kTilePs * (d / 128) per key tile; a split chunk adds the merge,
// kCombineFixedPs + (bytes moved) / 5 ps.  The split count is the one of
// 1..4 with the smallest time (more than one only below 8 CTAs per SM and at
// most the first row block's tile count).  These are the split planner's
// own costs.
namespace {

constexpr int64_t kTilePs = 1400000;
constexpr int64_t kCtaPs = 4000000;
constexpr int64_t kCombineFixedPs = 3000000;
constexpr int kModelMaxSplits = 4;

int64_t chunk_latency_ps(int64_t prefix, int64_t length, int64_t hq, int64_t hkv, int64_t d,
                         int sms, int splits, std::vector<int64_t> &loads) {
  const int64_t per_block = hkv * ((hq / hkv + 1) / 2);
  const int64_t tile_ps = kTilePs * d / 128;
  const int64_t q_blocks = (length + 127) / 128;
  loads.assign(static_cast<size_t>(sms), 0);  // a min-heap (std::greater)
  for (int64_t qb = q_blocks - 1; qb >= 0; --qb) {
    const int64_t kv_end = std::min(prefix + 128 * (qb + 1), prefix + length);
    const int64_t tiles = (kv_end + 127) / 128;
    for (int64_t u = 0; u < per_block; ++u)
      for (int j = 0; j < splits; ++j) {
        const int64_t nk = (j + 1) * tiles / splits - j * tiles / splits;
        std::pop_heap(loads.begin(), loads.end(), std::greater<int64_t>());
        loads.back() += kCtaPs + tile_ps * nk;
        std::push_heap(loads.begin(), loads.end(), std::greater<int64_t>());
      }
  }
  int64_t t = *std::max_element(loads.begin(), loads.end());
  if (splits > 1)
    t += kCombineFixedPs + length * hq * (splits * (4 * d + 4) + 2 * d + 4) / 5;
  return t;
}

int64_t chunk_latency_best_ps(int64_t prefix, int64_t length, int64_t hq, int64_t hkv, int64_t d,
                              int sms, std::vector<int64_t> &loads) {
  const int64_t ctas = ((length + 127) / 128) * hkv * ((hq / hkv + 1) / 2);
  int64_t best = chunk_latency_ps(prefix, length, hq, hkv, d, sms, 1, loads);
  if (ctas >= 8LL * sms) return best;
  const int64_t first_tiles = (std::min(prefix + 128, prefix + length) + 127) / 128;
  for (int sp = 2; sp <= kModelMaxSplits && sp <= first_tiles; ++sp)
    best = std::min(best, chunk_latency_ps(prefix, length, hq, hkv, d, sms, sp, loads));
  return best;
}

}  // namespace

extern "C" mocap_status mocap_lbcp_partition_dp_latency(int64_t seq_len, int32_t num_chunks,
                                                        int32_t num_stages, int32_t n_q_heads,
                                                        int32_t n_kv_heads, int32_t head_dim,
                                                        int32_t num_sms, int32_t window,
                                                        int64_t *boundaries) {
  constexpr int64_t g = 128;
  if (boundaries == nullptr || seq_len <= 0 || seq_len >= (int64_t(1) << 31) ||
      num_chunks < 1 || num_stages < 1 || window < 0)
    return MOCAP_EINVAL;
  if (n_q_heads < 1 || n_kv_heads < 1 || n_q_heads % n_kv_heads != 0 || n_q_heads > 4096)
    return MOCAP_EINVAL;
  if (head_dim != 64 && head_dim != 128) return MOCAP_EUNSUPPORTED;
  if (num_sms < 1 || num_sms > 4096) return MOCAP_EINVAL;
  if (static_cast<int64_t>(num_chunks) * g > seq_len) return MOCAP_EINVAL;
  const int64_t U = seq_len / g;
  const int64_t M = num_chunks;
  const int64_t W = std::min<int64_t>(window, U);
  // the closed-form split the windows are centred on
  std::vector<int64_t> closed(static_cast<size_t>(M + 1));
  const mocap_status cs = mocap_lbcp_partition(seq_len, num_chunks, static_cast<int32_t>(g),
                                               MOCAP_PART_LBCP, closed.data());
  if (cs != MOCAP_OK) return cs;
  std::vector<int64_t> lo(static_cast<size_t>(M + 1)), hi(static_cast<size_t>(M + 1));
  for (int64_t m = 0; m <= M; ++m) {
    if (m == 0) {
      lo[0] = hi[0] = 0;
    } else if (m == M) {
      lo[m] = hi[m] = U;
    } else {
      const int64_t c = closed[static_cast<size_t>(m)] / g;
      lo[m] = std::max(m, c - W);
      hi[m] = std::min(U - (M - m), c + W);
    }
  }
  // host work: every (start, end) pair of neighbouring windows is one chunk
  // evaluation of at most (2 W + U / M-ish) row blocks' CTAs
  const int64_t per_block = n_kv_heads * ((n_q_heads / n_kv_heads + 1) / 2);
  double work = 0.0;
  for (int64_t m = 1; m <= M; ++m) {
    const double pairs = static_cast<double>(hi[m - 1] - lo[m - 1] + 1) * (hi[m] - lo[m] + 1);
    const double blocks = static_cast<double>(hi[m] - lo[m - 1] + 1);
    work += pairs * blocks * per_block * kModelMaxSplits;
  }
  if (work > 4e9) return MOCAP_EUNSUPPORTED;  // use a smaller window

  std::vector<int64_t> loads;
  std::unordered_map<int64_t, int64_t> memo;
  auto evaluate = [&](int64_t s, int64_t k) {
    const int64_t key = s * (U + 1) + k;
    const auto it = memo.find(key);
    if (it != memo.end()) return it->second;
    const int64_t length = s + k == U ? seq_len - g * s : g * k;
    const int64_t t = chunk_latency_best_ps(g * s, length, n_q_heads, n_kv_heads, head_dim,
                                            num_sms, loads);
    memo.emplace(key, t);
    return t;
  };
  // suffix states (m, s) for s in boundary m-1's window; row M+1 holds only
  // the terminal (M+1, U)
  struct State {
    bool set = false;
    int64_t t_max = 0, t_sum = 0, k = 0;
  };
  std::vector<std::vector<State>> st(static_cast<size_t>(M + 2));
  for (int64_t m = 1; m <= M; ++m)
    st[static_cast<size_t>(m)].resize(static_cast<size_t>(hi[m - 1] - lo[m - 1] + 1));
  State terminal;  // (M + 1, U): t_max = t_sum = 0
  terminal.set = true;
  auto suffix = [&](int64_t m, int64_t s) -> const State * {  // state (m, s), s in window m-1
    if (m == M + 1) return s == U ? &terminal : nullptr;
    if (s < lo[m - 1] || s > hi[m - 1]) return nullptr;
    const State &x = st[static_cast<size_t>(m)][static_cast<size_t>(s - lo[m - 1])];
    return x.set ? &x : nullptr;
  };
  const __int128 nm1 = num_stages - 1;
  for (int64_t m = M; m >= 1; --m) {
    for (int64_t s = hi[m - 1]; s >= lo[m - 1]; --s) {
      State &cur = st[static_cast<size_t>(m)][static_cast<size_t>(s - lo[m - 1])];
      for (int64_t k = 1; k <= U - s - (M - m); ++k) {
        if (s + k < lo[m] || s + k > hi[m]) continue;
        const State *nxt = suffix(m + 1, s + k);
        if (nxt == nullptr) continue;
        const int64_t t = evaluate(s, k);
        const int64_t tmax_new = std::max(nxt->t_max, t);
        const int64_t tsum_new = nxt->t_sum + t;
        if (!cur.set || static_cast<__int128>(tsum_new) + nm1 * tmax_new <
                            static_cast<__int128>(cur.t_sum) + nm1 * cur.t_max) {
          cur.t_max = tmax_new;
          cur.t_sum = tsum_new;
          cur.k = k;
          cur.set = true;
        }
      }
    }
  }
  const State *first = suffix(1, 0);
  if (first == nullptr) return MOCAP_EINVAL;
  boundaries[0] = 0;
  int64_t pos = 0;
  for (int64_t m = 1; m <= M; ++m) {
    pos += suffix(m, pos)->k;
    boundaries[m] = g * pos;
  }
  boundaries[M] = seq_len;
  return MOCAP_OK;
}
