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
