// attn_combine.cuh -- the split-KV combine kernel (device code) on sm_103a.
#pragma once

#include <cmath>
#include <cuda_bf16.h>

#include "attn_kernel.cuh"

namespace mocap {
namespace {

// Split-KV combine: the softmax over the union of disjoint key ranges weighs
// each range's normalised output by exp(LSE_k - LSE), LSE = ln sum_k exp(LSE_k).
// A warp merges kCombineHeadsPerWarp (row, head) pairs; block (row, g) holds
// heads g * kCombineHeadsPerBlock .. + kCombineHeadsPerBlock - 1, so no index
// division is needed, and each lane owns D/32 consecutive columns.  All
// partial outputs of the warp's pairs are loaded before the range LSEs (they
// do not depend on the weights), so the DRAM round trips overlap.  Like the
// attention launch before it, it does nothing once a bounded wait has
// expired (the status word is set), so the outputs keep their contents.
constexpr int kCombineHeadsPerWarp = 2;
constexpr int kCombineHeadsPerBlock = 8 * kCombineHeadsPerWarp;

template <int D>
__global__ void __launch_bounds__(256) attn_combine_kernel(
    const float *__restrict__ o_part, const float *__restrict__ lse_part, int splits,
    int64_t len, int n_q_heads, __nv_bfloat16 *__restrict__ out, float *__restrict__ lse,
    int64_t lse_stride, const uint32_t *status) {
  constexpr int kPer = D / 32;
  constexpr int kH = kCombineHeadsPerWarp;
  if (*reinterpret_cast<const volatile uint32_t *>(status) != 0u) return;
  const int64_t row = blockIdx.x;
  const int h0 = static_cast<int>(blockIdx.y) * kCombineHeadsPerBlock +
                 static_cast<int>(threadIdx.x >> 5) * kH;
  if (row >= len || h0 >= n_q_heads) return;
  const int lane = threadIdx.x & 31;
  float o[kH][kMaxSplits][kPer];
#pragma unroll
  for (int j = 0; j < kH; ++j) {
#pragma unroll
    for (int k = 0; k < kMaxSplits; ++k) {
      if (k < splits && h0 + j < n_q_heads) {
        const float *src = o_part +
                           ((static_cast<int64_t>(k) * len + row) * n_q_heads + h0 + j) * D +
                           lane * kPer;
        if constexpr (kPer == 4) {
          const float4 v = __ldcs(reinterpret_cast<const float4 *>(src));
          o[j][k][0] = v.x;
          o[j][k][1] = v.y;
          o[j][k][2] = v.z;
          o[j][k][3] = v.w;
        } else {
          const float2 v = __ldcs(reinterpret_cast<const float2 *>(src));
          o[j][k][0] = v.x;
          o[j][k][1] = v.y;
        }
      }
    }
  }
#pragma unroll
  for (int j = 0; j < kH; ++j) {
    const int h = h0 + j;
    if (h >= n_q_heads) break;
    float lk[kMaxSplits];
    float mx = -INFINITY;
#pragma unroll
    for (int k = 0; k < kMaxSplits; ++k) {
      if (k < splits) {
        lk[k] = __ldcs(lse_part + (static_cast<int64_t>(k) * n_q_heads + h) * len + row);
        mx = fmaxf(mx, lk[k]);
      }
    }
    float wsum = 0.0f;
#pragma unroll
    for (int k = 0; k < kMaxSplits; ++k) {
      if (k < splits) {
        lk[k] = lk[k] > -INFINITY ? expf(lk[k] - mx) : 0.0f;
        wsum += lk[k];
      }
    }
    const float inv = 1.0f / wsum;
    float acc[kPer];
#pragma unroll
    for (int e = 0; e < kPer; ++e) acc[e] = 0.0f;
#pragma unroll
    for (int k = 0; k < kMaxSplits; ++k) {
      if (k < splits) {
        const float wk = lk[k] * inv;
#pragma unroll
        for (int e = 0; e < kPer; ++e) acc[e] += wk * o[j][k][e];
      }
    }
    __nv_bfloat16 *dst = out + (row * n_q_heads + h) * D + lane * kPer;
    if constexpr (kPer == 4) {
      const __nv_bfloat162 a = __floats2bfloat162_rn(acc[0], acc[1]);
      const __nv_bfloat162 b = __floats2bfloat162_rn(acc[2], acc[3]);
      uint2 pk;
      pk.x = *reinterpret_cast<const uint32_t *>(&a);
      pk.y = *reinterpret_cast<const uint32_t *>(&b);
      *reinterpret_cast<uint2 *>(dst) = pk;
    } else {
      *reinterpret_cast<__nv_bfloat162 *>(dst) = __floats2bfloat162_rn(acc[0], acc[1]);
    }
    if (lane == 0) lse[static_cast<int64_t>(h) * lse_stride + row] = mx + logf(wsum);
  }
}

}  // namespace
}  // namespace mocap
