// attn_combine.cuh -- the split-KV combine kernel (device code) on sm_103a.
#pragma once

#include <cmath>
#include <cuda_bf16.h>

#include "attn_kernel.cuh"

namespace mocap {
namespace {

// Split-KV combine: the softmax over the union of disjoint key ranges weighs
// each range's normalised output by exp(LSE_k - LSE), LSE = ln sum_k exp(LSE_k).
// Block (row, g) merges heads g * kCombineHeadsPerBlock .. + kCombineHeadsPerBlock
// - 1 of one row.  Those heads' partial outputs are contiguous in every
// split (o_part [splits, len, Hq, D]), so one thread moves them into shared
// memory with one TMA bulk copy per split (no registers held while the
// bytes are in flight; several blocks per SM keep enough of them in flight
// to cover DRAM latency), while the block loads the range LSEs.  Then each
// warp merges kCombineHeadsPerBlock / 8 heads, lane = D/32 consecutive
// columns.  Like the attention launch before it, it does nothing once a
// bounded wait has expired (the status word is set), so the outputs keep
// their contents; its own wait for the copies is bounded the same way.
constexpr int kCombineThreads = 256;
constexpr int kCombineHeadsPerBlock = 32;

__device__ __forceinline__ void bulk_load_g2s(uint32_t dst, const void *src, uint32_t bytes,
                                              uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
      ::"r"(dst), "l"(src), "r"(bytes), "r"(bar)
      : "memory");
}

// Dynamic shared memory: splits x heads x D fp32 partials (1024-byte aligned
// base), then splits x heads fp32 LSEs, then one mbarrier.
template <int D>
__host__ __device__ constexpr size_t combine_smem_bytes(int splits) {
  return static_cast<size_t>(splits) * kCombineHeadsPerBlock * D * 4 +
         static_cast<size_t>(kMaxSplits) * kCombineHeadsPerBlock * 4 + 16 + 1024;
}

template <int D>
__global__ void __launch_bounds__(kCombineThreads) attn_combine_kernel(
    const float *__restrict__ o_part, const float *__restrict__ lse_part, int splits,
    int64_t len, int n_q_heads, __nv_bfloat16 *__restrict__ out, float *__restrict__ lse,
    int64_t lse_stride, uint32_t *status) {
  constexpr int kPer = D / 32;
  constexpr int kHB = kCombineHeadsPerBlock;
  extern __shared__ uint8_t smem_raw[];
  if (*reinterpret_cast<const volatile uint32_t *>(status) != 0u) return;
  const int64_t row = blockIdx.x;
  const int h0 = static_cast<int>(blockIdx.y) * kHB;
  if (row >= len || h0 >= n_q_heads) return;
  const int nh = min(kHB, n_q_heads - h0);
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  float *part = reinterpret_cast<float *>(smem_raw + (base - raw));
  float *lse_s = part + static_cast<size_t>(splits) * kHB * D;
  const uint32_t bar = base + static_cast<uint32_t>(
                                  (static_cast<size_t>(splits) * kHB * D + kMaxSplits * kHB) * 4);
  const uint32_t bytes = static_cast<uint32_t>(nh) * D * 4;  // per split, a multiple of 16
  if (threadIdx.x == 0) {
    mbar_init(bar, 1);
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    mbar_arrive_expect_tx(bar, bytes * static_cast<uint32_t>(splits));
    for (int k = 0; k < splits; ++k)
      bulk_load_g2s(base + static_cast<uint32_t>(k) * kHB * D * 4,
                    o_part + ((static_cast<int64_t>(k) * len + row) * n_q_heads + h0) * D, bytes,
                    bar);
  }
  for (int i = threadIdx.x; i < splits * nh; i += kCombineThreads) {
    const int k = i / nh, j = i % nh;
    lse_s[k * kHB + j] = __ldcs(lse_part + (static_cast<int64_t>(k) * n_q_heads + h0 + j) * len +
                                row);
  }
  // One thread waits (bounded) for the copies and tells the block, so the
  // decision is the same for every thread.
  __shared__ int copies_landed;
  if (threadIdx.x == 0) {
    copies_landed = mbar_wait(bar, 0, status) ? 1 : 0;
    // after an expired wait the copies may still be landing in this block's
    // shared memory: give them the drain limit before the block exits
    if (!copies_landed) mbar_wait(bar, 0, status, kDrainLimitNs, false);
  }
  __syncthreads();
  if (!copies_landed) return;
  const int warp = static_cast<int>(threadIdx.x >> 5);
  const int lane = static_cast<int>(threadIdx.x & 31);
  for (int j = warp; j < nh; j += kCombineThreads / 32) {
    const int h = h0 + j;
    float lk[kMaxSplits];
    float mx = -INFINITY;
#pragma unroll
    for (int k = 0; k < kMaxSplits; ++k) {
      if (k < splits) {
        lk[k] = lse_s[k * kHB + j];
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
        const float *src = part + (static_cast<size_t>(k) * kHB + j) * D + lane * kPer;
        if constexpr (kPer == 4) {
          const float4 v = *reinterpret_cast<const float4 *>(src);
          acc[0] += wk * v.x;
          acc[1] += wk * v.y;
          acc[2] += wk * v.z;
          acc[3] += wk * v.w;
        } else {
          const float2 v = *reinterpret_cast<const float2 *>(src);
          acc[0] += wk * v.x;
          acc[1] += wk * v.y;
        }
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
