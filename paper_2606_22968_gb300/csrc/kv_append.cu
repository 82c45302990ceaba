// kv_append.cu -- append one chunk's K and V rows to the contiguous KV cache.
//
// Sec. 2.2 / Sec. 3.1: every chunk's KV stays live for the chunks after it.
// The cache is [capacity, n_kv_heads, head_dim] bf16 row-major, so rows
// [offset, offset + len) of the cache are one contiguous byte range and the
// append is a straight 16-byte-vector copy of two ranges (K and V) in a single
// launch.  HBM-bound: 2 tensors x (read + write) x len x Hkv x d x 2 bytes.
#include <algorithm>

#include "internal.h"

namespace {

constexpr int kThreads = 256;
constexpr int kUnroll = 4;        // 16-byte vectors in flight per thread
constexpr int kCtasPerSm = 32;    // grid cap; the loop strides over the rest

__device__ __forceinline__ uint4 ld_stream(const uint4 *p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

// Vectors [0, n) come from k_src -> k_dst, vectors [n, 2n) from v_src -> v_dst.
__global__ void __launch_bounds__(kThreads) kv_append_kernel(const uint4 *__restrict__ k_src,
                                                             const uint4 *__restrict__ v_src,
                                                             uint4 *__restrict__ k_dst,
                                                             uint4 *__restrict__ v_dst,
                                                             int64_t n) {
  const int64_t total = 2 * n;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * kThreads * kUnroll;
  for (int64_t base = static_cast<int64_t>(blockIdx.x) * kThreads * kUnroll + threadIdx.x;
       base < total; base += stride) {
    uint4 v[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int64_t i = base + static_cast<int64_t>(u) * kThreads;
      if (i < total) v[u] = ld_stream(i < n ? k_src + i : v_src + (i - n));
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int64_t i = base + static_cast<int64_t>(u) * kThreads;
      if (i < total) {
        if (i < n) k_dst[i] = v[u];
        else v_dst[i - n] = v[u];
      }
    }
  }
}

// The same copy sized to run beside a running attention launch: one warp per
// CTA and at most 32 registers per thread (1024 registers per CTA), which is
// what an attention CTA (384 threads x 168 registers) leaves free on its SM,
// and no shared memory.  Each thread keeps four 16-byte loads in flight.
constexpr int kOverlapThreads = 32;
constexpr int kOverlapCtasPerSm = 4;

__device__ __forceinline__ void copy_stream(const uint4 *__restrict__ src, uint4 *__restrict__ dst,
                                            int64_t n) {
  const int64_t stride = static_cast<int64_t>(gridDim.x) * kOverlapThreads * kUnroll;
  for (int64_t base = static_cast<int64_t>(blockIdx.x) * kOverlapThreads * kUnroll + threadIdx.x;
       base < n; base += stride) {
    uint4 v[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u)
      if (base + u * kOverlapThreads < n) v[u] = ld_stream(src + base + u * kOverlapThreads);
#pragma unroll
    for (int u = 0; u < kUnroll; ++u)
      if (base + u * kOverlapThreads < n) dst[base + u * kOverlapThreads] = v[u];
  }
}

__global__ void __maxnreg__(32)
    kv_append_overlap_kernel(const uint4 *__restrict__ k_src, const uint4 *__restrict__ v_src,
                             uint4 *__restrict__ k_dst, uint4 *__restrict__ v_dst, int64_t n) {
  copy_stream(k_src, k_dst, n);
  copy_stream(v_src, v_dst, n);
}

// Argument checks shared by both entry points; on success *n is the number
// of 16-byte vectors per tensor and *dst_off the destination offset.
mocap_status check_append(const void *k_chunk, const void *v_chunk, void *k_cache, void *v_cache,
                          int64_t cache_capacity, int64_t offset, int64_t len, int32_t n_kv_heads,
                          int32_t head_dim, int64_t *n, int64_t *dst_off) {
  if (!k_chunk || !v_chunk || !k_cache || !v_cache) return MOCAP_EINVAL;
  if (!mocap::aligned16(k_chunk) || !mocap::aligned16(v_chunk) || !mocap::aligned16(k_cache) ||
      !mocap::aligned16(v_cache))
    return MOCAP_EINVAL;
  if (n_kv_heads < 1 || head_dim < 1 || offset < 0 || len < 0 || cache_capacity < 0)
    return MOCAP_EINVAL;
  const int64_t row_elems = static_cast<int64_t>(n_kv_heads) * head_dim;
  if (row_elems % 8 != 0) return MOCAP_EINVAL;  // rows must be whole 16-byte vectors
  if (offset > cache_capacity || len > cache_capacity - offset) return MOCAP_EINVAL;
  *n = len * row_elems / 8;
  *dst_off = offset * row_elems / 8;
  return MOCAP_OK;
}

}  // namespace

extern "C" mocap_status mocap_kv_append_overlap(const void *k_chunk, const void *v_chunk,
                                                void *k_cache, void *v_cache,
                                                int64_t cache_capacity, int64_t offset,
                                                int64_t len, int32_t n_kv_heads,
                                                int32_t head_dim, mocap_stream_t stream) {
  int64_t n = 0, dst_off = 0;
  const mocap_status st = check_append(k_chunk, v_chunk, k_cache, v_cache, cache_capacity,
                                       offset, len, n_kv_heads, head_dim, &n, &dst_off);
  if (st != MOCAP_OK || len == 0) return st;
  const int64_t want = (2 * n + kOverlapThreads * kUnroll - 1) / (kOverlapThreads * kUnroll);
  const int64_t cap = static_cast<int64_t>(mocap::device_sm_count()) * kOverlapCtasPerSm;
  const int blocks = static_cast<int>(std::max<int64_t>(1, std::min(want, cap)));
  kv_append_overlap_kernel<<<blocks, kOverlapThreads, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
      static_cast<const uint4 *>(k_chunk), static_cast<const uint4 *>(v_chunk),
      static_cast<uint4 *>(k_cache) + dst_off, static_cast<uint4 *>(v_cache) + dst_off, n);
  return cudaGetLastError() == cudaSuccess ? MOCAP_OK : MOCAP_ECUDA;
}

extern "C" mocap_status mocap_kv_append(const void *k_chunk, const void *v_chunk, void *k_cache,
                                        void *v_cache, int64_t cache_capacity, int64_t offset,
                                        int64_t len, int32_t n_kv_heads, int32_t head_dim,
                                        mocap_stream_t stream) {
  int64_t n = 0, dst_off = 0;  // 16-byte vectors per tensor, destination offset
  const mocap_status st = check_append(k_chunk, v_chunk, k_cache, v_cache, cache_capacity,
                                       offset, len, n_kv_heads, head_dim, &n, &dst_off);
  if (st != MOCAP_OK || len == 0) return st;
  const int64_t want = (2 * n + kThreads * kUnroll - 1) / (kThreads * kUnroll);
  const int64_t cap = static_cast<int64_t>(mocap::device_sm_count()) * kCtasPerSm;
  const int blocks = static_cast<int>(std::max<int64_t>(1, std::min(want, cap)));
  kv_append_kernel<<<blocks, kThreads, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
      static_cast<const uint4 *>(k_chunk), static_cast<const uint4 *>(v_chunk),
      static_cast<uint4 *>(k_cache) + dst_off, static_cast<uint4 *>(v_cache) + dst_off, n);
  return cudaGetLastError() == cudaSuccess ? MOCAP_OK : MOCAP_ECUDA;
}
