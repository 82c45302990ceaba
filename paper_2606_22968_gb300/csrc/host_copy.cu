// host_copy.cu -- copies between page-locked host memory and device memory
// done by the SMs, through the host pages' device mapping.
//
// A prompt's Q/K/V reach the GPU from host memory before its chunks run
// (Sec. 2.2: the chunks of a prefill-only request stream through the
// pipeline).  On the GB300 machines this library runs on, copy-engine uploads
// from page-locked memory right after heavy device work ran at about
// 20 GB/s (15-28 ms for 475 MB) in 12 of 16 trials, while SM loads of the
// same pages ran at the link's 200 GB/s in 15 of 16; returns (380 MB back)
// behaved the same way, 14 of 16 slow on the copy engines against 2 of 16
// with SM stores.  So the pipeline moves a prompt's data with these kernels:
// all SMs while nothing else runs, or one warp per SM (32 registers, no
// shared memory: what an attention CTA leaves free) beside the attention
// launches.  Each launch copies up to MOCAP_COPY_MAX_ITEMS ranges (for
// example a chunk's Q, K and V rows).
#include <algorithm>

#include "internal.h"

namespace {

constexpr int kThreads = 256;
constexpr int kUnroll = 4;        // 16-byte vectors in flight per thread
constexpr int kCtasPerSm = 8;
constexpr int kBesideThreads = 32;

struct CopySeg {
  const uint4 *src;
  uint4 *dst;
  int64_t n;  // 16-byte vectors
};

struct CopyParams {
  CopySeg seg[MOCAP_COPY_MAX_ITEMS];
  int32_t n_seg;
};

// blockIdx.y = segment; the segment's CTAs stride over its vectors.
template <int THREADS>
__device__ __forceinline__ void copy_segment(const CopySeg &s) {
  const int64_t stride = static_cast<int64_t>(gridDim.x) * THREADS * kUnroll;
  for (int64_t base = static_cast<int64_t>(blockIdx.x) * THREADS * kUnroll + threadIdx.x;
       base < s.n; base += stride) {
    uint4 v[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u)
      if (base + u * THREADS < s.n) v[u] = s.src[base + u * THREADS];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u)
      if (base + u * THREADS < s.n) s.dst[base + u * THREADS] = v[u];
  }
}

__global__ void __launch_bounds__(kThreads) host_copy_kernel(const __grid_constant__ CopyParams p) {
  copy_segment<kThreads>(p.seg[blockIdx.y]);
}

__global__ void __maxnreg__(32) host_copy_beside_kernel(const __grid_constant__ CopyParams p) {
  copy_segment<kBesideThreads>(p.seg[blockIdx.y]);
}

// Page-locked host memory mapped at the same address on the device (unified
// addressing), checked at both ends of the range.
bool host_range_ok(const void *src, int64_t bytes) {
  for (const char *p : {static_cast<const char *>(src), static_cast<const char *>(src) + bytes - 1}) {
    cudaPointerAttributes a{};
    if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
      cudaGetLastError();
      return false;
    }
    if (a.type != cudaMemoryTypeHost || a.devicePointer != p) return false;
  }
  return true;
}

// Device (or managed) memory at both ends of the range.
bool device_range_ok(const void *dst, int64_t bytes) {
  for (const char *p : {static_cast<const char *>(dst), static_cast<const char *>(dst) + bytes - 1}) {
    cudaPointerAttributes a{};
    if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
      cudaGetLastError();
      return false;
    }
    if (a.type != cudaMemoryTypeDevice && a.type != cudaMemoryTypeManaged) return false;
  }
  return true;
}

mocap_status copy_items(const mocap_copy_item *items, int32_t n_items, int32_t beside_kernels,
                        mocap_stream_t stream, bool to_host) {
  if (n_items < 0 || n_items > MOCAP_COPY_MAX_ITEMS) return MOCAP_EINVAL;
  if (n_items > 0 && items == nullptr) return MOCAP_EINVAL;
  CopyParams prm{};
  int64_t most = 0;
  for (int i = 0; i < n_items; ++i) {
    const mocap_copy_item &it = items[i];
    if (it.bytes < 0 || it.bytes % 16 != 0) return MOCAP_EINVAL;
    if (it.bytes == 0) continue;
    if (!it.dst || !it.src || !mocap::aligned16(it.dst) || !mocap::aligned16(it.src))
      return MOCAP_EINVAL;
    const bool ok = to_host ? device_range_ok(it.src, it.bytes) && host_range_ok(it.dst, it.bytes)
                            : host_range_ok(it.src, it.bytes) && device_range_ok(it.dst, it.bytes);
    if (!ok) return MOCAP_EINVAL;
    CopySeg &s = prm.seg[prm.n_seg++];
    s.src = static_cast<const uint4 *>(it.src);
    s.dst = static_cast<uint4 *>(it.dst);
    s.n = it.bytes / 16;
    most = std::max(most, s.n);
  }
  if (prm.n_seg == 0) return MOCAP_OK;
  const int sms = mocap::device_sm_count();
  const cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (beside_kernels) {
    // one warp per SM in all, shared among the segments
    const int64_t want = (most + kBesideThreads * kUnroll - 1) / (kBesideThreads * kUnroll);
    const int per = static_cast<int>(std::max<int64_t>(1, std::min<int64_t>(want, sms / prm.n_seg)));
    host_copy_beside_kernel<<<dim3(per, prm.n_seg), kBesideThreads, 0, st>>>(prm);
  } else {
    const int64_t want = (most + kThreads * kUnroll - 1) / (kThreads * kUnroll);
    const int per = static_cast<int>(
        std::max<int64_t>(1, std::min<int64_t>(want, (int64_t)sms * kCtasPerSm / prm.n_seg)));
    host_copy_kernel<<<dim3(per, prm.n_seg), kThreads, 0, st>>>(prm);
  }
  return cudaGetLastError() == cudaSuccess ? MOCAP_OK : MOCAP_ECUDA;
}

}  // namespace

extern "C" mocap_status mocap_copy_from_host(const mocap_copy_item *items, int32_t n_items,
                                             int32_t beside_kernels, mocap_stream_t stream) {
  return copy_items(items, n_items, beside_kernels, stream, false);
}

extern "C" mocap_status mocap_copy_to_host(const mocap_copy_item *items, int32_t n_items,
                                           int32_t beside_kernels, mocap_stream_t stream) {
  return copy_items(items, n_items, beside_kernels, stream, true);
}
