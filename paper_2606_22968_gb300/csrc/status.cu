// status.cu -- per-device runtime state shared by the kernels' host code:
// the status word for bounded-wait timeouts, the SM count, the tensor-map
// encoder; status strings.
#include <atomic>
#include <mutex>

#include "internal.h"
#include "sm103_ptx.cuh"

namespace {
__device__ uint32_t g_device_status;  // 0 = OK, MOCAP_ETIMEOUT after an expired wait

constexpr int kMaxDevices = 64;
uint32_t *g_status_ptr[kMaxDevices] = {};
std::mutex g_status_mu;
}  // namespace

namespace mocap {

int device_sm_count() {
  // atomics: threads may race to fill an entry (with the same value)
  static std::atomic<int> cached[kMaxDevices] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return 152;
  int n = cached[dev].load(std::memory_order_relaxed);
  if (n == 0) {
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
      n = 152;
    cached[dev].store(n, std::memory_order_relaxed);
  }
  return n;
}

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *ptr = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  });
  return fn;
}

uint32_t *device_status_ptr() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lock(g_status_mu);
  if (g_status_ptr[dev] == nullptr) {
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_device_status) != cudaSuccess) return nullptr;
    g_status_ptr[dev] = static_cast<uint32_t *>(p);
  }
  return g_status_ptr[dev];
}

}  // namespace mocap

extern "C" mocap_status mocap_last_device_status(mocap_stream_t stream) {
  uint32_t *p = mocap::device_status_ptr();
  if (p == nullptr) return MOCAP_ECUDA;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  uint32_t value = 0;
  if (cudaMemcpyAsync(&value, p, sizeof(value), cudaMemcpyDeviceToHost, s) != cudaSuccess)
    return MOCAP_ECUDA;
  if (cudaMemsetAsync(p, 0, sizeof(uint32_t), s) != cudaSuccess) return MOCAP_ECUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return MOCAP_ECUDA;
  return value == 0 ? MOCAP_OK : static_cast<mocap_status>(value);
}

extern "C" const char *mocap_status_string(mocap_status status) {
  switch (status) {
    case MOCAP_OK: return "MOCAP_OK";
    case MOCAP_EINVAL: return "MOCAP_EINVAL: invalid argument";
    case MOCAP_ECUDA: return "MOCAP_ECUDA: CUDA call failed";
    case MOCAP_EUNSUPPORTED: return "MOCAP_EUNSUPPORTED: unsupported shape";
    case MOCAP_ETIMEOUT: return "MOCAP_ETIMEOUT: device wait expired";
  }
  return "MOCAP_UNKNOWN";
}

namespace {
// One thread waits, through the same bounded wait the attention kernel uses,
// on an mbarrier that nothing ever arrives on.
__global__ void bounded_wait_selftest_kernel(uint32_t *status, uint64_t limit_ns) {
  __shared__ alignas(8) uint64_t bar;
  if (threadIdx.x == 0) {
    const uint32_t b = mocap::smem_u32(&bar);
    mocap::mbar_init(b, 1);
    mocap::fence_mbar_init();
    mocap::mbar_wait(b, 0, status, limit_ns, false);
  }
}
}  // namespace

extern "C" mocap_status mocap_selftest_bounded_wait(uint32_t limit_us, mocap_stream_t stream) {
  if (limit_us == 0 || limit_us > 1000000u) return MOCAP_EINVAL;
  uint32_t *status = mocap::device_status_ptr();
  if (status == nullptr) return MOCAP_ECUDA;
  bounded_wait_selftest_kernel<<<1, 32, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
      status, static_cast<uint64_t>(limit_us) * 1000u);
  return cudaGetLastError() == cudaSuccess ? MOCAP_OK : MOCAP_ECUDA;
}
