// status.cu -- runtime state shared by the kernels' host code: the current
// context, the status word for bounded-wait timeouts (per context), the SM
// count (per device), the tensor-map encoder; status strings.
#include <atomic>
#include <mutex>

#include "internal.h"
#include "sm103_ptx.cuh"

namespace {
__device__ uint32_t g_device_status;  // 0 = OK, else the first error a kernel recorded

constexpr int kMaxDevices = 64;
std::vector<std::pair<uint64_t, uint32_t *>> g_status_ptr;  // per context ID
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

uint64_t current_context() {
  static PFN_cuCtxGetCurrent_v4000 get_current = nullptr;
  static PFN_cuCtxGetId_v12000 get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *ptr = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(ptr);
    ptr = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &ptr, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<PFN_cuCtxGetId_v12000>(ptr);
  });
  CUcontext c = nullptr;
  unsigned long long id = 0;
  if (get_current == nullptr || get_id == nullptr || get_current(&c) != CUDA_SUCCESS ||
      c == nullptr || get_id(c, &id) != CUDA_SUCCESS)
    return 0;
  return static_cast<uint64_t>(id);
}

uint32_t *device_status_ptr() {
  std::lock_guard<std::mutex> lock(g_status_mu);
  uint64_t c = current_context();
  if (c != 0)
    for (const auto &e : g_status_ptr)
      if (e.first == c) return e.second;
  // resolving the symbol binds the runtime's context to this thread if
  // none was current yet
  void *p = nullptr;
  if (cudaGetSymbolAddress(&p, g_device_status) != cudaSuccess) return nullptr;
  c = current_context();
  if (c == 0) return nullptr;
  for (const auto &e : g_status_ptr)
    if (e.first == c) return e.second;
  g_status_ptr.emplace_back(c, static_cast<uint32_t *>(p));
  return static_cast<uint32_t *>(p);
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
