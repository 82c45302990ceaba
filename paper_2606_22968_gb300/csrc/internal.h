// internal.h -- declarations shared by the library's translation units.
#pragma once

#include <algorithm>
#include <cstdint>
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <vector>

#include "mocap.h"

namespace mocap {

// The unique ID (cuCtxGetId: never reused within the process, unlike a
// context handle) of the CUDA context current on the calling thread: the
// device's primary context (the runtime API's) unless the caller made
// another one current through the driver API; 0 before the runtime has
// bound one to the thread.  State that belongs to a context (symbol
// addresses, kernel attributes) is cached under it.
uint64_t current_context();

// Contexts in which a one-time step (setting a kernel's attributes) is done.
// Not synchronised: each owner calls it under its own launch mutex.
class ContextOnce {
 public:
  bool done(uint64_t c) const { return std::find(ctx_.begin(), ctx_.end(), c) != ctx_.end(); }
  void mark(uint64_t c) {
    if (!done(c)) ctx_.push_back(c);
  }

 private:
  std::vector<uint64_t> ctx_;
};

// Device address of the status word that bounded waits set on timeout, in
// the current context (resolved once per context).  nullptr on CUDA
// failure.  Binds the runtime's context to the thread if none is current.
uint32_t *device_status_ptr();

inline bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Number of SMs of the current device, read once per device; 152 (a
// GB300's count) if the device cannot be queried.  Grids are sized by it.
int device_sm_count();

// The driver's cuTensorMapEncodeTiled, looked up once; nullptr if the
// driver does not provide it.
PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder();

}  // namespace mocap
