// internal.h -- declarations shared by the library's translation units.
#pragma once

#include <cstdint>
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include "mocap.h"

namespace mocap {

// Device address of the status word that bounded waits set on timeout, for
// the current device (resolved once per device).  nullptr on CUDA failure.
uint32_t *device_status_ptr();

inline bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Number of SMs of the current device, read once per device; 152 (a
// GB300's count) if the device cannot be queried.  Grids are sized by it.
int device_sm_count();

// The driver's cuTensorMapEncodeTiled, looked up once; nullptr if the
// driver does not provide it.
PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder();

}  // namespace mocap
