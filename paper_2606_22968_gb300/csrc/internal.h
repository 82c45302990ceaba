// internal.h -- declarations shared by the library's translation units.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "mocap.h"

namespace mocap {

// Device address of the status word that bounded waits set on timeout, for
// the current device (resolved once per device).  nullptr on CUDA failure.
uint32_t *device_status_ptr();

inline bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace mocap
