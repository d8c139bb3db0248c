// rf_host.h -- host-side helpers shared by the C-ABI translation units.
#pragma once
#include <cuda_runtime.h>

#include <cstdint>

#include "rf.h"

namespace rf {

struct DeviceInfo {
  int device = -1;
  int sm_count = 0;
  int cc_major = 0;
  int cc_minor = 0;
  int max_smem_optin = 0;
  int l2_bytes = 0;
};

// Properties of the current device, cached per device ordinal (thread-safe).
rf_status current_device_info(DeviceInfo* out);

// Record a failure detail for rf_last_error() and return `st`.
rf_status fail(rf_status st, const char* what, cudaError_t err = cudaSuccess);

inline rf_status launch_status(const char* what) {
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? RF_OK : fail(RF_ERR_CUDA, what, e);
}

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace rf
