// rf_capi.cpp -- status strings, version and the per-device property cache.
#include <cstdio>
#include <mutex>

#include "rf_host.h"

namespace rf {

namespace {
constexpr int kMaxDevices = 64;
DeviceInfo g_info[kMaxDevices];
std::mutex g_info_mu;
thread_local char g_last_error[256] = "";
}  // namespace

rf_status fail(rf_status st, const char* what, cudaError_t err) {
  if (err != cudaSuccess)
    std::snprintf(g_last_error, sizeof(g_last_error), "%s: %s (%s)", what, cudaGetErrorName(err),
                  cudaGetErrorString(err));
  else
    std::snprintf(g_last_error, sizeof(g_last_error), "%s", what);
  return st;
}

rf_status current_device_info(DeviceInfo* out) {
  int dev = 0;
  if (cudaError_t e = cudaGetDevice(&dev)) return fail(RF_ERR_CUDA, "cudaGetDevice", e);
  if (dev < 0 || dev >= kMaxDevices) return fail(RF_ERR_UNSUPPORTED, "device ordinal >= 64");
  std::lock_guard<std::mutex> lock(g_info_mu);
  DeviceInfo& d = g_info[dev];
  if (d.device != dev) {
    DeviceInfo n;
    n.device = dev;
    if (cudaDeviceGetAttribute(&n.sm_count, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&n.cc_major, cudaDevAttrComputeCapabilityMajor, dev) !=
            cudaSuccess ||
        cudaDeviceGetAttribute(&n.cc_minor, cudaDevAttrComputeCapabilityMinor, dev) !=
            cudaSuccess ||
        cudaDeviceGetAttribute(&n.max_smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) !=
            cudaSuccess ||
        cudaDeviceGetAttribute(&n.l2_bytes, cudaDevAttrL2CacheSize, dev) != cudaSuccess)
      return fail(RF_ERR_CUDA, "cudaDeviceGetAttribute", cudaGetLastError());
    d = n;
  }
  *out = d;
  return RF_OK;
}

}  // namespace rf

extern "C" const char* rf_status_str(int status) {
  switch (status) {
    case RF_OK: return "RF_OK";
    case RF_ERR_INVALID_ARG: return "RF_ERR_INVALID_ARG";
    case RF_ERR_UNSUPPORTED: return "RF_ERR_UNSUPPORTED";
    case RF_ERR_MISALIGNED: return "RF_ERR_MISALIGNED";
    case RF_ERR_CUDA: return "RF_ERR_CUDA";
    case RF_ERR_DEVICE_TIMEOUT: return "RF_ERR_DEVICE_TIMEOUT";
    default: return "RF_ERR_UNKNOWN";
  }
}

extern "C" int rf_version(void) { return 100; }

extern "C" const char* rf_last_error(void) { return rf::g_last_error; }
