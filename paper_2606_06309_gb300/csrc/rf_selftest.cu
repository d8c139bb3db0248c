// rf_selftest.cu -- exercises the device-side bounded wait on the GPU without faulting it.
//
// Every mbarrier wait of the attention kernel goes through mbar_wait(): bounded in time, and on
// expiry the CTA raises an abort flag, writes RF_ERR_DEVICE_TIMEOUT to the caller's status word,
// releases its tensor memory and returns.  This kernel runs the same wait on a barrier that no
// thread or copy ever arrives at, inside a CTA that holds TMEM, so the expiry path can be
// checked end to end: the status word is set, the launch completes, TMEM is free again.
#include <cuda_runtime.h>

#include "rf_host.h"
#include "rf_ptx.cuh"

namespace rf {
namespace {

__global__ void __launch_bounds__(128) selftest_wait_kernel(int32_t* status, uint64_t limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ uint32_t tmem_slot;
  __shared__ int abort_flag;
  const int warp = threadIdx.x >> 5;
  if (threadIdx.x == 0) {
    mbar_init(smem_u32(&bar), 1);  // one arrival expected; none ever comes
    abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc(smem_u32(&tmem_slot), 32);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const bool ok = mbar_wait(smem_u32(&bar), 0, &abort_flag, limit_ns);
  if (!ok && threadIdx.x == 0) atomicOr(status, RF_ERR_DEVICE_TIMEOUT);
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem_slot, 32);
  }
}

}  // namespace
}  // namespace rf

extern "C" rf_status rf_selftest_bounded_wait(int32_t* d_status, int limit_us, rf_stream_t stream) {
  if (!d_status) return RF_ERR_INVALID_ARG;
  if (limit_us < 100 || limit_us > 2000000) return RF_ERR_INVALID_ARG;
  rf::DeviceInfo di;
  if (rf_status st = rf::current_device_info(&di)) return st;
  if (di.cc_major != 10) return rf::fail(RF_ERR_UNSUPPORTED, "needs an sm_10x device");
  rf::selftest_wait_kernel<<<1, 128, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
      d_status, static_cast<uint64_t>(limit_us) * 1000ull);
  return rf::launch_status("selftest_wait_kernel launch");
}
