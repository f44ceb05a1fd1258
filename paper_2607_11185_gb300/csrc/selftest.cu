// selftest.cu - a check, runnable on any deployment, that the library's bounded
// device waits give up and report instead of hanging.
//
// Every pipeline wait in the attention kernels is an mbarrier wait bounded by a
// cycle limit: when the limit runs out the kernel records VCS_ERR_DEVICE_TIMEOUT
// in the call's status word.  vcs_selftest_bounded_wait runs that wait primitive
// alone, on a barrier that nothing ever arrives on, with a caller-chosen limit,
// so the host can read the status it leaves.  It does not exercise how a whole
// attention CTA gives up (its warpgroups' joint decisions, TMEM release).
#include <cstdint>

#include "internal.h"
#include "sm100.cuh"

namespace vcs {
namespace {

using namespace dev;

__global__ void __launch_bounds__(1) selftest_wait_kernel(int32_t* status, long long limit_cycles) {
  __shared__ uint64_t bar;
  mbar_init(&bar, 1);
  fence_mbar_init();
  // phase 0 of `bar` completes only when its one expected arrival lands, and none is made
  if (mbar_try_wait(&bar, 0)) return;
  const long long t0 = clock64();
  while (!mbar_try_wait(&bar, 0)) {
    if (clock64() - t0 > limit_cycles) {
      set_status(status, VCS_ERR_DEVICE_TIMEOUT);
      return;
    }
  }
}

}  // namespace
}  // namespace vcs

extern "C" vcs_status vcs_selftest_bounded_wait(int32_t* dev_status, int64_t limit_cycles, void* stream) {
  vcs::ApiRange nvtx_range("vcs_selftest_bounded_wait");
  if (dev_status == nullptr || (reinterpret_cast<uintptr_t>(dev_status) & 3u) != 0) return VCS_ERR_INVALID_ARG;
  if (limit_cycles <= 0 || limit_cycles > vcs::dev::kWaitLimitCycles) return VCS_ERR_INVALID_ARG;
  vcs::selftest_wait_kernel<<<1, 1, 0, static_cast<cudaStream_t>(stream)>>>(dev_status,
                                                                           static_cast<long long>(limit_cycles));
  return cudaGetLastError() == cudaSuccess ? VCS_OK : VCS_ERR_CUDA;
}
