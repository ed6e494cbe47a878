// mpm_selftest_wait_timeout: exercises the bounded wait and the device
// status report that every MPM kernel relies on, with a barrier that no
// thread ever completes (see include/mpm.h).
#include <cuda_runtime.h>
#include <stdint.h>

#include "mpm.h"
#include "common.cuh"
#include "ptx.cuh"

namespace mpm {
namespace {

constexpr int kSelftestThreads = 64;
constexpr int32_t kSelftestDetail = 99;

__global__ void __launch_bounds__(kSelftestThreads) wait_timeout_kernel(int32_t* status, uint64_t limit_ns) {
  __shared__ uint64_t never;  // expects one arrival that nobody makes
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    ptx::mbar_init(&never, 1);
    abort_flag = 0;
    ptx::fence_barrier_init();
  }
  __syncthreads();
  if (!ptx::mbar_wait(&never, 0, &abort_flag, limit_ns)) report(status, MPM_ERR_DEVICE_TIMEOUT, kSelftestDetail);
}

}  // namespace
}  // namespace mpm

extern "C" mpm_status mpm_selftest_wait_timeout(int32_t* device_status, uint32_t limit_us, void* stream) {
  if (device_status == nullptr || limit_us == 0 || limit_us > 10000000u) return MPM_ERR_INVALID_ARG;
  mpm::wait_timeout_kernel<<<1, mpm::kSelftestThreads, 0, static_cast<cudaStream_t>(stream)>>>(
      device_status, static_cast<uint64_t>(limit_us) * 1000ull);
  return cudaGetLastError() == cudaSuccess ? MPM_OK : MPM_ERR_CUDA;
}
