// mpm_merge_no_alloc: the merge entry point for callers that must not
// allocate device memory.
//
// mpm_merge takes its scratch space (row norms, arg-max keys, the list of
// representatives, per-image counts, the status word) from a workspace the
// caller allocates.  Some callers cannot do that: a plug-in running inside a
// host framework that has already reserved the whole device memory pool
// (and tracks every byte of it), or a latency-critical loop where
// cudaMalloc / cudaFree are banned because they can block and synchronise
// the device.  For them this file keeps the scratch in a fixed array in the
// library's own device memory and runs the ordinary merge on it.
//
// The array is a file-scope __device__ variable: every GPU that loads the
// library holds one copy of it until the process exits.  Host code cannot
// use its name as a device address, so the first call on each device looks
// the address up with cudaGetSymbolAddress (with that device current) and
// caches it.  That first call can load the module and must therefore come
// before any stream capture on that device.
//
// All calls on a device share the one array and it keeps whatever the last
// call left in it; calls that overlap on the GPU (two streams, two host
// threads) would race on it, so callers must serialise them.  What has to
// start at zero (the status block) is cleared at the start of every call;
// the merge kernels overwrite everything else before reading it.
#include <cuda_runtime.h>

#include <mutex>

#include "mpm.h"

namespace {

static __device__ __align__(256) unsigned char g_no_alloc_scratch[MPM_NO_ALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
constexpr size_t kStatusBlockBytes = 256;  // the status words lead the workspace
std::mutex g_setup_mutex;
void* g_scratch_ptr[kMaxDevices] = {};     // device address of the array, per device

// Device address of the scratch array on the current device (set up once).
mpm_status scratch_on_current_device(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return MPM_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return MPM_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  if (g_scratch_ptr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_no_alloc_scratch) != cudaSuccess || p == nullptr) return MPM_ERR_CUDA;
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
  return MPM_OK;
}

}  // namespace

extern "C" mpm_status mpm_merge_no_alloc(const void* tokens, const int64_t* offsets, int32_t batch,
                                         int64_t rows, int32_t dim, mpm_dtype dtype, void* out_tokens,
                                         int64_t* out_offsets, int32_t* out_map, void* stream) {
  const size_t need = mpm_merge_workspace_size(rows, batch, dim, dtype);
  if (need == 0) return MPM_ERR_INVALID_ARG;
  if (need > MPM_NO_ALLOC_SCRATCH_BYTES) return MPM_ERR_WORKSPACE;  // beyond the fixed scratch
  void* scratch = nullptr;
  const mpm_status st = scratch_on_current_device(&scratch);
  if (st != MPM_OK) return st;
  if (cudaMemsetAsync(scratch, 0, kStatusBlockBytes, static_cast<cudaStream_t>(stream)) != cudaSuccess)
    return MPM_ERR_CUDA;
  return mpm_merge(tokens, offsets, batch, rows, dim, dtype, out_tokens, out_offsets, out_map, scratch,
                   MPM_NO_ALLOC_SCRATCH_BYTES, stream);
}
