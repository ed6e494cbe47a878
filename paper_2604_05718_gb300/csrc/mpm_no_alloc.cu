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
// use its name as a device address.  The set-up looks the address up with
// cudaGetSymbolAddress, with the device current, once per device context:
// the first call on a device does it (it can load the module, so that first
// call must come before any stream capture on the device), and it is done
// again only if the device's context changed since (a cudaDeviceReset
// between calls), so a stale address is never used.
//
// All calls on a device share the one array and it keeps whatever the last
// call left in it; calls that overlap on the GPU (two streams, two host
// threads) would race on it, so callers must serialise them.  What has to
// start at zero (the status block) is cleared at the start of every call;
// the merge kernels overwrite everything else before reading it.
#include <cuda.h>
#include <cuda_runtime.h>

#include <mutex>

#include "mpm.h"

namespace {

static __device__ __align__(256) unsigned char g_no_alloc_scratch[MPM_NO_ALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
constexpr size_t kStatusBlockBytes = 256;  // the status words lead the workspace
std::mutex g_setup_mutex;
void* g_scratch_ptr[kMaxDevices] = {};             // device address of the array, per device
unsigned long long g_scratch_ctx[kMaxDevices] = {};  // ID of the context that address belongs to

// Unique ID of the current context (cuCtxGetId, through the runtime's
// driver entry points so that the library needs no -lcuda); 0 when no
// context is current or the driver cannot say.
unsigned long long current_context_id() {
  using GetCurrent = CUresult (*)(CUcontext*);
  using GetId = CUresult (*)(CUcontext, unsigned long long*);
  static GetCurrent get_current = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      return static_cast<GetCurrent>(nullptr);
    return reinterpret_cast<GetCurrent>(p);
  }();
  static GetId get_id = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      return static_cast<GetId>(nullptr);
    return reinterpret_cast<GetId>(p);
  }();
  if (get_current == nullptr || get_id == nullptr) return 0;
  CUcontext ctx = nullptr;
  unsigned long long id = 0;
  if (get_current(&ctx) != CUDA_SUCCESS || ctx == nullptr) return 0;
  if (get_id(ctx, &id) != CUDA_SUCCESS) return 0;
  return id;
}

// Device address of the scratch array on the current device.  Looked up
// once per device context; without a context ID it is looked up each call.
mpm_status scratch_on_current_device(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return MPM_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return MPM_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  const unsigned long long ctx = current_context_id();
  if (g_scratch_ptr[dev] == nullptr || ctx == 0 || ctx != g_scratch_ctx[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_no_alloc_scratch) != cudaSuccess || p == nullptr) return MPM_ERR_CUDA;
    g_scratch_ptr[dev] = p;
    g_scratch_ctx[dev] = current_context_id();  // the lookup made a context current if none was
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

extern "C" mpm_status mpm_no_alloc_get_device_status(int32_t* host_code, void* stream) {
  if (host_code == nullptr) return MPM_ERR_INVALID_ARG;
  void* scratch = nullptr;
  const mpm_status st = scratch_on_current_device(&scratch);
  if (st != MPM_OK) return st;
  return mpm_get_device_status(scratch, host_code, stream);
}
