// Padded batches for dense-attention consumers (Section 4, Analyses: the
// images of a batch are padded to the longest merged sequence and the
// padding is masked out).  pad_kernel writes [batch, L, dim] from the packed
// rows plus a key mask and the batch's N_b statistics; unpad_kernel is the
// inverse.  Both are bandwidth-bound copies: one warp per row, 16-byte
// vectors, grids sized from the SM count.
#include "mpm.h"
#include "common.cuh"
#include "launch.h"

namespace mpm {
namespace {

constexpr int kThreads = 256;
constexpr int kVecs = 4;  // 16-byte vectors per lane and pass

__device__ __forceinline__ int64_t clamp_off(int64_t v, int64_t rows) { return v < 0 ? 0 : (v > rows ? rows : v); }

// out[b, t] = tokens[off_b + t] for t < min(N_b, L), zero rows after;
// mask[b, t] = 1 for the copied rows.  Block 0 also reduces N_b to
// (min, max, total) into stats.  An image longer than L is cut and reported.
__global__ void __launch_bounds__(kThreads) pad_kernel(const uint8_t* __restrict__ tokens,
                                                       const int64_t* __restrict__ offsets, int batch,
                                                       int64_t rows, int64_t max_len, int row_bytes,
                                                       uint8_t* __restrict__ out, uint8_t* __restrict__ mask,
                                                       int64_t* __restrict__ stats, int32_t* status) {
  wait_for_previous_grid();
  if (blockIdx.x == 0 && stats != nullptr) {
    __shared__ int64_t sh_min[kThreads / 32], sh_max[kThreads / 32], sh_sum[kThreads / 32];
    int64_t mn = INT64_MAX, mx = 0, sm = 0;
    for (int b = threadIdx.x; b < batch; b += kThreads) {
      const int64_t n = clamp_off(offsets[b + 1], rows) - clamp_off(offsets[b], rows);
      const int64_t nn = n > 0 ? n : 0;
      mn = nn < mn ? nn : mn;
      mx = nn > mx ? nn : mx;
      sm += nn;
    }
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) {
      const int64_t a = __shfl_xor_sync(0xFFFFFFFFu, mn, d), c = __shfl_xor_sync(0xFFFFFFFFu, mx, d);
      mn = a < mn ? a : mn;
      mx = c > mx ? c : mx;
      sm += __shfl_xor_sync(0xFFFFFFFFu, sm, d);
    }
    const int w = threadIdx.x >> 5;
    if ((threadIdx.x & 31) == 0) {
      sh_min[w] = mn;
      sh_max[w] = mx;
      sh_sum[w] = sm;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      for (int i = 1; i < kThreads / 32; ++i) {
        mn = sh_min[i] < mn ? sh_min[i] : mn;
        mx = sh_max[i] > mx ? sh_max[i] : mx;
        sm += sh_sum[i];
      }
      stats[0] = batch > 0 ? mn : 0;
      stats[1] = mx;
      stats[2] = sm;
    }
  }
  const int lane = threadIdx.x & 31;
  const int64_t warp = (static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x) >> 5;
  const int64_t nwarps = (static_cast<int64_t>(gridDim.x) * kThreads) >> 5;
  const int64_t total = static_cast<int64_t>(batch) * max_len;
  const int nvec = row_bytes >> 4;
  for (int64_t q = warp; q < total; q += nwarps) {
    const int b = static_cast<int>(q / max_len);
    const int64_t t = q - static_cast<int64_t>(b) * max_len;
    const int64_t lo = clamp_off(__ldg(offsets + b), rows), hi = clamp_off(__ldg(offsets + b + 1), rows);
    const bool live = lo + t < hi;
    if (t == max_len - 1 && hi - lo > max_len && lane == 0) report(status, MPM_ERR_DEVICE_CHECK, b);
    if (mask != nullptr && lane == 0) mask[q] = live ? 1 : 0;
    const uint4* src = reinterpret_cast<const uint4*>(tokens + (live ? lo + t : 0) * row_bytes);
    uint4* dst = reinterpret_cast<uint4*>(out + q * row_bytes);
    for (int v0 = lane; v0 < nvec; v0 += 32 * kVecs) {
      uint4 val[kVecs];
#pragma unroll
      for (int u = 0; u < kVecs; ++u) {
        const int v = v0 + 32 * u;
        if (v < nvec) val[u] = live ? __ldg(src + v) : make_uint4(0, 0, 0, 0);
      }
#pragma unroll
      for (int u = 0; u < kVecs; ++u) {
        const int v = v0 + 32 * u;
        if (v < nvec) dst[v] = val[u];
      }
    }
  }
}

// out[off_b + t] = padded[b, t] for t < min(N_b, L): one warp per padded
// row, like pad_kernel, so that no row needs an image search.  Rows of an
// image longer than L are left untouched and reported.
__global__ void __launch_bounds__(kThreads) unpad_kernel(const uint8_t* __restrict__ padded, int batch,
                                                         int64_t max_len, const int64_t* __restrict__ offsets,
                                                         int64_t rows, int row_bytes, uint8_t* __restrict__ out,
                                                         int32_t* status) {
  wait_for_previous_grid();
  const int lane = threadIdx.x & 31;
  const int64_t warp = (static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x) >> 5;
  const int64_t nwarps = (static_cast<int64_t>(gridDim.x) * kThreads) >> 5;
  const int64_t total = static_cast<int64_t>(batch) * max_len;
  const int nvec = row_bytes >> 4;
  for (int64_t q = warp; q < total; q += nwarps) {
    const int b = static_cast<int>(q / max_len);
    const int64_t t = q - static_cast<int64_t>(b) * max_len;
    const int64_t lo = clamp_off(__ldg(offsets + b), rows), hi = clamp_off(__ldg(offsets + b + 1), rows);
    if (t == max_len - 1 && hi - lo > max_len && lane == 0) report(status, MPM_ERR_DEVICE_CHECK, b);
    if (lo + t >= hi) continue;  // padding
    const uint4* src = reinterpret_cast<const uint4*>(padded + q * row_bytes);
    uint4* dst = reinterpret_cast<uint4*>(out + (lo + t) * row_bytes);
    for (int v0 = lane; v0 < nvec; v0 += 32 * kVecs) {
      uint4 val[kVecs];
#pragma unroll
      for (int u = 0; u < kVecs; ++u) {
        const int v = v0 + 32 * u;
        if (v < nvec) val[u] = __ldg(src + v);
      }
#pragma unroll
      for (int u = 0; u < kVecs; ++u) {
        const int v = v0 + 32 * u;
        if (v < nvec) dst[v] = val[u];
      }
    }
  }
}

int pad_grid(int num_sms, int per_sm) { return (num_sms > 0 ? num_sms : 1) * per_sm; }

}  // namespace

cudaError_t launch_pad(const void* tokens, const int64_t* offsets, int batch, int64_t rows, int64_t max_len,
                       int dim, bool bf16, void* out, uint8_t* mask, int64_t* stats, int32_t* status, int num_sms,
                       cudaStream_t stream) {
  const int row_bytes = dim * (bf16 ? 2 : 4);
  static const int per_sm = resident_per_sm(pad_kernel, kThreads, 8);
  return launch_dependent(pad_kernel, dim3(pad_grid(num_sms, per_sm)), dim3(kThreads), 0, stream,
                          static_cast<const uint8_t*>(tokens), offsets, batch, rows, max_len, row_bytes,
                          static_cast<uint8_t*>(out), mask, stats, status);
}

cudaError_t launch_unpad(const void* padded, int batch, int64_t max_len, const int64_t* offsets, int64_t rows,
                         int dim, bool bf16, void* out, int32_t* status, int num_sms, cudaStream_t stream) {
  const int row_bytes = dim * (bf16 ? 2 : 4);
  static const int per_sm = resident_per_sm(unpad_kernel, kThreads, 8);
  return launch_dependent(unpad_kernel, dim3(pad_grid(num_sms, per_sm)), dim3(kThreads), 0, stream,
                          static_cast<const uint8_t*>(padded), batch, max_len, offsets, rows, row_bytes,
                          static_cast<uint8_t*>(out), status);
}

}  // namespace mpm
