// Device helpers shared by the MPM kernels: status reporting, offsets
// lookup, the packed arg-max key and 16-byte vector arithmetic.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>

#include "launch.h"
#include "mpm.h"

namespace mpm {

// Programmatic dependent launch: every MPM kernel is launched so that its
// grid can be set up while the previous kernel in the stream drains, and
// starts by waiting for that kernel's completion and memory flush.
__device__ __forceinline__ void wait_for_previous_grid() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
// Lets the next kernel in the stream be scheduled onto SMs this grid frees;
// it still waits (wait_for_previous_grid) for this grid to finish.
__device__ __forceinline__ void allow_next_grid() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

template <typename... Params, typename... Args>
inline cudaError_t launch_dependent(void (*kernel)(Params...), dim3 grid, dim3 block, size_t smem,
                                    cudaStream_t stream, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// Blocks of `threads` threads of `kernel` that one SM holds at once
// (registers and static shared memory permitting), at most `cap`.  The
// bandwidth-bound kernels stride over rows with num_sms times this many
// blocks: one wave, so no block waits for another to retire before its
// share of the rows starts streaming (measured: a 2-wave grid of the same
// kernels made the vit_b step 2% slower).  Occupancy depends only on the
// kernel and the architecture, so callers keep the answer in a static.
template <typename... Params>
inline int resident_per_sm(void (*kernel)(Params...), int threads, int cap) {
  int n = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kernel, threads, 0) != cudaSuccess || n < 1) return cap;
  return n < cap ? n : cap;
}

// ---------------------------------------------------------------------------
// Device timeline (libmpm_trace.so only; see mpm_trace_read in mpm.h).  Each
// translation unit with traced kernels keeps its own table, which
// trace_copy_<unit> reads or resets from the host.
// ---------------------------------------------------------------------------
#ifdef MPM_TRACE
static __device__ unsigned long long g_trace[MPM_TRACE_KINDS][3];
__device__ __forceinline__ unsigned long long trace_now() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
struct TraceScope {
  int kind;
  __device__ explicit TraceScope(int k) : kind(k) {
    if (threadIdx.x == 0) atomicMin(&g_trace[kind][0], trace_now());
  }
  __device__ void waited() const {
    if (threadIdx.x == 0) atomicMin(&g_trace[kind][1], trace_now());
  }
  __device__ ~TraceScope() {
    if ((threadIdx.x & 31) == 0) atomicMax(&g_trace[kind][2], trace_now());
  }
};
// Reads (reset == false) or resets this translation unit's table.
static inline cudaError_t trace_table(unsigned long long* out, bool reset) {
  if (!reset) return cudaMemcpyFromSymbol(out, g_trace, sizeof(g_trace));
  unsigned long long v[MPM_TRACE_KINDS][3];
  for (int k = 0; k < MPM_TRACE_KINDS; ++k) {
    v[k][0] = v[k][1] = ~0ull;
    v[k][2] = 0ull;
  }
  return cudaMemcpyToSymbol(g_trace, v, sizeof(v));
}
#define MPM_TRACE_BEGIN(kind) const ::mpm::TraceScope mpm_trace_scope_(kind)
#define MPM_TRACE_WAITED() mpm_trace_scope_.waited()
#else
#define MPM_TRACE_BEGIN(kind) \
  do {                         \
  } while (0)
#define MPM_TRACE_WAITED() \
  do {                     \
  } while (0)
#endif

// First error wins; `st` may be null (not reported).
__device__ __forceinline__ void report(int32_t* st, int32_t code, int32_t detail) {
  if (st != nullptr && atomicCAS(st, 0, code) == 0) st[1] = detail;
}

// Index of the image that owns global row g: the largest b < batch with
// off[b] <= g.  `off` must be non-decreasing (sanitised offsets are).
__device__ __forceinline__ int find_image(const int64_t* __restrict__ off, int batch, int64_t g) {
  int lo = 0, hi = batch - 1;
  while (lo < hi) {
    int mid = (lo + hi + 1) >> 1;
    if (__ldg(off + mid) <= g) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// Same search over the work plan (prefix of work items per image).
__device__ __forceinline__ int find_item_image(const int64_t* __restrict__ plan, int batch, int64_t w) {
  int lo = 0, hi = batch - 1;
  while (lo < hi) {
    int mid = (lo + hi + 1) >> 1;
    if (__ldg(plan + mid) <= w) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// Work items (tiles) of the affinity pass for one image of n tokens.  Dense:
// every rows x cols tile.  Symmetric (cols == 2 * rows): row block I needs
// only the column tiles T holding a block J >= I, i.e. 2T + 1 >= I, so it
// has C - (I >> 1) of them; row blocks 2m and 2m+1 have 2(C - m) together.
// Upper square (rows == cols): the R (R + 1) / 2 tiles with J >= I.
__host__ __device__ __forceinline__ int64_t affinity_tiles(int64_t n, int rows, int cols, int mode) {
  const int64_t r = (n + rows - 1) / rows, c = (n + cols - 1) / cols;
  if (mode == AffinityTile::kDense) return r * c;
  if (mode == AffinityTile::kUpperSquare) return r * (r + 1) / 2;
  const int64_t q = r / 2;
  return 2 * q * c - q * (q - 1) + (r & 1) * (c - q);
}

// Work items of an image of n tokens: the tiles of every chunk (the whole
// image when t.chunk == 0; the last chunk may be shorter).
__host__ __device__ __forceinline__ int64_t image_items(int64_t n, const AffinityTile& t) {
  if (t.chunk <= 0 || n <= t.chunk) return affinity_tiles(n, t.rows, t.cols, t.mode);
  const int64_t full = n / t.chunk, last = n - full * t.chunk;
  return full * affinity_tiles(t.chunk, t.rows, t.cols, t.mode) +
         (last > 0 ? affinity_tiles(last, t.rows, t.cols, t.mode) : 0);
}

// The chunk of work item `local` of an image of n tokens: its first token,
// its length and the item's index within it.
struct ChunkItem {
  int64_t start, len, local;
};
__device__ __forceinline__ ChunkItem locate_chunk(int64_t local, int64_t n, const AffinityTile& t) {
  if (t.chunk <= 0 || n <= t.chunk) return {0, n, local};
  const int64_t per = affinity_tiles(t.chunk, t.rows, t.cols, t.mode);
  const int64_t full = n / t.chunk;
  const int64_t c = local / per;
  if (c < full) return {c * t.chunk, t.chunk, local - c * per};
  return {full * t.chunk, n - full * t.chunk, local - full * per};
}

// A total order on floats as unsigned integers (larger float -> larger key).
__device__ __forceinline__ uint32_t order_f32(float f) {
  uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float unorder_f32(uint32_t k) {
  uint32_t u = (k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k;
  return __uint_as_float(u);
}

// Packed arg-max key: the larger score wins, and on equal scores the lower
// column j wins, so a 64-bit atomicMax merges partial results in any order
// to the same answer.  -0 is folded into +0 so that equal scores compare
// equal.  Key 0 means "no candidate" (it is below every real key).
__device__ __forceinline__ unsigned long long make_key(float s, int32_t j) {
  if (s == 0.0f) s = 0.0f;
  return (static_cast<unsigned long long>(order_f32(s)) << 32) |
         static_cast<unsigned long long>(0xFFFFFFFFu - static_cast<uint32_t>(j));
}
__device__ __forceinline__ int32_t key_index(unsigned long long key) {
  if (key == 0ull) return -1;
  return static_cast<int32_t>(0xFFFFFFFFu - static_cast<uint32_t>(key & 0xFFFFFFFFull));
}
__device__ __forceinline__ float key_score(unsigned long long key) {
  return unorder_f32(static_cast<uint32_t>(key >> 32));
}

// ---------------------------------------------------------------------------
// 16-byte vectors: 8 bf16 or 4 fp32 lanes.
// ---------------------------------------------------------------------------
// x rounded to tf32 (10 explicit mantissa bits, round half to even); the
// tensor core's kind::tf32 products use exactly these bits.  Values whose
// rounding would overflow are truncated instead; infinities and NaNs pass.
__device__ __forceinline__ float round_tf32(float x) {
  const uint32_t u = __float_as_uint(x);
  if ((u & 0x7F800000u) == 0x7F800000u) return x;
  uint32_t r = (u + 0x0FFFu + ((u >> 13) & 1u)) & 0xFFFFE000u;
  if ((r & 0x7F800000u) == 0x7F800000u) r = u & 0xFFFFE000u;
  return __uint_as_float(r);
}

// Splits four fp32 values into tf32 high parts and the exact remainders
// x - hi (hi + lo = x; lo is again rounded to tf32 by the products).
__device__ __forceinline__ void split_tf32(uint4 v, uint4& hi, uint4& lo) {
  const float* f = reinterpret_cast<const float*>(&v);
  float* h = reinterpret_cast<float*>(&hi);
  float* l = reinterpret_cast<float*>(&lo);
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    h[k] = round_tf32(f[k]);
    l[k] = f[k] - h[k];
  }
}

__device__ __forceinline__ float sumsq16(uint4 v, bool bf16) {
  float s = 0.f;
  if (bf16) {
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      float2 f = __bfloat1622float2(h[k]);
      s = fmaf(f.x, f.x, s);
      s = fmaf(f.y, f.y, s);
    }
  } else {
    const float* f = reinterpret_cast<const float*>(&v);
#pragma unroll
    for (int k = 0; k < 4; ++k) s = fmaf(f[k], f[k], s);
  }
  return s;
}

// (a + b) / 2 lane by lane: fp32 add, exact halving, round to nearest even.
__device__ __forceinline__ uint4 avg16(uint4 a, uint4 b, bool bf16) {
  uint4 r;
  if (bf16) {
    const __nv_bfloat162* ha = reinterpret_cast<const __nv_bfloat162*>(&a);
    const __nv_bfloat162* hb = reinterpret_cast<const __nv_bfloat162*>(&b);
    __nv_bfloat162* hr = reinterpret_cast<__nv_bfloat162*>(&r);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      float2 fa = __bfloat1622float2(ha[k]);
      float2 fb = __bfloat1622float2(hb[k]);
      hr[k] = __floats2bfloat162_rn((fa.x + fb.x) * 0.5f, (fa.y + fb.y) * 0.5f);
    }
  } else {
    const float* fa = reinterpret_cast<const float*>(&a);
    const float* fb = reinterpret_cast<const float*>(&b);
    float* fr = reinterpret_cast<float*>(&r);
#pragma unroll
    for (int k = 0; k < 4; ++k) fr[k] = (fa[k] + fb[k]) * 0.5f;
  }
  return r;
}

__device__ __forceinline__ uint4 ld_stream(const uint4* p) { return __ldcs(p); }
__device__ __forceinline__ void st_stream(uint4* p, uint4 v) { __stcs(p, v); }

// ---------------------------------------------------------------------------
// Warp / block scans (inclusive), blockDim a multiple of 32, <= 1024.
// ---------------------------------------------------------------------------
template <typename T>
__device__ __forceinline__ T warp_incl_sum(T v) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    T o = __shfl_up_sync(0xFFFFFFFFu, v, d);
    if (lane >= d) v += o;
  }
  return v;
}

template <typename T>
__device__ __forceinline__ T warp_incl_max(T v) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    T o = __shfl_up_sync(0xFFFFFFFFu, v, d);
    if (lane >= d) v = v > o ? v : o;
  }
  return v;
}

// Inclusive block sum scan; returns the block total in *total.  `sh` needs
// 32 elements of shared memory.  Must be called by all threads.
template <typename T>
__device__ __forceinline__ T block_incl_sum(T v, T* sh, T* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nwarps = (blockDim.x + 31) >> 5;
  T x = warp_incl_sum(v);
  if (lane == 31) sh[warp] = x;
  __syncthreads();
  if (warp == 0) {
    T w = lane < nwarps ? sh[lane] : T(0);
    w = warp_incl_sum(w);
    sh[lane] = w;
  }
  __syncthreads();
  T base = warp > 0 ? sh[warp - 1] : T(0);
  *total = sh[nwarps - 1];
  __syncthreads();
  return x + base;
}

template <typename T>
__device__ __forceinline__ T block_incl_max(T v, T* sh, T* total, T lowest) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nwarps = (blockDim.x + 31) >> 5;
  T x = warp_incl_max(v);
  if (lane == 31) sh[warp] = x;
  __syncthreads();
  if (warp == 0) {
    T w = lane < nwarps ? sh[lane] : lowest;
    w = warp_incl_max(w);
    sh[lane] = w;
  }
  __syncthreads();
  T base = warp > 0 ? sh[warp - 1] : lowest;
  *total = sh[nwarps - 1];
  __syncthreads();
  return x > base ? x : base;
}

}  // namespace mpm
