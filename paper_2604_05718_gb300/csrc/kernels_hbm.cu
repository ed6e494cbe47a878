// Bandwidth-bound MPM kernels: row norms (Eq. 1), the mutual check and
// left-to-right representative scan (Algorithm 1 steps 4-6), the pair
// average with compaction (Eq. 2), map composition (Eq. 3) and the gather
// reconstruction (Eq. 4).  All token traffic moves in 16-byte vectors, one
// warp per row; grids are sized from the SM count and loop over rows.
#include <math.h>

#include "mpm.h"
#include "common.cuh"

namespace mpm {
namespace {

constexpr int kThreads = 256;
constexpr int kPrepRows = 2;   // rows per warp iteration in prep_kernel
constexpr int kPrepVecs = 3;   // 16-byte vectors per lane and row per pass (one pass at D = 768 bf16)

__device__ __forceinline__ int64_t clamp64(int64_t v, int64_t lo, int64_t hi) {
  return v < lo ? lo : (v > hi ? hi : v);
}

// Finds the image of row p, reusing the previous answer when p is still in
// the same image (rows are visited in increasing order by each warp).
struct ImageCursor {
  int b = 0;
  int64_t lo = 1, hi = 0;  // empty: forces the first search
  __device__ __forceinline__ void locate(const int64_t* off, int batch, int64_t p) {
    if (p >= lo && p < hi) return;
    b = find_image(off, batch, p);
    lo = __ldg(off + b);
    hi = __ldg(off + b + 1);
  }
};

// ---------------------------------------------------------------------------
// Prep: status reset, offsets sanitisation + work plan (block 0), inverse
// row norms and key reset (all blocks).
// ---------------------------------------------------------------------------
// SPLIT: also write the tf32 high / low parts of fp32 tokens (ws.split_hi /
// split_lo) for the three-product tensor-core path.
template <bool SPLIT>
__global__ void __launch_bounds__(kThreads) prep_kernel(const uint8_t* __restrict__ tokens,
                                                        const int64_t* __restrict__ offsets,
                                                        int batch, int64_t rows, int row_bytes,
                                                        bool bf16, AffinityTile tile,
                                                        Workspace ws) {
  MPM_TRACE_BEGIN(MPM_TRACE_PREP);
  wait_for_previous_grid();
  MPM_TRACE_WAITED();
  // The affinity kernel that follows only sets up barriers and tensor memory
  // before it waits for this grid, so it may take SMs as this grid drains.
  // (The other kernels do not trigger early: blocks of a dependent grid
  // parked on SMs were measured to slow the bandwidth-bound kernels.)
  allow_next_grid();
  if (blockIdx.x == 0) {
    __shared__ int64_t sh[32];
    __shared__ int bad;
    if (threadIdx.x == 0) {
      ws.status[0] = 0;
      ws.status[1] = 0;
      ws.status[2] = 0;
      bad = -1;
    }
    __syncthreads();
    // soff[b] = min(rows, max_{b' <= b} max(off[b'], 0)): non-decreasing and
    // in range whatever the caller passed; violations are reported.
    int64_t carry = 0;
    for (int base = 0; base <= batch; base += kThreads) {
      const int idx = base + threadIdx.x;
      int64_t raw = 0, prev = 0;
      if (idx <= batch) {
        raw = offsets[idx];
        prev = idx > 0 ? offsets[idx - 1] : 0;
        if ((idx == 0 && raw != 0) || raw < prev || raw > rows) atomicCAS(&bad, -1, idx);
      }
      int64_t v = idx <= batch ? clamp64(raw, 0, rows) : 0;
      int64_t total;
      int64_t m = block_incl_max<int64_t>(v, sh, &total, 0);
      m = m > carry ? m : carry;
      if (idx <= batch) ws.soff[idx] = m;
      carry = total > carry ? total : carry;
    }
    __syncthreads();
    if (threadIdx.x == 0 && bad >= 0) report(ws.status, MPM_ERR_DEVICE_CHECK, bad);
    // plan[b] = number of affinity tiles of the images before b.
    __threadfence_block();
    int64_t acc = 0;
    for (int base = 0; base <= batch; base += kThreads) {
      const int idx = base + threadIdx.x;
      int64_t items = 0;
      if (idx < batch) {
        const int64_t n = ws.soff[idx + 1] - ws.soff[idx];
        items = image_items(n, tile);
      }
      int64_t total;
      const int64_t incl = block_incl_sum<int64_t>(items, sh, &total);
      if (idx <= batch) ws.plan[idx] = acc + incl - items;
      acc += total;
    }
  }

  // Inverse norms of every used row, and the arg-max keys reset to "none".
  // Each warp takes kPrepRows consecutive rows at a time and issues all of
  // their 16-byte loads before reducing, to keep enough bytes in flight.
  // The sweep runs from the last row to the first: the affinity kernel
  // starts with the first images, and those are then the ones this sweep
  // left in L2 (measured: 3.5 instead of 3.8 us per tile on vit_b).
  const int64_t used = clamp64(offsets[batch], 0, rows);
  auto row_of = [used](int64_t i) { return used - 1 - i; };
  const int lane = threadIdx.x & 31;
  const int64_t warp = (static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x) >> 5;
  const int64_t nwarps = (static_cast<int64_t>(gridDim.x) * kThreads) >> 5;
  const int nvec = row_bytes >> 4;
  for (int64_t g0 = warp * kPrepRows; g0 < used; g0 += nwarps * kPrepRows) {
    float s[kPrepRows];
#pragma unroll
    for (int r = 0; r < kPrepRows; ++r) s[r] = 0.f;
    for (int v0 = lane; v0 < nvec; v0 += 32 * kPrepVecs) {
      uint4 buf[kPrepRows][kPrepVecs];
#pragma unroll
      for (int r = 0; r < kPrepRows; ++r) {
        const uint4* src = reinterpret_cast<const uint4*>(tokens + row_of(g0 + r) * row_bytes);
#pragma unroll
        for (int u = 0; u < kPrepVecs; ++u) {
          const int v = v0 + 32 * u;
          buf[r][u] = (g0 + r < used && v < nvec) ? __ldg(src + v) : make_uint4(0, 0, 0, 0);
        }
      }
#pragma unroll
      for (int r = 0; r < kPrepRows; ++r)
#pragma unroll
        for (int u = 0; u < kPrepVecs; ++u) s[r] += sumsq16(buf[r][u], bf16);
      if constexpr (SPLIT) {
#pragma unroll
        for (int r = 0; r < kPrepRows; ++r)
#pragma unroll
          for (int u = 0; u < kPrepVecs; ++u) {
            const int v = v0 + 32 * u;
            if (g0 + r < used && v < nvec) {
              uint4 hi, lo;
              split_tf32(buf[r][u], hi, lo);
              const int64_t at = row_of(g0 + r) * (row_bytes >> 4) + v;
              reinterpret_cast<uint4*>(ws.split_hi)[at] = hi;
              reinterpret_cast<uint4*>(ws.split_lo)[at] = lo;
            }
          }
      }
    }
#pragma unroll
    for (int r = 0; r < kPrepRows; ++r) {
#pragma unroll
      for (int d = 16; d > 0; d >>= 1) s[r] += __shfl_xor_sync(0xFFFFFFFFu, s[r], d);
    }
    if (lane < kPrepRows && g0 + lane < used) {
      float mine = s[0];
#pragma unroll
      for (int r = 1; r < kPrepRows; ++r) mine = lane == r ? s[r] : mine;
      ws.inv_norm[row_of(g0 + lane)] = 1.0f / fmaxf(sqrtf(mine), 1e-12f);
      ws.keys[row_of(g0 + lane)] = 0ull;
    }
  }
}

// ---------------------------------------------------------------------------
// Mutual check + left-to-right representative scan, one block per image.
// The last block to finish turns the per-image counts into out_offsets.
// ---------------------------------------------------------------------------
constexpr int kScanThreads = 1024;

__global__ void __launch_bounds__(kScanThreads) mutual_compact_kernel(int batch, int64_t chunk, Workspace ws,
                                                                      int32_t* __restrict__ out_map,
                                                                      int64_t* __restrict__ out_offsets) {
  MPM_TRACE_BEGIN(MPM_TRACE_MUTUAL);
  wait_for_previous_grid();
  MPM_TRACE_WAITED();
  __shared__ int32_t sh[32];
  __shared__ int64_t sh64[32];
  __shared__ int is_last;
  const int b = blockIdx.x;
  const int64_t base = ws.soff[b];
  const int n = static_cast<int>(ws.soff[b + 1] - base);
  int carry = 0;
  for (int c0 = 0; c0 < n; c0 += kScanThreads) {
    const int i = c0 + threadIdx.x;
    int rep = 0, partner = -1;
    if (i < n) {
      int j = key_index(ws.keys[base + i]);
      // b(i) lies in i's chunk (the whole image without chunking), and only a
      // token alone in its chunk has none.
      const int64_t cstart = chunk > 0 ? (i / chunk) * chunk : 0;
      const int64_t clen = chunk > 0 ? (n - cstart < chunk ? n - cstart : chunk) : n;
      if (j >= n || j == i || (j < 0 && clen > 1) || (j >= 0 && (j < cstart || j >= cstart + clen))) {
        report(ws.status, MPM_ERR_DEVICE_CHECK, static_cast<int32_t>(base + i));
        j = -1;
      }
      // (i, j) is a pair of P when b(j) = i as well (Section 3.2).
      if (j >= 0 && key_index(ws.keys[base + j]) == i) partner = j;
      rep = (partner < 0 || i < partner) ? 1 : 0;
    }
    int total;
    const int incl = block_incl_sum<int>(rep, sh, &total);
    if (rep) {
      const int r = carry + incl - 1;
      out_map[base + i] = r;
      if (partner > i) out_map[base + partner] = r;
      ws.reps[base + r] = make_int2(i, partner);
    }
    carry += total;
  }
  if (threadIdx.x == 0) {
    ws.count[b] = carry;
    // The ticket increment releases this block's count and, in the last
    // block, acquires every other block's (their increments came first).
    int prev;
    asm volatile("atom.add.acq_rel.gpu.global.s32 %0, [%1], 1;" : "=r"(prev) : "l"(ws.status + 2) : "memory");
    is_last = (prev == batch - 1);
  }
  __syncthreads();
  if (!is_last) return;
  int64_t acc = 0;
  for (int c0 = 0; c0 <= batch; c0 += kScanThreads) {
    const int idx = c0 + threadIdx.x;
    const int64_t v = idx < batch ? static_cast<int64_t>(__ldcg(ws.count + idx)) : 0;
    int64_t total;
    const int64_t incl = block_incl_sum<int64_t>(v, sh64, &total);
    if (idx <= batch) out_offsets[idx] = acc + incl - v;
    acc += total;
  }
  if (threadIdx.x == 0) ws.status[2] = 0;
}

// ---------------------------------------------------------------------------
// Pair average + compaction (Eq. 2): one warp per output row.
// ---------------------------------------------------------------------------
template <int R, int U>
__global__ void __launch_bounds__(kThreads) pair_average_kernel(const uint8_t* __restrict__ tokens,
                                                                uint8_t* __restrict__ out,
                                                                int batch, int64_t rows, int row_bytes,
                                                                bool bf16, Workspace ws,
                                                                const int64_t* __restrict__ out_offsets) {
  MPM_TRACE_BEGIN(MPM_TRACE_PAIR_AVERAGE);
  wait_for_previous_grid();
  MPM_TRACE_WAITED();
  const int lane = threadIdx.x & 31;
  const int64_t warp = (static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x) >> 5;
  const int64_t nwarps = (static_cast<int64_t>(gridDim.x) * kThreads) >> 5;
  const int64_t total = clamp64(out_offsets[batch], 0, rows);
  const int nvec = row_bytes >> 4;
  ImageCursor cur;
  // Each warp writes R consecutive output rows per iteration; all loads of
  // a pass are issued before any store.
  for (int64_t t0 = warp * R; t0 < total; t0 += nwarps * R) {
    const uint4* a[R];
    const uint4* p[R];
    uint4* dst[R];
    bool live[R], pair[R];
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const int64_t t = t0 + r;
      live[r] = t < total;
      pair[r] = false;
      a[r] = p[r] = nullptr;
      dst[r] = reinterpret_cast<uint4*>(out + t * row_bytes);
      if (live[r]) {
        cur.locate(out_offsets, batch, t);
        const int64_t in_base = ws.soff[cur.b];
        const int2 rep = ws.reps[in_base + (t - cur.lo)];
        pair[r] = rep.y >= 0;
        a[r] = reinterpret_cast<const uint4*>(tokens + (in_base + rep.x) * row_bytes);
        p[r] = reinterpret_cast<const uint4*>(tokens + (in_base + (pair[r] ? rep.y : rep.x)) * row_bytes);
      }
    }
    for (int v0 = lane; v0 < nvec; v0 += 32 * U) {
      uint4 va[R][U], vb[R][U];
#pragma unroll
      for (int r = 0; r < R; ++r)
#pragma unroll
        for (int u = 0; u < U; ++u) {
          const int v = v0 + 32 * u;
          if (live[r] && v < nvec) {
            va[r][u] = __ldcs(a[r] + v);
            if (pair[r]) vb[r][u] = __ldcs(p[r] + v);
          }
        }
#pragma unroll
      for (int r = 0; r < R; ++r)
#pragma unroll
        for (int u = 0; u < U; ++u) {
          const int v = v0 + 32 * u;
          if (live[r] && v < nvec) dst[r][v] = pair[r] ? avg16(va[r][u], vb[r][u], bf16) : va[r][u];
        }
    }
  }
}

// ---------------------------------------------------------------------------
// Keys -> nearest neighbour and cosine (test / diagnostics hook).
// ---------------------------------------------------------------------------
__global__ void decode_nn_kernel(int batch, int64_t rows, Workspace ws, int32_t* __restrict__ nn,
                                 float* __restrict__ score) {
  wait_for_previous_grid();
  const int64_t used = ws.soff[batch];
  for (int64_t g = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; g < used;
       g += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const unsigned long long k = ws.keys[g];
    nn[g] = key_index(k);
    if (score != nullptr) score[g] = k == 0ull ? -INFINITY : key_score(k) * ws.inv_norm[g];
  }
}

// ---------------------------------------------------------------------------
// Map composition (Eq. 3).
// ---------------------------------------------------------------------------
// map1 may alias out (in-place composition): each thread reads map1[p]
// before writing out[p], and no other thread touches row p.
__global__ void compose_kernel(const int32_t* map1, const int64_t* __restrict__ off0,
                               int64_t rows0, const int32_t* __restrict__ map2,
                               const int64_t* __restrict__ off1, int64_t rows1, int batch,
                               int32_t* out, int32_t* status) {
  MPM_TRACE_BEGIN(MPM_TRACE_COMPOSE);
  wait_for_previous_grid();
  MPM_TRACE_WAITED();
  const int64_t used = clamp64(off0[batch], 0, rows0);
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t p = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; p < used; p += stride) {
    const int b = find_image(off0, batch, p);
    const int64_t lo0 = __ldg(off0 + b), hi0 = __ldg(off0 + b + 1);
    const int64_t lo1 = __ldg(off1 + b), hi1 = __ldg(off1 + b + 1);
    const int32_t m1 = map1[p];
    int32_t r = -1;
    if (p >= lo0 && p < hi0 && m1 >= 0 && m1 < hi1 - lo1 && lo1 >= 0 && lo1 + m1 < rows1) {
      r = __ldg(map2 + lo1 + m1);
    } else {
      report(status, MPM_ERR_DEVICE_CHECK, static_cast<int32_t>(p));
    }
    out[p] = r;
  }
}

// ---------------------------------------------------------------------------
// Gather reconstruction (Eq. 4), a pure copy.  A warp takes 32 consecutive
// grid rows: lane l resolves row p0 + l (its image, its map entry and the
// source row, all independent loads across the lanes), then the warp copies
// the rows RG at a time with every lane moving 16-byte vectors.  With
// COMPOSE the source is composed on the way (Eq. 3):
// r*(p) = map2[off1_b + map1[p]], and r* is written to out_map if given.
// ---------------------------------------------------------------------------
template <int U, int RG, bool COMPOSE>
__global__ void __launch_bounds__(kThreads) gather_kernel(const uint8_t* __restrict__ merged,
                                                          const int64_t* __restrict__ moff,
                                                          int64_t merged_rows,
                                                          const int32_t* map,
                                                          const int64_t* __restrict__ goff,
                                                          int64_t grid_rows,
                                                          const int32_t* __restrict__ map2,
                                                          const int64_t* __restrict__ off1, int64_t rows1,
                                                          int32_t* out_map, int batch, int row_bytes,
                                                          uint8_t* __restrict__ out, int32_t* status) {
  MPM_TRACE_BEGIN(MPM_TRACE_GATHER);
  wait_for_previous_grid();
  MPM_TRACE_WAITED();
  const int lane = threadIdx.x & 31;
  const int64_t warp = (static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x) >> 5;
  const int64_t nwarps = (static_cast<int64_t>(gridDim.x) * kThreads) >> 5;
  const int64_t used = clamp64(goff[batch], 0, grid_rows);
  const int nvec = row_bytes >> 4;
  ImageCursor cur;
  for (int64_t p0 = warp * 32; p0 < used; p0 += nwarps * 32) {
    // Lane l resolves grid row p0 + l.
    const int64_t p = p0 + lane;
    int64_t src = -1;  // merged row to copy, -1 = none (zero row)
    if (p < used) {
      cur.locate(goff, batch, p);
      const int64_t mlo = __ldg(moff + cur.b), mhi = __ldg(moff + cur.b + 1);
      int32_t m = map[p];
      bool ok = p >= cur.lo && p < cur.hi;
      if (COMPOSE) {
        // Stage-1 index of this grid row, then its stage-2 (merged) index.
        const int64_t lo1 = __ldg(off1 + cur.b), hi1 = __ldg(off1 + cur.b + 1);
        ok = ok && m >= 0 && m < hi1 - lo1 && lo1 >= 0 && lo1 + m < rows1;
        m = ok ? __ldg(map2 + lo1 + m) : -1;
      }
      ok = ok && m >= 0 && m < mhi - mlo && mlo >= 0 && mlo + m < merged_rows;
      if (!ok) report(status, MPM_ERR_DEVICE_CHECK, static_cast<int32_t>(p));
      // This lane alone reads and writes entry p, so out_map may alias map.
      if (COMPOSE && out_map != nullptr) out_map[p] = ok ? m : -1;
      src = ok ? mlo + m : -1;
    }
    const int nrows = static_cast<int>(used - p0 < 32 ? used - p0 : 32);
    for (int r0 = 0; r0 < nrows; r0 += RG) {
      int64_t s[RG];
#pragma unroll
      for (int g = 0; g < RG; ++g) s[g] = __shfl_sync(0xFFFFFFFFu, src, (r0 + g) & 31);
      for (int v0 = lane; v0 < nvec; v0 += 32 * U) {
        uint4 val[RG][U];
#pragma unroll
        for (int g = 0; g < RG; ++g)
#pragma unroll
          for (int u = 0; u < U; ++u) {
            const int v = v0 + 32 * u;
            if (r0 + g < nrows && v < nvec)
              val[g][u] = s[g] >= 0 ? __ldg(reinterpret_cast<const uint4*>(merged + s[g] * row_bytes) + v)
                                    : make_uint4(0, 0, 0, 0);
          }
#pragma unroll
        for (int g = 0; g < RG; ++g)
#pragma unroll
          for (int u = 0; u < U; ++u) {
            const int v = v0 + 32 * u;
            if (r0 + g < nrows && v < nvec)
              __stcs(reinterpret_cast<uint4*>(out + (p0 + r0 + g) * row_bytes) + v, val[g][u]);
          }
      }
    }
  }
}

int grid_for(int num_sms, int per_sm) { return (num_sms > 0 ? num_sms : 1) * per_sm; }

}  // namespace

#ifdef MPM_TRACE
cudaError_t trace_copy_hbm(unsigned long long* out, bool reset) { return trace_table(out, reset); }
#endif

cudaError_t launch_prep(const void* tokens, const int64_t* offsets, int batch, int64_t rows, int dim,
                        bool bf16, AffinityTile tile, const Workspace& ws, int num_sms,
                        cudaStream_t stream) {
  const int row_bytes = dim * (bf16 ? 2 : 4);
  if (ws.split_hi != nullptr) {
    static const int per_sm = resident_per_sm(prep_kernel<true>, kThreads, 8);
    return launch_dependent(prep_kernel<true>, dim3(grid_for(num_sms, per_sm)), dim3(kThreads), 0, stream,
                            static_cast<const uint8_t*>(tokens), offsets, batch, rows, row_bytes, bf16, tile, ws);
  }
  static const int per_sm = resident_per_sm(prep_kernel<false>, kThreads, 8);
  return launch_dependent(prep_kernel<false>, dim3(grid_for(num_sms, per_sm)), dim3(kThreads), 0, stream,
                          static_cast<const uint8_t*>(tokens), offsets, batch, rows, row_bytes, bf16, tile, ws);
}

cudaError_t launch_mutual_compact(int batch, int64_t chunk, const Workspace& ws, int32_t* out_map,
                                  int64_t* out_offsets, cudaStream_t stream) {
  return launch_dependent(mutual_compact_kernel, dim3(batch), dim3(kScanThreads), 0, stream, batch, chunk, ws,
                          out_map, out_offsets);
}

cudaError_t launch_pair_average(const void* tokens, void* out_tokens, int batch, int64_t rows,
                                int dim, bool bf16, const Workspace& ws,
                                const int64_t* out_offsets, int num_sms, cudaStream_t stream) {
  const int row_bytes = dim * (bf16 ? 2 : 4);
  static const int per_sm = resident_per_sm(pair_average_kernel<1, 4>, kThreads, 8);
  return launch_dependent(pair_average_kernel<1, 4>, dim3(grid_for(num_sms, per_sm)), dim3(kThreads), 0, stream,
                          static_cast<const uint8_t*>(tokens), static_cast<uint8_t*>(out_tokens), batch, rows,
                          row_bytes, bf16, ws, out_offsets);
}

cudaError_t launch_decode_nn(int batch, int64_t rows, const Workspace& ws, int32_t* out_nn,
                             float* out_score, int num_sms, cudaStream_t stream) {
  (void)rows;
  return launch_dependent(decode_nn_kernel, dim3(grid_for(num_sms, 4)), dim3(kThreads), 0, stream, batch, rows, ws,
                          out_nn, out_score);
}

cudaError_t launch_compose(const int32_t* map1, const int64_t* off0, int64_t rows0,
                           const int32_t* map2, const int64_t* off1, int64_t rows1, int batch,
                           int32_t* out, int32_t* status, int num_sms, cudaStream_t stream) {
  return launch_dependent(compose_kernel, dim3(grid_for(num_sms, 4)), dim3(kThreads), 0, stream, map1, off0, rows0,
                          map2, off1, rows1, batch, out, status);
}

cudaError_t launch_gather(const void* merged, const int64_t* moff, int64_t merged_rows,
                          const int32_t* map, const int64_t* goff, int64_t grid_rows, int batch,
                          int dim, bool bf16, void* out, int32_t* status, int num_sms,
                          cudaStream_t stream) {
  const int row_bytes = dim * (bf16 ? 2 : 4);
  static const int per_sm = resident_per_sm(gather_kernel<3, 4, false>, kThreads, 8);
  return launch_dependent(gather_kernel<3, 4, false>, dim3(grid_for(num_sms, per_sm)), dim3(kThreads), 0, stream,
                          static_cast<const uint8_t*>(merged), moff, merged_rows, map, goff, grid_rows,
                          static_cast<const int32_t*>(nullptr), static_cast<const int64_t*>(nullptr),
                          static_cast<int64_t>(0), static_cast<int32_t*>(nullptr), batch, row_bytes,
                          static_cast<uint8_t*>(out), status);
}

cudaError_t launch_compose_gather(const void* merged, const int64_t* moff, int64_t merged_rows,
                                  const int32_t* map1, const int64_t* off0, int64_t rows0,
                                  const int32_t* map2, const int64_t* off1, int64_t rows1, int batch, int dim,
                                  bool bf16, void* out, int32_t* out_map, int32_t* status, int num_sms,
                                  cudaStream_t stream) {
  const int row_bytes = dim * (bf16 ? 2 : 4);
  static const int per_sm = resident_per_sm(gather_kernel<3, 4, true>, kThreads, 8);
  return launch_dependent(gather_kernel<3, 4, true>, dim3(grid_for(num_sms, per_sm)), dim3(kThreads), 0, stream,
                          static_cast<const uint8_t*>(merged), moff, merged_rows, map1, off0, rows0, map2, off1,
                          rows1, out_map, batch, row_bytes, static_cast<uint8_t*>(out), status);
}

}  // namespace mpm
