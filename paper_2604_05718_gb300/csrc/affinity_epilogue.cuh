// Arg-max candidates from one 32 x 32 block of the dot-product tile, shared
// by the tensor-core affinity kernels (affinity_tc.cu, affinity_pair.cu).
//
// A warp holds 32 rows of the tile (one row per lane, as tcgen05.ld with the
// 32x32b shape delivers them) and 32 consecutive columns c..c+31 in v[].
// Row candidates: row i scores column j by G_ij / |x_j| (sc[] holds 1/|x_j|,
// NaN outside the image so that such columns never win), kept as a running
// (best score, lowest column) per thread.  Column candidates (symmetric
// tilings, blocks above the diagonal): column j scores row i by
// G_ij / |x_i|; a float warp max gives each column's best score and a ballot
// the rows reaching it, the lowest of which wins.  Equal scores always keep
// the lowest index, and -0 counts as +0, so every tiling gives the same
// answer as scoring each row against all of its columns at once.
#pragma once

#include <stdint.h>

#include "common.cuh"
#include "ptx.cuh"

namespace mpm {

// Max of x over the 32 lanes of the warp (fp32).
__device__ __forceinline__ float warp_max_f32(float x) {
  float m;
  asm volatile("redux.sync.max.f32 %0, %1, 0xffffffff;" : "=f"(m) : "f"(x));
  return m;
}

// scratch: 32 uint2 per warp in shared memory (column max bits, winning lanes).
// Returns, in lane L, the packed key of column c + L's candidate from these
// 32 rows (0 when there is none); the caller merges it with atomicMax.
template <bool DIAG, bool COL>
__device__ __forceinline__ unsigned long long epilogue_chunk(const uint32_t (&v)[32], const float* sc, int c,
                                                             int jd, float& best, int& bj, float inv_i, int lane,
                                                             int row_base, int n, int col0, uint2* scratch) {
#pragma unroll
  for (int k = 0; k < 32; k += 4) {
    const float4 s4 = *reinterpret_cast<const float4*>(sc + c + k);
    const float sv[4] = {s4.x, s4.y, s4.z, s4.w};
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const float s = __uint_as_float(v[k + u]) * sv[u];
      if (s > best && (!DIAG || c + k + u != jd)) {
        best = s;
        bj = c + k + u;
      }
    }
  }
  if (COL) {
    // Rows outside the image only occur in an image's last row block, whose
    // column candidates (blocks above it) lie wholly outside the image and
    // are dropped by the column check below; the row check is a guard.
    const bool writer = lane == 0;
#pragma unroll
    for (int k = 0; k < 32; ++k) {
      const float s = __uint_as_float(v[k]) * inv_i;
      const float m = warp_max_f32(s);
      const uint32_t ball = __ballot_sync(0xFFFFFFFFu, s == m);
      if (writer) scratch[k] = make_uint2(__float_as_uint(m), ball);
    }
    __syncwarp();
    const uint2 r = scratch[lane];
    __syncwarp();
    const int winner = row_base + __ffs(static_cast<int>(r.y)) - 1;
    if (r.y != 0u && winner < n && col0 + c + lane < n) return make_key(__uint_as_float(r.x), winner);
  }
  return 0ull;
}

// One 16-column piece of a warp's slice: row candidates into two running
// maxima (even and odd columns), and, with COL, the column maxima and their
// winning rows of these 16 columns into the per-warp scratch entries
// slot .. slot + 15.
template <bool DIAG, bool COL>
__device__ __forceinline__ void epilogue_piece(const uint32_t (&v)[16], const float* sc, int c, int jd, float& best0,
                                               int& bj0, float& best1, int& bj1, float inv_i, int lane,
                                               uint2* scratch, int slot) {
#pragma unroll
  for (int k = 0; k < 16; k += 4) {
    const float4 s4 = *reinterpret_cast<const float4*>(sc + c + k);
    const float sv[4] = {s4.x, s4.y, s4.z, s4.w};
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const float s = __uint_as_float(v[k + u]) * sv[u];
      const int j = c + k + u;
      if (u & 1) {
        if (s > best1 && (!DIAG || j != jd)) {
          best1 = s;
          bj1 = j;
        }
      } else {
        if (s > best0 && (!DIAG || j != jd)) {
          best0 = s;
          bj0 = j;
        }
      }
    }
  }
  if (COL) {
    const bool writer = lane == 0;
#pragma unroll
    for (int k = 0; k < 16; ++k) {
      const float s = __uint_as_float(v[k]) * inv_i;
      const float m = warp_max_f32(s);
      const uint32_t ball = __ballot_sync(0xFFFFFFFFu, s == m);
      if (writer) scratch[slot + k] = make_uint2(__float_as_uint(m), ball);
    }
  }
}

// Column candidate of tile column c + lane from the scratch entries of the
// 32 columns c .. c + 31 (0 when there is none).  `origin` is added to the
// winning row for the key: the tile's first token within its image.
__device__ __forceinline__ unsigned long long column_candidate(const uint2* scratch, int lane, int row_base, int n,
                                                               int col, int origin) {
  __syncwarp();
  const uint2 r = scratch[lane];
  __syncwarp();
  const int winner = row_base + __ffs(static_cast<int>(r.y)) - 1;
  return (r.y != 0u && winner < n && col < n) ? make_key(__uint_as_float(r.x), origin + winner) : 0ull;
}

// A warp's whole COLS-column slice of one accumulator (TMEM columns
// taddr .. taddr + COLS - 1, tile columns c0 ..), read in 16-column pieces
// with the next piece's load in flight while the current one is processed.
// The loop body covers two pieces (32 columns).  Row candidates use two independent running maxima (even and odd columns),
// merged at the end with the lowest-index rule, to halve the dependent
// chain.  colcand[h] receives the column candidate of tile column
// c0 + 32 h + lane (0 when none).
template <int COLS, bool DIAG, bool COL>
__device__ __forceinline__ void epilogue_slice(uint32_t taddr, const float* sc, int c0, int jd, float& best,
                                               int& bj, float inv_i, int lane, int row_base, int n, int col0,
                                               int origin, uint2* scratch,
                                               unsigned long long (&colcand)[COLS / 32]) {
  static_assert(COLS % 32 == 0, "slices are whole 32-column pairs of pieces");
  float best0 = -INFINITY, best1 = -INFINITY;
  int bj0 = -1, bj1 = -1;
  uint32_t va[16], vb[16];
  ptx::tmem_ld_32x32b_x16(taddr, va);
  ptx::tmem_wait_ld(va);
#pragma unroll
  for (int h = 0; h < COLS / 32; ++h) {
    const int c = c0 + 32 * h;
    ptx::tmem_ld_32x32b_x16(taddr + 32 * h + 16, vb);
    epilogue_piece<DIAG, COL>(va, sc, c, jd, best0, bj0, best1, bj1, inv_i, lane, scratch, 0);
    ptx::tmem_wait_ld(vb);
    if (h + 1 < COLS / 32) ptx::tmem_ld_32x32b_x16(taddr + 32 * h + 32, va);
    epilogue_piece<DIAG, COL>(vb, sc, c + 16, jd, best0, bj0, best1, bj1, inv_i, lane, scratch, 16);
    if (COL) {
      const unsigned long long key = column_candidate(scratch, lane, row_base, n, col0 + c + lane, origin);
#pragma unroll
      for (int g = 0; g < COLS / 32; ++g)
        if (g == h) colcand[g] = key;
    }
    if (h + 1 < COLS / 32) ptx::tmem_wait_ld(va);
  }
  // Merge the two chains: larger score, lower column on equal scores.
  if (best1 > best0 || (best1 == best0 && bj1 >= 0 && (bj0 < 0 || bj1 < bj0))) {
    best0 = best1;
    bj0 = bj1;
  }
  if (bj0 >= 0 && (bj < 0 || best0 > best || (best0 == best && bj0 < bj))) {
    best = best0;
    bj = bj0;
  }
}

// The same slice with the 32-column loop left rolled (`steps` steps of 32
// columns), for 128-column slices, whose unrolled code is twice as long:
// the column candidate of tile column c0 + 32 h + lane goes straight to
// colkeys[32 h] (colkeys points at this lane's first column) instead of a
// register array, which would need the loop unrolled.  (Measured on vit_b: step 0.2051-0.2054
// against 0.2069-0.2073 ms unrolled; the 64-column slices of the 16-warp
// epilogue stay unrolled, where the rolled loop was 1.4% slower.)
template <bool DIAG, bool COL>
__device__ __forceinline__ void epilogue_slice_rolled(uint32_t taddr, const float* sc, int c0, int jd, float& best,
                                                      int& bj, float inv_i, int lane, int row_base, int n,
                                                      int col0, int origin, uint2* scratch,
                                                      unsigned long long* colkeys, int steps) {
  float best0 = -INFINITY, best1 = -INFINITY;
  int bj0 = -1, bj1 = -1;
  uint32_t va[16], vb[16];
  ptx::tmem_ld_32x32b_x16(taddr, va);
  ptx::tmem_wait_ld(va);
#pragma unroll 1
  for (int h = 0; h < steps; ++h) {
    const int c = c0 + 32 * h;
    ptx::tmem_ld_32x32b_x16(taddr + 32 * h + 16, vb);
    epilogue_piece<DIAG, COL>(va, sc, c, jd, best0, bj0, best1, bj1, inv_i, lane, scratch, 0);
    ptx::tmem_wait_ld(vb);
    const bool more = h + 1 < steps;
    if (more) ptx::tmem_ld_32x32b_x16(taddr + 32 * h + 32, va);
    epilogue_piece<DIAG, COL>(vb, sc, c + 16, jd, best0, bj0, best1, bj1, inv_i, lane, scratch, 16);
    if (COL) {
      const unsigned long long key = column_candidate(scratch, lane, row_base, n, col0 + c + lane, origin);
      if (key != 0ull) atomicMax(colkeys + 32 * h, key);
    }
    if (more) ptx::tmem_wait_ld(va);
  }
  if (best1 > best0 || (best1 == best0 && bj1 >= 0 && (bj0 < 0 || bj1 < bj0))) {
    best0 = best1;
    bj0 = bj1;
  }
  if (bj0 >= 0 && (bj < 0 || best0 > best || (best0 == best && bj0 < bj))) {
    best = best0;
    bj = bj0;
  }
}

}  // namespace mpm
