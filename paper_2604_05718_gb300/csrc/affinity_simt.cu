// CUDA-core affinity + arg max (Eq. 1 and Algorithm 1 step 3) for any
// dtype: 64 x 64 tiles of the dot-product matrix accumulated with fp32 FMA,
// then an epilogue that scales column j by 1/|x_j|, masks the diagonal and
// columns outside the image, and merges each row's best (score, lowest j)
// into the packed key with a 64-bit atomicMax.  Used for fp32 tokens, where
// tensor-core precision would not be faithful to the fp32 definition.
#include <math.h>

#include "mpm.h"
#include "common.cuh"

namespace mpm {
namespace {

constexpr int BM = 64, BN = 64, BK = 32, kThreads = 256;

template <bool BF16>
__device__ __forceinline__ float load_elem(const uint8_t* tokens, int64_t row, int k, int row_bytes) {
  if (BF16) return __bfloat162float(__ldg(reinterpret_cast<const __nv_bfloat16*>(tokens + row * row_bytes) + k));
  return __ldg(reinterpret_cast<const float*>(tokens + row * row_bytes) + k);
}

template <bool BF16>
__global__ void __launch_bounds__(kThreads) affinity_simt_kernel(const uint8_t* __restrict__ tokens, int batch,
                                                                 int dim, int64_t chunk, Workspace ws) {
  wait_for_previous_grid();
  __shared__ __align__(16) float As[BK][BM + 4];
  __shared__ __align__(16) float Bs[BK][BN + 4];
  __shared__ float scale[BN];
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  const int row_bytes = dim * (BF16 ? 2 : 4);
  const int64_t total = ws.plan[batch];
  for (int64_t w = blockIdx.x; w < total; w += gridDim.x) {
    const int b = find_item_image(ws.plan, batch, w);
    // Tiles of the item's chunk (the whole image without chunking); keys
    // hold indices within the image, so chunk-relative columns get `origin`.
    const ChunkItem ch = locate_chunk(w - ws.plan[b], ws.soff[b + 1] - ws.soff[b],
                                      AffinityTile{BM, BN, AffinityTile::kDense, chunk});
    const int64_t local = ch.local;
    const int64_t base = ws.soff[b] + ch.start;
    const int n = static_cast<int>(ch.len);
    const int origin = static_cast<int>(ch.start);
    const int ct = (n + BN - 1) / BN;
    const int r0 = static_cast<int>(local / ct) * BM;
    const int c0 = static_cast<int>(local % ct) * BN;
    float acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
    for (int k0 = 0; k0 < dim; k0 += BK) {
      for (int e = tid; e < BM * BK; e += kThreads) {
        const int r = e / BK, k = e % BK, kk = k0 + k;
        float va = 0.f, vb = 0.f;
        if (kk < dim) {
          if (r0 + r < n) va = load_elem<BF16>(tokens, base + r0 + r, kk, row_bytes);
          if (c0 + r < n) vb = load_elem<BF16>(tokens, base + c0 + r, kk, row_bytes);
        }
        As[k][r] = va;
        Bs[k][r] = vb;
      }
      __syncthreads();
#pragma unroll 8
      for (int k = 0; k < BK; ++k) {
        const float4 a = *reinterpret_cast<const float4*>(&As[k][ty * 4]);
        const float4 c = *reinterpret_cast<const float4*>(&Bs[k][tx * 4]);
        const float av[4] = {a.x, a.y, a.z, a.w};
        const float cv[4] = {c.x, c.y, c.z, c.w};
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
          for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(av[i], cv[j], acc[i][j]);
      }
      __syncthreads();
    }
    if (tid < BN) {
      const int j = c0 + tid;
      scale[tid] = j < n ? ws.inv_norm[base + j] : __int_as_float(0x7fc00000);  // NaN never wins
    }
    __syncthreads();
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int row = r0 + ty * 4 + i;
      float best = -INFINITY;
      int bj = -1;
#pragma unroll
      for (int jj = 0; jj < 4; ++jj) {
        const int col = tx * 4 + jj;
        const float s = acc[i][jj] * scale[col];
        if (s > best && c0 + col != row) {
          best = s;
          bj = c0 + col;
        }
      }
      unsigned long long key = bj >= 0 ? make_key(best, origin + bj) : 0ull;
#pragma unroll
      for (int d = 8; d > 0; d >>= 1) {
        const unsigned long long o = __shfl_xor_sync(0xFFFFFFFFu, key, d);
        key = o > key ? o : key;
      }
      if (tx == 0 && key != 0ull && row < n) atomicMax(ws.keys + base + row, key);
    }
    __syncthreads();
  }
}

}  // namespace

AffinityTile simt_tile() { return {BM, BN, AffinityTile::kDense}; }

cudaError_t launch_affinity_simt(const void* tokens, int batch, int dim, bool bf16, int64_t chunk,
                                 const Workspace& ws, int num_sms, cudaStream_t stream) {
  const int grid = (num_sms > 0 ? num_sms : 1) * 4;
  const uint8_t* t = static_cast<const uint8_t*>(tokens);
  if (bf16)
    return launch_dependent(affinity_simt_kernel<true>, dim3(grid), dim3(kThreads), 0, stream, t, batch, dim, chunk,
                            ws);
  return launch_dependent(affinity_simt_kernel<false>, dim3(grid), dim3(kThreads), 0, stream, t, batch, dim, chunk,
                          ws);
}

}  // namespace mpm
