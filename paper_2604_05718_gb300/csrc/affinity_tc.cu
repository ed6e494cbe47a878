// Tensor-core affinity + arg max for bf16 tokens (Eq. 1 and Algorithm 1
// step 3), the one dense contraction of MPM.
//
// For an image b, G = X X^T holds the dot products of its raw bf16 tokens.
// The kernel
//   * stages 128 rows (A) and 256 rows (B) of the RAW tokens, 64 features at
//     a time, into shared memory with TMA (128-byte swizzle);
//   * accumulates a 128 x 256 tile of G in fp32 in tensor memory with
//     tcgen05.mma (M = 128, N = 256, K = 16 per instruction; bf16 products
//     are exact in fp32);
//   * reads the tile back with tcgen05.ld and turns it into arg-max
//     candidates: row i scores column j by G_ij / max(|x_j|, 1e-12) in fp32
//     (the row factor 1/|x_i| of the cosine does not change a row's arg
//     max).  The diagonal and columns outside the image are skipped, and a
//     running (max, lowest j) per row goes into a packed 64-bit key with
//     atomicMax.  The N x N matrix never reaches global memory.
//
// Dense mode computes every tile of G.  Symmetric mode (the default) uses
// G_ij = G_ji.  With 128-wide blocks I (rows) and J (columns), it computes
// only the tiles that contain a block with J >= I.  From an off-diagonal
// block it takes both the row candidates (rows of I over columns of J) and
// the column candidates: row j of block J scores row i of block I by
// G_ij / |x_i|, which is the same quantity its own row would have produced.
// A warp max and a ballot per column of each 32 x 32 block give every
// column its best (score, lowest i).  Shared-memory 64-bit atomicMax combines the four row
// groups, and the last warp to finish a tile flushes the 256 column keys to
// global memory.  Both modes merge candidates with the same packed-key
// atomicMax, so the result does not depend on which tile saw a pair first.
//
// The kernel is persistent (one CTA per SM) and warp-specialised:
//   warp 0    TMA producer (4-stage shared-memory ring)
//   warp 1    TMEM allocator and MMA issuer (two 256-column accumulators)
//   warps 2-17 epilogue: each of the 4 TMEM lane groups (32 rows) is read by
//             four warps, one per 64-column quarter, so a tile's epilogue
//             overlaps the next tile's MMAs.
// Every wait is bounded.  On expiry the kernel records
// MPM_ERR_DEVICE_TIMEOUT, lets in-flight copies and MMAs finish, frees its
// tensor memory and returns.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <math.h>

#include <atomic>
#include <mutex>

#include "mpm.h"
#include "affinity_epilogue.cuh"
#include "common.cuh"
#include "ptx.cuh"

namespace mpm {
namespace {

constexpr int BM = 128;                        // tile rows = TMEM lanes = one 128 block
constexpr int BN = 256;                        // tile columns = MMA N = two 128 blocks
constexpr int BK = 64;                         // bf16 features per swizzled row
constexpr int TMA_ROWS = 128;                  // rows per TMA box
constexpr int STAGES = 4;
constexpr int A_BYTES = BM * BK * 2;           // 16 KiB
constexpr int B_BYTES = BN * BK * 2;           // 32 KiB
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int EPI_WARPS = 16;                  // 4 per TMEM lane group, 64 columns each
constexpr int EPI_COLS = BN / (EPI_WARPS / 4);  // columns read by one epilogue warp
constexpr int THREADS = (2 + EPI_WARPS) * 32;
constexpr uint32_t TMEM_COLS = 2 * BN;         // double-buffered accumulator
constexpr uint32_t IDESC = ptx::idesc_bf16_f32(BM, BN);
constexpr uint32_t IDESC_HALF = ptx::idesc_bf16_f32(BM, BN / 2);  // upper 128-column block only
constexpr uint64_t WAIT_LIMIT_NS = 2000000000ull;  // 2 s per wait

struct Control {
  uint64_t full[STAGES];       // TMA bytes landed in stage s
  uint64_t empty[STAGES];      // MMAs reading stage s completed
  uint64_t acc_full[2];        // accumulator a complete
  uint64_t acc_empty[2];       // epilogue finished reading accumulator a
  uint64_t scale_ready[2];     // column scales of accumulator a written
  uint64_t drain;              // all MMAs completed (teardown)
  unsigned long long colkey[2][BN];  // symmetric mode: column candidates of accumulator a
  int colcount[2];             // epilogue warps done with accumulator a's column keys
  uint32_t tmem_base;
  int abort_flag;
};

struct Item {
  int64_t base;  // first row of the image
  int n;         // tokens in the image
  int row0;      // first local row of the tile (row block I = row0 / 128)
  int col0;      // first local column of the tile (column blocks 2T, 2T+1 with T = col0 / 256)
  bool upper_only;  // symmetric mode: block 2T lies below the diagonal, so only
                    // block 2T+1 (the diagonal block) is loaded and multiplied
};

// A CTA decodes its first kMaxItems work items once, at kernel start, into
// shared memory (one binary search per item, done in parallel) instead of
// every role repeating the search for every tile.
constexpr int kMaxItems = 160;

constexpr size_t SMEM_BYTES = 1024 + static_cast<size_t>(STAGES) * STAGE_BYTES + 2 * BN * sizeof(float) +
                              sizeof(Control) + 16 + kMaxItems * sizeof(Item) + EPI_WARPS * 32 * sizeof(uint2);

template <bool SYM>
__device__ __forceinline__ Item decode_item(const Workspace& ws, int batch, int64_t w) {
  const int b = find_item_image(ws.plan, batch, w);
  int64_t local = w - __ldg(ws.plan + b);
  Item it;
  it.base = __ldg(ws.soff + b);
  it.n = static_cast<int>(__ldg(ws.soff + b + 1) - it.base);
  const int64_t c = (it.n + BN - 1) / BN;
  if (!SYM) {
    it.row0 = static_cast<int>(local / c) * BM;
    it.col0 = static_cast<int>(local % c) * BN;
    it.upper_only = false;
    return it;
  }
  // Symmetric tiling (see affinity_tiles): row blocks 2m and 2m+1 start at
  // prefix P(m) = 2mC - m(m-1); find the last pair whose prefix is <= local
  // by bisection, then the block within the pair.
  const int64_t r = (it.n + BM - 1) / BM;
  int64_t lo = 0, hi = (r - 1) / 2;
  while (lo < hi) {
    const int64_t mid = (lo + hi + 1) / 2;
    if (2 * mid * c - mid * (mid - 1) <= local) lo = mid; else hi = mid - 1;
  }
  local -= 2 * lo * c - lo * (lo - 1);
  const int64_t per = c - lo;  // tiles of each row block of the pair
  const int64_t blk = 2 * lo + (local >= per ? 1 : 0);
  if (local >= per) local -= per;
  it.row0 = static_cast<int>(blk) * BM;
  it.col0 = static_cast<int>(lo + local) * BN;
  it.upper_only = it.col0 / BM < blk;
  return it;
}

__device__ __forceinline__ void fail(Control* ctl, int32_t* status, int32_t role) {
  ctl->abort_flag = 1;
  report(status, MPM_ERR_DEVICE_TIMEOUT, role);
}

template <bool SYM>
__global__ void __launch_bounds__(THREADS, 1)
    affinity_tc_kernel(const __grid_constant__ CUtensorMap tmap, int batch, int ksteps, Workspace ws) {
  extern __shared__ uint8_t smem_raw[];
  wait_for_previous_grid();
  uint8_t* smem = smem_raw + ((1024u - (ptx::smem_addr(smem_raw) & 1023u)) & 1023u);
  uint8_t* stages = smem;
  float* scale = reinterpret_cast<float*>(smem + STAGES * STAGE_BYTES);  // [2][BN]
  Control* ctl = reinterpret_cast<Control*>(smem + STAGES * STAGE_BYTES + 2 * BN * sizeof(float));
  Item* items = reinterpret_cast<Item*>(
      (reinterpret_cast<uintptr_t>(ctl + 1) + 15) & ~static_cast<uintptr_t>(15));
  uint2* scratch_all = reinterpret_cast<uint2*>(items + kMaxItems);  // [EPI_WARPS][32]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // This CTA's items are w = blockIdx.x + k * gridDim.x, k < count.
  const int64_t total = __ldg(ws.plan + batch);
  const int64_t count = total > blockIdx.x ? (total - 1 - blockIdx.x) / gridDim.x + 1 : 0;
  for (int64_t k = threadIdx.x; k < count && k < kMaxItems; k += THREADS)
    items[k] = decode_item<SYM>(ws, batch, blockIdx.x + k * gridDim.x);
  auto item = [&](int64_t k) -> Item {
    return k < kMaxItems ? items[k] : decode_item<SYM>(ws, batch, blockIdx.x + k * gridDim.x);
  };
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      ptx::mbar_init(&ctl->full[s], 1);
      ptx::mbar_init(&ctl->empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      ptx::mbar_init(&ctl->acc_full[a], 1);
      ptx::mbar_init(&ctl->acc_empty[a], EPI_WARPS * 32);
      ptx::mbar_init(&ctl->scale_ready[a], EPI_WARPS * 32);
      ctl->colcount[a] = 0;
    }
    ptx::mbar_init(&ctl->drain, 1);
    ctl->abort_flag = 0;
    ptx::fence_barrier_init();
    ptx::prefetch_tensor_map(&tmap);
  }
  if (SYM) {
    for (int e = threadIdx.x; e < 2 * BN; e += THREADS) (&ctl->colkey[0][0])[e] = 0ull;
  }
  if (warp == 1) {
    ptx::tmem_alloc(&ctl->tmem_base, TMEM_COLS);
    ptx::tmem_relinquish();
  }
  ptx::tc_fence_before_sync();
  __syncthreads();
  ptx::tc_fence_after_sync();
  const uint32_t tmem = ctl->tmem_base;
  volatile int* abort_flag = &ctl->abort_flag;

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int issued = 0;                 // bit s: stage s has a load in flight or landed
      uint32_t issued_phase = 0;      // bit s: parity of that load's phase
      bool ok = true;
      for (int64_t k = 0; ok && k < count; ++k) {
        const Item it = item(k);
        const int32_t arow = static_cast<int32_t>(it.base + it.row0);
        const int32_t brow = static_cast<int32_t>(it.base + it.col0);
        for (int kb = 0; kb < ksteps; ++kb) {
          if (!ptx::mbar_wait(&ctl->empty[stage], phase ^ 1u, abort_flag, WAIT_LIMIT_NS)) {
            fail(ctl, ws.status, 1);
            ok = false;
            break;
          }
          uint8_t* sa = stages + stage * STAGE_BYTES;
          uint8_t* sb = sa + A_BYTES;
          ptx::mbar_arrive_expect_tx(&ctl->full[stage], it.upper_only ? A_BYTES + B_BYTES / 2 : STAGE_BYTES);
          ptx::tma_load_2d(sa, &tmap, &ctl->full[stage], kb * BK, arow);
          if (!it.upper_only) ptx::tma_load_2d(sb, &tmap, &ctl->full[stage], kb * BK, brow);
          ptx::tma_load_2d(sb + B_BYTES / 2, &tmap, &ctl->full[stage], kb * BK, brow + TMA_ROWS);
          issued |= 1 << stage;
          issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (!ok) {
        // Let every copy already issued land before shared memory goes away.
        for (int s = 0; s < STAGES; ++s)
          if (issued & (1 << s)) ptx::mbar_wait(&ctl->full[s], (issued_phase >> s) & 1u, nullptr, WAIT_LIMIT_NS);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      int stage = 0, acc = 0;
      uint32_t phase = 0, acc_phase = 0;
      bool ok = true;
      for (int64_t k = 0; ok && k < count; ++k) {
        // Tiles whose lower 128-column block is below the diagonal multiply
        // only the upper block (N = 128) into the upper half of the accumulator.
        const bool upper_only = SYM && item(k).upper_only;
        const uint32_t idesc = upper_only ? IDESC_HALF : IDESC;
        const uint32_t b_off = upper_only ? B_BYTES / 2 : 0;
        if (!ptx::mbar_wait(&ctl->acc_empty[acc], acc_phase ^ 1u, abort_flag, WAIT_LIMIT_NS)) {
          fail(ctl, ws.status, 2);
          break;
        }
        ptx::tc_fence_after_sync();
        const uint32_t d_tmem = tmem + static_cast<uint32_t>(acc * BN) + (upper_only ? BN / 2 : 0);
        for (int kb = 0; kb < ksteps; ++kb) {
          if (!ptx::mbar_wait(&ctl->full[stage], phase, abort_flag, WAIT_LIMIT_NS)) {
            fail(ctl, ws.status, 3);
            ok = false;
            break;
          }
          ptx::tc_fence_after_sync();
          const uint32_t a_addr = ptx::smem_addr(stages + stage * STAGE_BYTES);
          const uint32_t b_addr = a_addr + A_BYTES + b_off;
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            // Advancing the start address by 32 bytes steps K by 16 inside
            // the 128-byte swizzled row.
            ptx::mma_bf16(d_tmem, ptx::sdesc_k_sw128(a_addr + k * 32), ptx::sdesc_k_sw128(b_addr + k * 32), idesc,
                          (kb | k) != 0 ? 1u : 0u);
          }
          ptx::mma_commit(&ctl->empty[stage]);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        ptx::mma_commit(&ctl->acc_full[acc]);
        if (++acc == 2) {
          acc = 0;
          acc_phase ^= 1u;
        }
      }
      // Every MMA issued by this thread must finish before TMEM is freed.
      ptx::mma_commit(&ctl->drain);
      ptx::mbar_wait(&ctl->drain, 0, nullptr, WAIT_LIMIT_NS);
    }
    __syncwarp();
  } else {
    // ---------------- epilogue ----------------
    const int ew = warp - 2;                 // 0..EPI_WARPS-1
    const int q = warp & 3;                  // TMEM lane group of this warp
    const int quarter = ew >> 2;             // 64-column slice of the tile
    const int et = ew * 32 + lane;           // column whose scale this thread loads (if < BN)
    const uint32_t lane_addr = static_cast<uint32_t>(q * 32) << 16;
    int acc = 0;
    uint32_t acc_phase = 0;
    // The global values a tile needs (its column scale for this thread, and
    // 1/|x_i| of this thread's row when it takes column candidates) are
    // fetched one tile ahead, so their latency hides behind the current tile.
    float pf_scale = 0.f, pf_inv = 0.f;
    auto prefetch = [&](const Item& nx) {
      const int j = nx.col0 + et;
      pf_scale = (et < BN && j < nx.n) ? __ldg(ws.inv_norm + nx.base + j) : __int_as_float(0x7fc00000);
      const int r = nx.row0 + q * 32 + lane;
      const bool col = SYM && (nx.col0 + quarter * EPI_COLS) / BM > nx.row0 / BM;
      pf_inv = (col && r < nx.n) ? __ldg(ws.inv_norm + nx.base + r) : 0.f;
    };
    if (count > 0) prefetch(item(0));
    for (int64_t k = 0; k < count; ++k) {
      const Item it = item(k);
      float* sc = scale + acc * BN;
      if (et < BN) sc[et] = pf_scale;  // NaN for columns outside the image: never wins
      const float inv_i = pf_inv;
      ptx::mbar_arrive(&ctl->scale_ready[acc]);
      if (!ptx::mbar_wait(&ctl->scale_ready[acc], acc_phase, abort_flag, WAIT_LIMIT_NS) ||
          !ptx::mbar_wait(&ctl->acc_full[acc], acc_phase, abort_flag, WAIT_LIMIT_NS)) {
        fail(ctl, ws.status, 4);
        break;
      }
      if (k + 1 < count) prefetch(item(k + 1));
      ptx::tc_fence_after_sync();
      const int row_base = it.row0 + q * 32;
      const int row = row_base + lane;             // local row owned by this thread
      const int jd = row - it.col0;                // its diagonal column within the tile
      const int c0 = quarter * EPI_COLS;           // first tile column of this warp
      const int iblk = it.row0 / BM;
      const int jblk = (it.col0 + c0) / BM;        // the 128-column block of this warp's slice
      // Symmetric mode skips blocks below the diagonal (their pairs come from
      // the mirrored block) and takes column candidates above it.
      const bool diag = jblk == iblk;
      const bool read = !SYM || jblk >= iblk;
      const bool col_update = SYM && jblk > iblk;
      float best = -INFINITY;
      int bj = -1;
      if (read) {
#pragma unroll 1
        for (int c = c0; c < c0 + EPI_COLS; c += 32) {
          uint32_t v[32];
          ptx::tmem_ld_32x32b_x32(tmem + lane_addr + static_cast<uint32_t>(acc * BN + c), v);
          ptx::tmem_wait_ld(v);
          uint2* scr = scratch_all + ew * 32;
          if (diag) {
            epilogue_chunk<true, false>(v, sc, c, jd, best, bj, inv_i, lane, row_base, it.n, it.col0, scr);
          } else if (col_update) {
            const unsigned long long key =
                epilogue_chunk<false, true>(v, sc, c, jd, best, bj, inv_i, lane, row_base, it.n, it.col0, scr);
            if (key != 0ull) atomicMax(&ctl->colkey[acc][c + lane], key);
          } else {
            epilogue_chunk<false, false>(v, sc, c, jd, best, bj, inv_i, lane, row_base, it.n, it.col0, scr);
          }
        }
      }
      ptx::tc_fence_before_sync();
      ptx::mbar_arrive(&ctl->acc_empty[acc]);
      if (bj >= 0 && row < it.n) atomicMax(ws.keys + it.base + row, make_key(best, it.col0 + bj));
      if (SYM) {
        // The last epilogue warp to finish this tile flushes its column keys.
        __threadfence_block();
        __syncwarp();
        int last = 0;
        if (lane == 0) last = atomicAdd(&ctl->colcount[acc], 1) == EPI_WARPS - 1;
        last = __shfl_sync(0xFFFFFFFFu, last, 0);
        if (last) {
          __threadfence_block();
          for (int e = lane; e < BN; e += 32) {
            const unsigned long long k = ctl->colkey[acc][e];
            if (k != 0ull) {
              atomicMax(ws.keys + it.base + it.col0 + e, k);
              ctl->colkey[acc][e] = 0ull;
            }
          }
          if (lane == 0) ctl->colcount[acc] = 0;
          __threadfence_block();
        }
      }
      if (++acc == 2) {
        acc = 0;
        acc_phase ^= 1u;
      }
    }
  }

  ptx::tc_fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    ptx::tc_fence_after_sync();
    ptx::tmem_dealloc(tmem, TMEM_COLS);
  }
}

PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// The shared-memory opt-in is a per-device attribute: set it once per
// device and kernel instance.
template <bool SYM>
cudaError_t ensure_smem_attr() {
  static std::atomic<uint64_t> done{0};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = 1ull << (dev & 63);
  if (!(done.load() & bit)) {
    e = cudaFuncSetAttribute(affinity_tc_kernel<SYM>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(SMEM_BYTES));
    if (e != cudaSuccess) return e;
    done.fetch_or(bit);
  }
  return cudaSuccess;
}

}  // namespace

AffinityTile tc_tile(bool symmetric) {
  return {BM, BN, symmetric ? AffinityTile::kSymmetric : AffinityTile::kDense};
}

bool tc_available() { return get_encode() != nullptr; }

cudaError_t launch_affinity_tc(const void* tokens, int batch, int64_t rows, int dim, bool symmetric,
                               const Workspace& ws, int num_sms, cudaStream_t stream) {
  PFN_cuTensorMapEncodeTiled_v12000 encode = get_encode();
  if (encode == nullptr) return cudaErrorNotSupported;
  CUtensorMap map;
  const cuuint64_t gdim[2] = {static_cast<cuuint64_t>(dim), static_cast<cuuint64_t>(rows)};
  const cuuint64_t gstride[1] = {static_cast<cuuint64_t>(dim) * 2};
  const cuuint32_t box[2] = {BK, TMA_ROWS};
  const cuuint32_t estride[2] = {1, 1};
  if (encode(&map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(tokens), gdim, gstride, box, estride,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  const int ksteps = (dim + BK - 1) / BK;
  const int grid = num_sms > 0 ? num_sms : 1;
  cudaError_t e;
  if (symmetric) {
    e = ensure_smem_attr<true>();
    if (e != cudaSuccess) return e;
    return launch_dependent(affinity_tc_kernel<true>, dim3(grid), dim3(THREADS), SMEM_BYTES, stream, map, batch,
                            ksteps, ws);
  }
  e = ensure_smem_attr<false>();
  if (e != cudaSuccess) return e;
  return launch_dependent(affinity_tc_kernel<false>, dim3(grid), dim3(THREADS), SMEM_BYTES, stream, map, batch, ksteps,
                          ws);
}

}  // namespace mpm
