// Tensor-core affinity + arg max for bf16 tokens (Eq. 1 and Algorithm 1
// step 3), the one dense contraction of MPM.
//
// For every image b and every 128 x 256 tile of its N_b x N_b dot-product
// matrix X X^T, the kernel
//   * stages 128 rows (A) and 256 rows (B) of the RAW bf16 tokens, 64
//     features at a time, into shared memory with TMA (128-byte swizzle);
//   * accumulates A B^T in fp32 in tensor memory with tcgen05.mma
//     (M = 128, N = 256, K = 16 per instruction; bf16 products are exact in
//     fp32);
//   * reads the accumulator back with tcgen05.ld and scales column j by
//     1/max(|x_j|, 1e-12) in fp32.  Because 1/|x_i| is constant along a row,
//     the row arg max of this score is the arg max of the cosine S_ij.  The
//     diagonal and columns outside the image are skipped; a running
//     (max, lowest j) per row is merged into the packed 64-bit key with
//     atomicMax.  The N x N matrix never reaches global memory.
//
// The kernel is persistent (one CTA per SM) and warp-specialised:
//   warp 0    TMA producer (4-stage shared-memory ring)
//   warp 1    TMEM allocator and MMA issuer (two 256-column accumulators)
//   warps 2-9 epilogue: each of the 4 TMEM lane groups is read by two warps,
//             one per 128-column half, so a tile's epilogue overlaps the
//             next tile's MMAs.
// Every wait is bounded; on expiry the kernel records
// MPM_ERR_DEVICE_TIMEOUT, lets in-flight copies and MMAs finish, frees its
// tensor memory and returns.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <math.h>

#include <atomic>
#include <mutex>

#include "../../include/mpm.h"
#include "common.cuh"
#include "ptx.cuh"

namespace mpm {
namespace {

constexpr int BM = 128;                        // tile rows = TMEM lanes
constexpr int BN = 256;                        // tile columns = MMA N
constexpr int BK = 64;                         // bf16 features per swizzled row
constexpr int TMA_ROWS = 128;                  // rows per TMA box
constexpr int STAGES = 4;
constexpr int A_BYTES = BM * BK * 2;           // 16 KiB
constexpr int B_BYTES = BN * BK * 2;           // 32 KiB
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int EPI_WARPS = 8;
constexpr int THREADS = (2 + EPI_WARPS) * 32;
constexpr uint32_t TMEM_COLS = 2 * BN;         // double-buffered accumulator
constexpr uint32_t IDESC = ptx::idesc_bf16_f32(BM, BN);
constexpr uint64_t WAIT_LIMIT_NS = 2000000000ull;  // 2 s per wait

struct Control {
  uint64_t full[STAGES];       // TMA bytes landed in stage s
  uint64_t empty[STAGES];      // MMAs reading stage s completed
  uint64_t acc_full[2];        // accumulator a complete
  uint64_t acc_empty[2];       // epilogue finished reading accumulator a
  uint64_t scale_ready[2];     // column scales of accumulator a written
  uint64_t drain;              // all MMAs completed (teardown)
  uint32_t tmem_base;
  int abort_flag;
};

constexpr size_t SMEM_BYTES = 1024 + static_cast<size_t>(STAGES) * STAGE_BYTES + 2 * BN * sizeof(float) +
                              sizeof(Control);

struct Item {
  int64_t base;  // first row of the image
  int n;         // tokens in the image
  int row0;      // first local row of the tile
  int col0;      // first local column of the tile
};

__device__ __forceinline__ Item decode_item(const Workspace& ws, int batch, int64_t w) {
  const int b = find_item_image(ws.plan, batch, w);
  const int64_t local = w - __ldg(ws.plan + b);
  Item it;
  it.base = __ldg(ws.soff + b);
  it.n = static_cast<int>(__ldg(ws.soff + b + 1) - it.base);
  const int ct = (it.n + BN - 1) / BN;
  it.row0 = static_cast<int>(local / ct) * BM;
  it.col0 = static_cast<int>(local % ct) * BN;
  return it;
}

__device__ __forceinline__ void fail(Control* ctl, int32_t* status, int32_t role) {
  ctl->abort_flag = 1;
  report(status, MPM_ERR_DEVICE_TIMEOUT, role);
}

__global__ void __launch_bounds__(THREADS, 1)
    affinity_tc_kernel(const __grid_constant__ CUtensorMap tmap, int batch, int ksteps, Workspace ws) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (ptx::smem_addr(smem_raw) & 1023u)) & 1023u);
  uint8_t* stages = smem;
  float* scale = reinterpret_cast<float*>(smem + STAGES * STAGE_BYTES);  // [2][BN]
  Control* ctl = reinterpret_cast<Control*>(smem + STAGES * STAGE_BYTES + 2 * BN * sizeof(float));

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      ptx::mbar_init(&ctl->full[s], 1);
      ptx::mbar_init(&ctl->empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      ptx::mbar_init(&ctl->acc_full[a], 1);
      ptx::mbar_init(&ctl->acc_empty[a], EPI_WARPS * 32);
      ptx::mbar_init(&ctl->scale_ready[a], EPI_WARPS * 32);
    }
    ptx::mbar_init(&ctl->drain, 1);
    ctl->abort_flag = 0;
    ptx::fence_barrier_init();
    ptx::prefetch_tensor_map(&tmap);
  }
  if (warp == 1) {
    ptx::tmem_alloc(&ctl->tmem_base, TMEM_COLS);
    ptx::tmem_relinquish();
  }
  ptx::tc_fence_before_sync();
  __syncthreads();
  ptx::tc_fence_after_sync();
  const uint32_t tmem = ctl->tmem_base;
  const int64_t total = __ldg(ws.plan + batch);
  volatile int* abort_flag = &ctl->abort_flag;

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int issued = 0;                 // bit s: stage s has a load in flight or landed
      uint32_t issued_phase = 0;      // bit s: parity of that load's phase
      bool ok = true;
      for (int64_t w = blockIdx.x; ok && w < total; w += gridDim.x) {
        const Item it = decode_item(ws, batch, w);
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
          ptx::mbar_arrive_expect_tx(&ctl->full[stage], STAGE_BYTES);
          ptx::tma_load_2d(sa, &tmap, &ctl->full[stage], kb * BK, arow);
          ptx::tma_load_2d(sb, &tmap, &ctl->full[stage], kb * BK, brow);
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
      for (int64_t w = blockIdx.x; ok && w < total; w += gridDim.x) {
        if (!ptx::mbar_wait(&ctl->acc_empty[acc], acc_phase ^ 1u, abort_flag, WAIT_LIMIT_NS)) {
          fail(ctl, ws.status, 2);
          break;
        }
        ptx::tc_fence_after_sync();
        const uint32_t d_tmem = tmem + static_cast<uint32_t>(acc * BN);
        for (int kb = 0; kb < ksteps; ++kb) {
          if (!ptx::mbar_wait(&ctl->full[stage], phase, abort_flag, WAIT_LIMIT_NS)) {
            fail(ctl, ws.status, 3);
            ok = false;
            break;
          }
          ptx::tc_fence_after_sync();
          const uint32_t a_addr = ptx::smem_addr(stages + stage * STAGE_BYTES);
          const uint32_t b_addr = a_addr + A_BYTES;
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            // Advancing the start address by 32 bytes steps K by 16 inside
            // the 128-byte swizzled row.
            ptx::mma_bf16(d_tmem, ptx::sdesc_k_sw128(a_addr + k * 32), ptx::sdesc_k_sw128(b_addr + k * 32), IDESC,
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
    const int ew = warp - 2;                 // 0..7
    const int q = warp & 3;                  // TMEM lane group of this warp
    const int half = ew >> 2;                // 128-column half of the tile
    const int et = ew * 32 + lane;           // 0..255: column whose scale this thread loads
    const uint32_t lane_addr = static_cast<uint32_t>(q * 32) << 16;
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int64_t w = blockIdx.x; w < total; w += gridDim.x) {
      const Item it = decode_item(ws, batch, w);
      float* sc = scale + acc * BN;
      {
        const int j = it.col0 + et;
        sc[et] = j < it.n ? __ldg(ws.inv_norm + it.base + j) : __int_as_float(0x7fc00000);  // NaN never wins
      }
      ptx::mbar_arrive(&ctl->scale_ready[acc]);
      if (!ptx::mbar_wait(&ctl->scale_ready[acc], acc_phase, abort_flag, WAIT_LIMIT_NS) ||
          !ptx::mbar_wait(&ctl->acc_full[acc], acc_phase, abort_flag, WAIT_LIMIT_NS)) {
        fail(ctl, ws.status, 4);
        break;
      }
      ptx::tc_fence_after_sync();
      const int row = it.row0 + q * 32 + lane;     // local row owned by this thread
      const int jd = row - it.col0;                // its diagonal column within the tile
      float best = -INFINITY;
      int bj = -1;
#pragma unroll 1
      for (int c = half * (BN / 2); c < (half + 1) * (BN / 2); c += 32) {
        uint32_t v[32];
        ptx::tmem_ld_32x32b_x32(tmem + lane_addr + static_cast<uint32_t>(acc * BN + c), v);
        ptx::tmem_wait_ld(v);
#pragma unroll
        for (int k = 0; k < 32; k += 4) {
          const float4 s4 = *reinterpret_cast<const float4*>(sc + c + k);
          const float sv[4] = {s4.x, s4.y, s4.z, s4.w};
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const float s = __uint_as_float(v[k + u]) * sv[u];
            if (s > best && c + k + u != jd) {
              best = s;
              bj = c + k + u;
            }
          }
        }
      }
      ptx::tc_fence_before_sync();
      ptx::mbar_arrive(&ctl->acc_empty[acc]);
      if (bj >= 0 && row < it.n) atomicMax(ws.keys + it.base + row, make_key(best, it.col0 + bj));
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

}  // namespace

AffinityTile tc_tile() { return {BM, BN}; }

bool tc_available() { return get_encode() != nullptr; }

cudaError_t launch_affinity_tc(const void* tokens, int batch, int64_t rows, int dim, const Workspace& ws,
                               int num_sms, cudaStream_t stream) {
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
  // The shared-memory opt-in is a per-device attribute: set it once per device.
  static std::atomic<uint64_t> attr_done{0};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = 1ull << (dev & 63);
  if (!(attr_done.load() & bit)) {
    e = cudaFuncSetAttribute(affinity_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(SMEM_BYTES));
    if (e != cudaSuccess) return e;
    attr_done.fetch_or(bit);
  }
  const int ksteps = (dim + BK - 1) / BK;
  affinity_tc_kernel<<<num_sms > 0 ? num_sms : 1, THREADS, SMEM_BYTES, stream>>>(map, batch, ksteps, ws);
  return cudaGetLastError();
}

}  // namespace mpm
