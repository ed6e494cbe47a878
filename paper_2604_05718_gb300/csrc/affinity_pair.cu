// Symmetric affinity + arg max on SM pairs: the default kernel for Eq. 1 and
// Algorithm 1 step 3, for bf16 and fp32 tokens.
//
// Same arithmetic as affinity_tc.cu (raw dot products accumulated in fp32 in
// tensor memory, scaled in fp32 by 1/max(|x|, 1e-12) in the epilogue, packed
// (score, lowest index) keys merged with atomicMax), laid out as follows:
//
//  * A cluster of two CTAs (an SM pair) computes a 256 x 256 tile of
//    G = X X^T with tcgen05.mma.cta_group::2 (M = 256, N = 256).  CTA r holds
//    128 tile rows of A (assigned crosswise, below) and tile columns
//    [128r, 128r + 128) of B in its own shared memory, and receives its 128
//    rows x 256 columns of the accumulator in its own tensor memory.  Each SM therefore stages 64
//    KiB per stage instead of 96 KiB, which leaves room for three stages and
//    cuts the shared-memory traffic of the tensor cores by a third.
//  * bf16 tokens: a stage holds 128 features (two 64-feature TMA boxes per
//    operand) and takes eight K = 16 MMAs.  fp32 tokens (TF32 = true): every
//    value is split as x = hi + lo (hi the tf32 rounding of x, written with
//    lo by the prep kernel), a stage holds 32 features of A hi, A lo, B hi
//    and B lo, and takes twelve K = 8 tf32 MMAs: hi.hi + hi.lo + lo.hi.
//    The MMA warp issues a whole stage and its release commit from one asm
//    block: its sub-partition also runs two epilogue warps, and every
//    instruction it saves per stage keeps the tensor core fed.
//  * Tiles are the 256 x 256 blocks on or above the diagonal of each image's
//    G (of each chunk's, with the chunked similarity), R(R + 1) / 2 of them
//    for R = ceil(N / 256).  Within a tile, every 128-column block above a
//    thread's 128-row block also yields column candidates (row j scores row
//    i by G_ij / |x_i|), as in affinity_tc.cu's symmetric mode; the block
//    below the diagonal of a diagonal tile is skipped.
//  * A tile whose column block holds at most 128 columns of its chunk (the
//    last block of a ragged image: 94 of 256 for an image of 862 tokens) is
//    narrow: its MMAs run with N = 128, each CTA staging 64 of its B rows,
//    and the 8-warp epilogue splits its 128 accumulator columns between
//    both column halves of warps.  With 8 epilogue warps, a last round of
//    tiles that would leave half of the SM pairs idle is dealt as narrow
//    256 x 128 halves instead; a launch of at most 38 tiles (half of the 76
//    SM pairs) is all last round, so each of its tiles is split.  The MMA
//    warp picks the tile shape once per tile, from a bit set while the items
//    were decoded, and issues the tile's stages with compile-time
//    instruction descriptors: a descriptor chosen at run time slowed every
//    tile's issue.
//
// Rows of the tile are assigned crosswise: the leader CTA (rank 0, whose
// warp 1 issues the MMAs) holds tile rows [128, 256) and the peer rows
// [0, 128).  In a diagonal tile the rows [128, 256) skip the block below the
// diagonal, so the lighter half of the epilogue runs on the SM that also
// issues the MMAs: epilogue instructions on the issuing warp's SM
// sub-partition are what slows the MMA issue.
//
// Roles per CTA (2 + EPIW warps): warp 0 loads its CTA's A and B slices with
// TMA and reports the bytes to the leader CTA's barrier; in the leader, warp 1
// allocates tensor memory (jointly with the peer) and issues the MMAs, whose
// completion is multicast to both CTAs; the other warps of each CTA read
// their own tensor memory in slices of 32 rows x 128 columns (EPIW = 8) or
// 32 x 64 (EPIW = 16, rows of few features).  Every wait is bounded; on
// expiry the kernel records MPM_ERR_DEVICE_TIMEOUT and unwinds.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <math.h>

#include <atomic>
#include <type_traits>

#include "mpm.h"
#include "affinity_epilogue.cuh"
#include "common.cuh"
#include "ptx.cuh"

namespace mpm {
namespace {

constexpr int TILE = 256;                      // tile rows and columns
constexpr int HALF = 128;                      // rows of A / B per CTA
constexpr int BOX_K = 64;                      // features per TMA box: one 128-byte swizzle row
constexpr int BK = 128;                        // features per pipeline stage
constexpr int ATOMS = BK / BOX_K;              // swizzle atoms (TMA boxes) per operand slice
constexpr int ATOM_BYTES = HALF * BOX_K * 2;   // 16 KiB
constexpr int STAGES = 3;
constexpr int SLICE_BYTES = ATOMS * ATOM_BYTES;  // 32 KiB: 128 rows x BK features
constexpr int STAGE_BYTES = 2 * SLICE_BYTES;     // A slice + B slice of this CTA
// Epilogue warps: EPIW per CTA, EPIW / 4 per SM sub-partition, each reading
// 32 TMEM lanes x TILE / (EPIW / 4) columns.  Eight (two per sub-partition,
// 128 columns each) leave the MMA-issuing warp most of its sub-partition's
// issue slots, which bounds tiles of many features (measured: 8 warps beat
// 16 and 4 at D = 768 and 1024).  With few features a tile's MMAs are short
// and its epilogue, latency-bound, sets the pace; sixteen warps of 64
// columns hide more of that latency (D = 384: 26.6 instead of 28.6 us).
template <int EPIW>
struct Epi {
  static constexpr int WARPS = EPIW;
  static constexpr int COLS = TILE / (EPIW / 4);
  static constexpr int THREADS = (2 + EPIW) * 32;
  static_assert(COLS <= HALF && HALF % COLS == 0 && COLS % 32 == 0, "a warp's columns lie in one 128-column block");
};
constexpr int kWideEpilogueMaxDim = 512;  // bf16 rows of at most this many features take 16 epilogue warps
constexpr uint32_t TMEM_COLS = 2 * TILE;
constexpr uint32_t IDESC = ptx::idesc_bf16_f32(2 * HALF, TILE);
// Narrow tiles (at most HALF columns of the tile inside the chunk) run
// N = HALF MMAs: half the tensor work, and each CTA holds HALF / 2 B rows.
constexpr uint32_t IDESC_NARROW = ptx::idesc_bf16_f32(2 * HALF, HALF);
// fp32 tokens: three tf32 products per K slice (hi hi + hi lo + lo hi, the
// "3xTF32" split), with a stage of 32 features holding four 16 KiB slices:
// A high, A low, B high, B low (one 128-byte swizzle row of fp32 each).
constexpr int TF_BOX_K = 32;
constexpr int TF_BK = TF_BOX_K;
constexpr uint32_t IDESC_TF32 = ptx::idesc_tf32_f32(2 * HALF, TILE);
constexpr uint32_t IDESC_TF32_NARROW = ptx::idesc_tf32_f32(2 * HALF, HALF);
static_assert(4 * ATOM_BYTES == STAGE_BYTES && HALF * TF_BOX_K * 4 == ATOM_BYTES, "same stage size for both paths");
constexpr uint64_t WAIT_LIMIT_NS = 2000000000ull;
constexpr int kMaxItems = 160;
constexpr int kMaxStagedImages = 511;  // plan and offsets staged in shared memory up to this batch

struct Control {
  uint64_t full[STAGES];        // leader: all four slices of stage s landed
  uint64_t empty[STAGES];       // both: MMAs reading stage s completed
  uint64_t acc_full[2];         // both: accumulator a complete
  uint64_t acc_empty[2];        // leader: both CTAs finished reading accumulator a
  uint64_t drain;               // leader: all MMAs completed
  uint32_t narrow_bits[(kMaxItems + 31) / 32];  // bit k: this cluster's item k is narrow
  uint32_t tmem_base;
  int abort_flag;
};

struct Item {
  int64_t base;  // global row of the first token of the tile's chunk
  int n;         // tokens in the chunk (the image without chunking)
  int row0;      // first row of the tile within the chunk (a multiple of 256)
  int col0;      // first column of the tile within the chunk (a multiple of 128)
  int origin;    // index of the chunk's first token within its image
  int narrow;    // 1: a 256 x 128 tile (N = 128 MMAs) of columns col0 .. col0 + 127
};

template <int EPIW>
constexpr size_t smem_bytes() {
  return 1024 + static_cast<size_t>(STAGES) * STAGE_BYTES + Epi<EPIW>::WARPS * Epi<EPIW>::COLS * sizeof(float) +
         sizeof(Control) + 16 + kMaxItems * sizeof(Item) + 2 * (kMaxStagedImages + 1) * sizeof(int64_t) +
         Epi<EPIW>::WARPS * 32 * sizeof(uint2);
}

// Item w of the launch: image by the plan, its chunk, then the
// upper-triangle tile (I, J), J >= I, of that chunk numbered row by row: row
// I starts at P(I) = I R - I (I - 1) / 2.  `plan` and `soff` are the work
// plan and sanitised offsets, in shared or global memory.
__device__ __forceinline__ Item decode_pair_item(const int64_t* plan, const int64_t* soff, int batch, int64_t w,
                                                 int64_t chunk) {
  int lo_b = 0, hi_b = batch - 1;
  while (lo_b < hi_b) {
    const int mid = (lo_b + hi_b + 1) >> 1;
    if (plan[mid] <= w) lo_b = mid; else hi_b = mid - 1;
  }
  const int b = lo_b;
  int64_t local = w - plan[b];
  const ChunkItem ch = locate_chunk(local, soff[b + 1] - soff[b], AffinityTile{TILE, TILE, AffinityTile::kUpperSquare, chunk});
  local = ch.local;
  Item it;
  it.base = soff[b] + ch.start;
  it.n = static_cast<int>(ch.len);
  it.origin = static_cast<int>(ch.start);
  const int64_t r = (it.n + TILE - 1) / TILE;
  int64_t lo = 0, hi = r - 1;
  while (lo < hi) {
    const int64_t mid = (lo + hi + 1) / 2;
    if (mid * r - mid * (mid - 1) / 2 <= local) lo = mid; else hi = mid - 1;
  }
  local -= lo * r - lo * (lo - 1) / 2;
  it.row0 = static_cast<int>(lo) * TILE;
  it.col0 = static_cast<int>(lo + local) * TILE;
  // At most HALF columns of the tile lie in its chunk: the last column block
  // of a ragged image, e.g. 94 of 256 for an image of 862 tokens.
  it.narrow = it.n - it.col0 <= HALF ? 1 : 0;
  return it;
}

__device__ __forceinline__ bool is_narrow(const Item& it) { return it.narrow != 0; }

// Item w of the launch.  The plan's tiles go to the SM pairs round-robin;
// when their last round (plan tiles split_from .. plan[batch] - 1) would
// leave at least half of the pairs idle, each of its tiles split_from + t is
// dealt as two 256 x 128 halves instead (items split_from + 2 t and
// split_from + 2 t + 1), so that the round takes one narrow tile's time.
__device__ __forceinline__ Item decode_launch_item(const int64_t* plan, const int64_t* soff, int batch, int64_t w,
                                                   int64_t chunk, int64_t split_from) {
  if (w < split_from) return decode_pair_item(plan, soff, batch, w, chunk);
  const int64_t h = w - split_from;
  Item it = decode_pair_item(plan, soff, batch, split_from + (h >> 1), chunk);
  if (h & 1) it.col0 += HALF;
  it.narrow = 1;
  return it;
}

// Item w, for items past the shared-memory list: out of line, so that the
// role loops that fall back on it stay small.
__device__ __noinline__ Item decode_item_slow(const int64_t* plan, const int64_t* soff, int batch, int64_t w,
                                              int64_t chunk, int64_t split_from) {
  return decode_launch_item(plan, soff, batch, w, chunk, split_from);
}

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_id() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%clusterid.x;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_count() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%nclusterid.x;" : "=r"(r));
  return r;
}
// Address of the same shared-memory location in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t map_to_rank(uint32_t saddr, uint32_t rank) {
  uint32_t out;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(out) : "r"(saddr), "r"(rank));
  return out;
}
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// Arrive on an mbarrier of the peer CTA.  The tensor-memory reads this
// releases are ordered by tcgen05.fence::before_thread_sync, so the arrive
// itself keeps the default (CTA-scope) semantics and does not wait for this
// thread's outstanding global atomics.
__device__ __forceinline__ void remote_arrive(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}
// TMA tile load into this CTA's shared memory whose completion is counted on
// an mbarrier of either CTA of the pair.
__device__ __forceinline__ void tma_load_2d_pair(void* dst, const CUtensorMap* map, uint32_t bar_cluster, int32_t x,
                                                 int32_t y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], "
      "[%2];" ::"r"(ptx::smem_addr(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar_cluster), "r"(x), "r"(y)
      : "memory");
}
__device__ __forceinline__ void mma_pair(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                         uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// The eight K = 16 MMAs of one full stage (BK = 128 features: two swizzle
// atoms of four 32-byte K slices each), then the commit that releases the
// stage in both CTAs.  a_desc describes the stage's A slice; the B slice
// follows it by SLICE_BYTES.  One asm block keeps the issuing thread's
// instruction stream short: the MMA warp shares its SM sub-partition with
// four epilogue warps, and the tensor core idles whenever this loop falls
// behind.
__device__ __forceinline__ void mma_stage_full(uint32_t d_tmem, uint64_t a_desc, uint32_t idesc, uint32_t accumulate,
                                               uint64_t* release) {
  static_assert(ATOMS == 2 && (ATOM_BYTES >> 4) == 1024 && (SLICE_BYTES >> 4) == 2048, "offsets below");
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t.reg .b64 a, b;\n\t"
      "setp.ne.b32 p, %3, 0;\n\t"
      "setp.ne.b32 q, %5, 0;\n\t"
      "add.s64 b, %1, 2048;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, b, %2, p;\n\t"
      "add.s64 a, %1, 2;\n\tadd.s64 b, %1, 2050;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], a, b, %2, q;\n\t"
      "add.s64 a, %1, 4;\n\tadd.s64 b, %1, 2052;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], a, b, %2, q;\n\t"
      "add.s64 a, %1, 6;\n\tadd.s64 b, %1, 2054;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], a, b, %2, q;\n\t"
      "add.s64 a, %1, 1024;\n\tadd.s64 b, %1, 3072;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], a, b, %2, q;\n\t"
      "add.s64 a, %1, 1026;\n\tadd.s64 b, %1, 3074;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], a, b, %2, q;\n\t"
      "add.s64 a, %1, 1028;\n\tadd.s64 b, %1, 3076;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], a, b, %2, q;\n\t"
      "add.s64 a, %1, 1030;\n\tadd.s64 b, %1, 3078;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], a, b, %2, q;\n\t"
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%4], %6;\n\t}"
      ::"r"(d_tmem), "l"(a_desc), "r"(idesc), "r"(accumulate), "r"(ptx::smem_addr(release)), "r"(1u),
      "h"(static_cast<uint16_t>(3))
      : "memory");
}

// The twelve MMAs of one full fp32 stage (32 features = four K = 8 slices of
// 32 bytes), three tf32 products per slice, then the release commit.  The
// stage's slices lie at a_desc (A high), +1024 (A low), +2048 (B high) and
// +3072 (B low) in descriptor units of 16 bytes.
__device__ __forceinline__ void mma_stage_tf32x3(uint32_t d_tmem, uint64_t a_desc, uint32_t idesc,
                                                 uint32_t accumulate, uint64_t* release) {
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t.reg .b64 ah, al, bh, bl;\n\t"
      "setp.ne.b32 p, %3, 0;\n\t"
      "setp.ne.b32 q, %5, 0;\n\t"
      "add.s64 al, %1, 1024;\n\tadd.s64 bh, %1, 2048;\n\tadd.s64 bl, %1, 3072;\n\t"
      "tcgen05.mma.cta_group::2.kind::tf32 [%0], %1, bh, %2, p;\n\t"
      "tcgen05.mma.cta_group::2.kind::tf32 [%0], %1, bl, %2, q;\n\t"
      "tcgen05.mma.cta_group::2.kind::tf32 [%0], al, bh, %2, q;\n\t"
      "add.s64 ah, %1, 2;\n\tadd.s64 al, %1, 1026;\n\tadd.s64 bh, %1, 2050;\n\tadd.s64 bl, %1, 3074;\n\t"
      "tcgen05.mma.cta_group::2.kind::tf32 [%0], ah, bh, %2, q;\n\t"
      "tcgen05.mma.cta_group::2.kind::tf32 [%0], ah, bl, %2, q;\n\t"
      "tcgen05.mma.cta_group::2.kind::tf32 [%0], al, bh, %2, q;\n\t"
      "add.s64 ah, %1, 4;\n\tadd.s64 al, %1, 1028;\n\tadd.s64 bh, %1, 2052;\n\tadd.s64 bl, %1, 3076;\n\t"
      "tcgen05.mma.cta_group::2.kind::tf32 [%0], ah, bh, %2, q;\n\t"
      "tcgen05.mma.cta_group::2.kind::tf32 [%0], ah, bl, %2, q;\n\t"
      "tcgen05.mma.cta_group::2.kind::tf32 [%0], al, bh, %2, q;\n\t"
      "add.s64 ah, %1, 6;\n\tadd.s64 al, %1, 1030;\n\tadd.s64 bh, %1, 2054;\n\tadd.s64 bl, %1, 3078;\n\t"
      "tcgen05.mma.cta_group::2.kind::tf32 [%0], ah, bh, %2, q;\n\t"
      "tcgen05.mma.cta_group::2.kind::tf32 [%0], ah, bl, %2, q;\n\t"
      "tcgen05.mma.cta_group::2.kind::tf32 [%0], al, bh, %2, q;\n\t"
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%4], %6;\n\t}"
      ::"r"(d_tmem), "l"(a_desc), "r"(idesc), "r"(accumulate), "r"(ptx::smem_addr(release)), "r"(1u),
      "h"(static_cast<uint16_t>(3))
      : "memory");
}

// One tf32 MMA (K = 8), issued by one thread.
__device__ __forceinline__ void mma_pair_tf32(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                              uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::tf32 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrives on the barrier at this offset in both CTAs once the MMAs issued so
// far completed.
__device__ __forceinline__ void commit_both(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(
          ptx::smem_addr(bar)),
      "h"(static_cast<uint16_t>(3))
      : "memory");
}
__device__ __forceinline__ void commit_local(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(ptx::smem_addr(bar))
               : "memory");
}

// Last, partial stage of a tile (the K slices that hold features), out of
// line: it runs only when D is not a multiple of the stage width, and the
// MMA warp's loop stays small.
__device__ __noinline__ void mma_partial_stage_bf16(uint32_t d_tmem, uint64_t a_desc, uint32_t idesc, int kb,
                                                    int dim, uint64_t* release) {
  for (int kk = 0; kk < BK / 16 && kb * BK + kk * 16 < dim; ++kk) {
    // K = 16 slice kk: swizzle atom kk / 4, 32 bytes per slice within it.
    const uint64_t off = static_cast<uint64_t>((kk / 4) * (ATOM_BYTES >> 4) + (kk % 4) * 2);
    mma_pair(d_tmem, a_desc + off, a_desc + (SLICE_BYTES >> 4) + off, idesc, (kb | kk) != 0 ? 1u : 0u);
  }
  commit_both(release);
}
__device__ __noinline__ void mma_partial_stage_tf32(uint32_t d_tmem, uint64_t a_desc, uint32_t idesc, int kb,
                                                    int dim, uint64_t* release) {
  for (int kk = 0; kk < TF_BK / 8 && kb * TF_BK + kk * 8 < dim; ++kk) {
    const uint64_t ah = a_desc + 2 * kk, al = ah + (ATOM_BYTES >> 4);
    const uint64_t bh = ah + 2 * (ATOM_BYTES >> 4), bl = ah + 3 * (ATOM_BYTES >> 4);
    mma_pair_tf32(d_tmem, ah, bh, idesc, (kb | kk) != 0 ? 1u : 0u);
    mma_pair_tf32(d_tmem, ah, bl, idesc, 1u);
    mma_pair_tf32(d_tmem, al, bh, idesc, 1u);
  }
  commit_both(release);
}

// Bounded wait for the producer and the epilogue: one probe inline, the
// retry loop out of line, so that their loops stay small.  (The MMA warp
// keeps ptx::mbar_wait inline: its waits are short and frequent.)
__device__ __noinline__ bool mbar_wait_retry(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                             uint64_t limit_ns) {
  return ptx::mbar_wait(bar, parity, abort_flag, limit_ns);
}
__device__ __forceinline__ bool mbar_wait_lean(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                               uint64_t limit_ns) {
  return ptx::mbar_try_wait(bar, parity) || mbar_wait_retry(bar, parity, abort_flag, limit_ns);
}

__device__ __forceinline__ void fail(Control* ctl, int32_t* status, int32_t role) {
  ctl->abort_flag = 1;
  report(status, MPM_ERR_DEVICE_TIMEOUT, role);
}

// TF32: fp32 tokens through the three-product tf32 split (tmap = high
// parts, tmap_lo = low parts); otherwise bf16 tokens (tmap_lo unused).
template <bool TF32, int EPIW>
__global__ void __launch_bounds__(Epi<EPIW>::THREADS, 1)
    affinity_pair_kernel(const __grid_constant__ CUtensorMap tmap, const __grid_constant__ CUtensorMap tmap_lo,
                         int batch, int dim, int64_t chunk, Workspace ws) {
  constexpr int kBK = TF32 ? TF_BK : BK;
  constexpr int EPI_WARPS = Epi<EPIW>::WARPS;
  constexpr int EPI_COLS = Epi<EPIW>::COLS;
  constexpr int THREADS = Epi<EPIW>::THREADS;
  MPM_TRACE_BEGIN(MPM_TRACE_AFFINITY);
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (ptx::smem_addr(smem_raw) & 1023u)) & 1023u);
  uint8_t* stages = smem;
  float* scale = reinterpret_cast<float*>(smem + STAGES * STAGE_BYTES);  // [EPI_WARPS][EPI_COLS]
  Control* ctl = reinterpret_cast<Control*>(smem + STAGES * STAGE_BYTES + EPI_WARPS * EPI_COLS * sizeof(float));
  Item* items = reinterpret_cast<Item*>((reinterpret_cast<uintptr_t>(ctl + 1) + 15) & ~static_cast<uintptr_t>(15));
  int64_t* plan_s = reinterpret_cast<int64_t*>(items + kMaxItems);
  int64_t* soff_s = plan_s + kMaxStagedImages + 1;
  uint2* scratch_all = reinterpret_cast<uint2*>(soff_s + kMaxStagedImages + 1);  // [EPI_WARPS][32]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_rank();
  const bool leader = rank == 0;
  const int ksteps = (dim + kBK - 1) / kBK;
  const int64_t clusters = cluster_count();
  const int64_t cid = cluster_id();

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      ptx::mbar_init(&ctl->full[s], 1);
      ptx::mbar_init(&ctl->empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      ptx::mbar_init(&ctl->acc_full[a], 1);
      // Leader's threads arrive one by one, the peer's warps once each.
      ptx::mbar_init(&ctl->acc_empty[a], EPI_WARPS * 32 + EPI_WARPS);
    }
    ptx::mbar_init(&ctl->drain, 1);
    ctl->abort_flag = 0;
    ptx::fence_barrier_init();
    ptx::prefetch_tensor_map(&tmap);
  }
  if (warp == 1) {
    // Both CTAs of the pair take part in the joint allocation.
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     ptx::smem_addr(&ctl->tmem_base)),
                 "r"(TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
  }
  ptx::tc_fence_before_sync();
  __syncthreads();
  cluster_sync();  // barriers of both CTAs exist before any remote signal
  ptx::tc_fence_after_sync();
  const uint32_t tmem = ctl->tmem_base;

  // Everything above touches no data of earlier kernels; from here on the
  // work plan, offsets and norms written by the prep kernel are read.
  wait_for_previous_grid();
  MPM_TRACE_WAITED();
  const bool staged = batch <= kMaxStagedImages;
  if (staged) {
    for (int e = threadIdx.x; e <= batch; e += THREADS) {
      plan_s[e] = ws.plan[e];
      soff_s[e] = ws.soff[e];
    }
    __syncthreads();
  }
  const int64_t* plan = staged ? plan_s : ws.plan;
  const int64_t* soff = staged ? soff_s : ws.soff;
  // A split last round pays only with 8 epilogue warps, whose column halves
  // share a narrow tile's columns; the 16-warp epilogue reads 64 columns per
  // warp for a half tile as for a full one (vit_s stage 2: 1 us slower).
  const int64_t tiles = plan[batch];
  const int64_t rest = tiles % clusters;
  const int64_t split_from = (EPI_WARPS == 8 && rest > 0 && 2 * rest <= clusters) ? tiles - rest : tiles;
  const int64_t total = tiles + (tiles - split_from);  // items: the split tiles count twice
  const int64_t count = total > cid ? (total - 1 - cid) / clusters + 1 : 0;
  static_assert(THREADS >= kMaxItems, "one thread decodes each listed item");
  {
    const int k = threadIdx.x;
    bool nb = false;
    if (k < count && k < kMaxItems) {
      items[k] = decode_launch_item(plan, soff, batch, cid + k * clusters, chunk, split_from);
      nb = is_narrow(items[k]);
    }
    // The MMA warp reads one bit per item instead of the item.
    const uint32_t bits = __ballot_sync(0xFFFFFFFFu, nb);
    if ((k & 31) == 0 && k < kMaxItems) ctl->narrow_bits[k >> 5] = bits;
  }
  __syncthreads();
  auto item = [&](int64_t k) -> Item {
    return k < kMaxItems ? items[k] : decode_item_slow(plan, soff, batch, cid + k * clusters, chunk, split_from);
  };
  volatile int* abort_flag = &ctl->abort_flag;

  if (warp == 0) {
    // ---------------- TMA producer (both CTAs) ----------------
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int issued = 0;
      uint32_t issued_phase = 0;
      bool ok = true;
      for (int64_t k = 0; ok && k < count; ++k) {
        const Item it = item(k);
        const int32_t arow = static_cast<int32_t>(it.base + it.row0 + HALF * (rank ^ 1u));
        const int32_t brow = static_cast<int32_t>(it.base + it.col0 + (is_narrow(it) ? HALF / 2 : HALF) * rank);
        for (int kb = 0; kb < ksteps; ++kb) {
          if (!mbar_wait_lean(&ctl->empty[stage], phase ^ 1u, abort_flag, WAIT_LIMIT_NS)) {
            fail(ctl, ws.status, 11);
            ok = false;
            break;
          }
          uint8_t* sa = stages + stage * STAGE_BYTES;
          const uint32_t full_leader = map_to_rank(ptx::smem_addr(&ctl->full[stage]), 0);
          if (leader) ptx::mbar_arrive_expect_tx(&ctl->full[stage], 2 * STAGE_BYTES);
          if constexpr (TF32) {
            tma_load_2d_pair(sa, &tmap, full_leader, kb * kBK, arow);                    // A high
            tma_load_2d_pair(sa + ATOM_BYTES, &tmap_lo, full_leader, kb * kBK, arow);    // A low
            tma_load_2d_pair(sa + 2 * ATOM_BYTES, &tmap, full_leader, kb * kBK, brow);   // B high
            tma_load_2d_pair(sa + 3 * ATOM_BYTES, &tmap_lo, full_leader, kb * kBK, brow);// B low
          } else {
#pragma unroll
            for (int t = 0; t < ATOMS; ++t) {
              tma_load_2d_pair(sa + t * ATOM_BYTES, &tmap, full_leader, kb * BK + t * BOX_K, arow);
              tma_load_2d_pair(sa + SLICE_BYTES + t * ATOM_BYTES, &tmap, full_leader, kb * BK + t * BOX_K, brow);
            }
          }
          issued |= 1 << stage;
          issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (!ok && leader) {
        for (int s = 0; s < STAGES; ++s)
          if (issued & (1 << s)) ptx::mbar_wait(&ctl->full[s], (issued_phase >> s) & 1u, nullptr, WAIT_LIMIT_NS);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------- MMA issuer (leader) ----------------
    if (leader && lane == 0) {
      int stage = 0, acc = 0;
      uint32_t phase = 0, acc_phase = 0;
      bool ok = true;
      // Descriptor of stage 0's A slice; the others differ only in the
      // start-address field (address / 16, no carry out of its 14 bits).
      const uint64_t desc0 = ptx::sdesc_k_sw128(ptx::smem_addr(stages));
      for (int64_t k = 0; ok && k < count; ++k) {
        if (!ptx::mbar_wait(&ctl->acc_empty[acc], acc_phase ^ 1u, abort_flag, WAIT_LIMIT_NS)) {
          fail(ctl, ws.status, 12);
          break;
        }
        ptx::tc_fence_after_sync();
        const uint32_t d_tmem = tmem + static_cast<uint32_t>(acc * TILE);
        const bool narrow = k < kMaxItems ? ((ctl->narrow_bits[k >> 5] >> (k & 31)) & 1u) != 0u
                                          : is_narrow(decode_item_slow(plan, soff, batch, cid + k * clusters, chunk,
                                                                       split_from));
        // One tile's stages, with its instruction descriptors as compile-time
        // constants (ID, ID_TF32): the tile shape is chosen once per tile,
        // outside the stage loop, so no descriptor is a run-time value.
        auto issue_tile = [&](auto id, auto id_tf32) {
          [[maybe_unused]] constexpr uint32_t ID = decltype(id)::value;            // bf16 instances
          [[maybe_unused]] constexpr uint32_t ID_TF32 = decltype(id_tf32)::value;  // tf32 instance
          for (int kb = 0; kb < ksteps; ++kb) {
            if (!ptx::mbar_wait(&ctl->full[stage], phase, abort_flag, WAIT_LIMIT_NS)) {
              fail(ctl, ws.status, 13);
              ok = false;
              break;
            }
            ptx::tc_fence_after_sync();
            const uint64_t a_desc = desc0 + static_cast<uint64_t>((stage * STAGE_BYTES) >> 4);
            if constexpr (TF32) {
              if ((kb + 1) * kBK <= dim) {
                mma_stage_tf32x3(d_tmem, a_desc, ID_TF32, kb != 0 ? 1u : 0u, &ctl->empty[stage]);
              } else {
                mma_partial_stage_tf32(d_tmem, a_desc, ID_TF32, kb, dim, &ctl->empty[stage]);
              }
            } else if ((kb + 1) * BK <= dim) {
              mma_stage_full(d_tmem, a_desc, ID, kb != 0 ? 1u : 0u, &ctl->empty[stage]);
            } else {
              mma_partial_stage_bf16(d_tmem, a_desc, ID, kb, dim, &ctl->empty[stage]);
            }
            if (++stage == STAGES) {
              stage = 0;
              phase ^= 1u;
            }
          }
        };
        using NarrowId = std::integral_constant<uint32_t, IDESC_NARROW>;
        using NarrowIdTf32 = std::integral_constant<uint32_t, IDESC_TF32_NARROW>;
        using FullId = std::integral_constant<uint32_t, IDESC>;
        using FullIdTf32 = std::integral_constant<uint32_t, IDESC_TF32>;
        if (narrow)
          issue_tile(NarrowId{}, NarrowIdTf32{});
        else
          issue_tile(FullId{}, FullIdTf32{});
        if (!ok) break;
        commit_both(&ctl->acc_full[acc]);
        if (++acc == 2) {
          acc = 0;
          acc_phase ^= 1u;
        }
      }
      commit_local(&ctl->drain);
      ptx::mbar_wait(&ctl->drain, 0, nullptr, WAIT_LIMIT_NS);
    }
    __syncwarp();
  } else {
    // ---------------- epilogue (both CTAs) ----------------
    // Warp (q, quarter) reads tile rows 32q..32q+31 of this CTA and tile
    // columns c0..c0+EPI_COLS-1, c0 = quarter * EPI_COLS.  A narrow tile's
    // accumulator holds HALF columns: the 8-warp epilogue splits them
    // between its two quarters (HALF / 2 each), and the 16-warp one leaves
    // its upper two quarters idle.  Each warp keeps its own copy of its
    // column scales, so no epilogue warp ever waits for another one.
    const int ew = warp - 2;
    const int q = warp & 3;
    const int quarter = ew >> 2;
    const uint32_t lane_addr = static_cast<uint32_t>(q * 32) << 16;
    auto first_col = [&](const Item& t) {
      return (EPI_WARPS == 8 && is_narrow(t)) ? quarter * (HALF / 2) : quarter * EPI_COLS;
    };
    float* my_scale = scale + ew * EPI_COLS;
    uint2* scr = scratch_all + ew * 32;
    int acc = 0;
    uint32_t acc_phase = 0;
    float pf_scale[EPI_COLS / 32], pf_inv = 0.f;
    auto prefetch = [&](const Item& nx) {
      const float nan = __int_as_float(0x7fc00000);  // columns outside the image never win
      const int c0 = first_col(nx);
#pragma unroll
      for (int h = 0; h < EPI_COLS / 32; ++h) {
        const int j = nx.col0 + c0 + 32 * h + lane;
        pf_scale[h] = j < nx.n ? __ldg(ws.inv_norm + nx.base + j) : nan;
      }
      const int r = nx.row0 + HALF * static_cast<int>(rank ^ 1u) + q * 32 + lane;
      const bool col = (nx.col0 + c0) / HALF > (nx.row0 + HALF * static_cast<int>(rank ^ 1u)) / HALF;
      pf_inv = (col && r < nx.n) ? __ldg(ws.inv_norm + nx.base + r) : 0.f;
    };
    const uint32_t empty_leader0 = map_to_rank(ptx::smem_addr(&ctl->acc_empty[0]), 0);
    const uint32_t empty_leader1 = map_to_rank(ptx::smem_addr(&ctl->acc_empty[1]), 0);
    if (count > 0) prefetch(item(0));
    for (int64_t k = 0; k < count; ++k) {
      const Item it = item(k);
#pragma unroll
      for (int h = 0; h < EPI_COLS / 32; ++h) my_scale[32 * h + lane] = pf_scale[h];
      const float inv_i = pf_inv;
      __syncwarp();
      if (!mbar_wait_lean(&ctl->acc_full[acc], acc_phase, abort_flag, WAIT_LIMIT_NS)) {
        fail(ctl, ws.status, 14);
        break;
      }
      if (k + 1 < count) prefetch(item(k + 1));
      ptx::tc_fence_after_sync();
      const bool narrow = is_narrow(it);
      const int c0 = first_col(it);
      const float* sc = my_scale - c0;  // indexed by tile column
      const int row_base = it.row0 + HALF * static_cast<int>(rank ^ 1u) + q * 32;
      const int row = row_base + lane;
      const int jd = row - it.col0;
      const int iblk = (it.row0 + HALF * static_cast<int>(rank ^ 1u)) / HALF;
      const int jblk = (it.col0 + c0) / HALF;
      const bool live = !narrow || c0 < HALF;  // inside the narrow accumulator
      const bool diag = live && jblk == iblk;
      const bool col_update = live && jblk > iblk;
      float best = -INFINITY;
      int bj = -1;
      unsigned long long colcand[EPI_COLS / 32];
#pragma unroll
      for (int h = 0; h < EPI_COLS / 32; ++h) colcand[h] = 0ull;
      const uint32_t taddr = tmem + lane_addr + static_cast<uint32_t>(acc * TILE + c0);
      if constexpr (EPI_COLS > 64) {
        // Column candidates go to the keys inside the slice loop.
        unsigned long long* const colkeys = ws.keys + it.base + it.col0 + c0 + lane;
        const int steps = narrow ? HALF / 2 / 32 : EPI_COLS / 32;
        if (diag) {
          epilogue_slice_rolled<true, false>(taddr, sc, c0, jd, best, bj, inv_i, lane, row_base, it.n, it.col0,
                                             it.origin, scr, colkeys, steps);
        } else if (col_update) {
          epilogue_slice_rolled<false, true>(taddr, sc, c0, jd, best, bj, inv_i, lane, row_base, it.n, it.col0,
                                             it.origin, scr, colkeys, steps);
        }
      } else if (diag) {
        epilogue_slice<EPI_COLS, true, false>(taddr, sc, c0, jd, best, bj, inv_i, lane, row_base, it.n, it.col0,
                                              it.origin, scr, colcand);
      } else if (col_update) {
        epilogue_slice<EPI_COLS, false, true>(taddr, sc, c0, jd, best, bj, inv_i, lane, row_base, it.n, it.col0,
                                              it.origin, scr, colcand);
      }
      // Release the accumulator first, then merge this tile's candidates
      // (the rolled slice has merged its column candidates already).
      ptx::tc_fence_before_sync();
      if (leader) {
        ptx::mbar_arrive(&ctl->acc_empty[acc]);
      } else {
        __syncwarp();
        if (lane == 0) remote_arrive(acc == 0 ? empty_leader0 : empty_leader1);
      }
      if (bj >= 0 && row < it.n) atomicMax(ws.keys + it.base + row, make_key(best, it.origin + it.col0 + bj));
#pragma unroll
      for (int h = 0; h < EPI_COLS / 32; ++h)
        if (colcand[h] != 0ull) atomicMax(ws.keys + it.base + it.col0 + c0 + 32 * h + lane, colcand[h]);
      __syncwarp();  // all lanes done reading my_scale before the next tile overwrites it
      if (++acc == 2) {
        acc = 0;
        acc_phase ^= 1u;
      }
    }
  }

  ptx::tc_fence_before_sync();
  __syncthreads();
  cluster_sync();  // no CTA leaves while its peer may still signal it
  if (warp == 1) {
    ptx::tc_fence_after_sync();
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(TMEM_COLS) : "memory");
  }
}

PFN_cuTensorMapEncodeTiled_v12000 encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      return static_cast<PFN_cuTensorMapEncodeTiled_v12000>(nullptr);
    return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }();
  return fn;
}

}  // namespace

#ifdef MPM_TRACE
cudaError_t trace_copy_pair(unsigned long long* out, bool reset) { return trace_table(out, reset); }
#endif

AffinityTile pair_tile() { return {TILE, TILE, AffinityTile::kUpperSquare}; }

cudaError_t launch_affinity_pair(const void* tokens, int batch, int64_t rows, int dim, bool tf32, int64_t chunk,
                                 const Workspace& ws, int num_sms, cudaStream_t stream) {
  PFN_cuTensorMapEncodeTiled_v12000 encode = encoder();
  if (encode == nullptr) return cudaErrorNotSupported;
  // bf16: the tokens themselves; fp32: the tf32 high and low copies that the
  // prep kernel wrote into the workspace.
  const int esize = tf32 ? 4 : 2;
  const cuuint64_t gdim[2] = {static_cast<cuuint64_t>(dim), static_cast<cuuint64_t>(rows)};
  const cuuint64_t gstride[1] = {static_cast<cuuint64_t>(dim) * esize};
  const cuuint32_t box[2] = {static_cast<cuuint32_t>(tf32 ? TF_BOX_K : BOX_K), HALF};
  const cuuint32_t estride[2] = {1, 1};
  const CUtensorMapDataType type = tf32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
  void* hi = tf32 ? static_cast<void*>(ws.split_hi) : const_cast<void*>(tokens);
  void* lo = tf32 ? static_cast<void*>(ws.split_lo) : const_cast<void*>(tokens);
  if (hi == nullptr || lo == nullptr) return cudaErrorInvalidValue;
  CUtensorMap map, map_lo;
  if (encode(&map, type, 2, hi, gdim, gstride, box, estride, CU_TENSOR_MAP_INTERLEAVE_NONE,
             CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) !=
          CUDA_SUCCESS ||
      encode(&map_lo, type, 2, lo, gdim, gstride, box, estride, CU_TENSOR_MAP_INTERLEAVE_NONE,
             CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) !=
          CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  // Kernel instances: fp32 tokens (8 epilogue warps), bf16 with 8, bf16 with
  // 16 (rows of at most kWideEpilogueMaxDim features).
  static std::atomic<uint64_t> attr_done[3] = {{0}, {0}, {0}};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = 1ull << (dev & 63);
  const int inst = tf32 ? 0 : (dim <= kWideEpilogueMaxDim ? 2 : 1);
  void (*const kernels[3])(CUtensorMap, CUtensorMap, int, int, int64_t, Workspace) = {
      affinity_pair_kernel<true, 8>, affinity_pair_kernel<false, 8>, affinity_pair_kernel<false, 16>};
  const size_t smem[3] = {smem_bytes<8>(), smem_bytes<8>(), smem_bytes<16>()};
  const int threads[3] = {Epi<8>::THREADS, Epi<8>::THREADS, Epi<16>::THREADS};
  auto kernel = kernels[inst];
  if (!(attr_done[inst].load() & bit)) {
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem[inst]));
    if (e != cudaSuccess) return e;
    attr_done[inst].fetch_or(bit);
  }
  const int grid = (num_sms > 1 ? num_sms : 2) & ~1;  // whole SM pairs
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(threads[inst]);
  cfg.dynamicSmemBytes = smem[inst];
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kernel, map, map_lo, batch, dim, chunk, ws);
}

}  // namespace mpm
