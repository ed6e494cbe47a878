/*
 * mpm.h - C ABI of the GB300 (sm_103a) Mutual Pair Merging library.
 *
 * Mutual Pair Merging (MPM, arxiv 2604.05718) shortens the image-token
 * sequence of a ViT: it L2-normalises each image's tokens, takes every
 * token's cosine nearest neighbour, averages each mutual nearest-neighbour
 * pair into one token and records an integer merge map (Section 3.2,
 * Eq. 1-2, Algorithm 1).  Maps of successive insertions are composed
 * (Eq. 3) and a gather restores the full token grid before the decoder
 * (Eq. 4).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - Batches are ragged and packed: image b owns rows [off[b], off[b+1]) of
 *    a row-major [rows, dim] token matrix.  `offsets` arrays are int64
 *    [batch + 1] in DEVICE memory with off[0] == 0, non-decreasing values and
 *    off[batch] <= rows.  Images are independent (Section 3.1); empty images
 *    and single-token images are legal (a single token is a singleton).
 *  - `rows` is the number of rows ALLOCATED for a token or map buffer.  It
 *    bounds every access, so the host never needs to read off[batch].
 *  - Every pointer is a device pointer owned by the caller; the library
 *    allocates and frees nothing.  Token buffers must be 16-byte aligned and
 *    dim must be a multiple of 8 (bf16) or 4 (fp32) so that rows are 16-byte
 *    aligned; otherwise MPM_ERR_ALIGNMENT.  1 <= dim <= 16384.
 *  - Merge maps are int32 and LOCAL: map[off[b] + p] is the output row of
 *    input row p within image b (0-based; Algorithm 1 counts from 1).
 *  - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *    stream).  Every call is asynchronous and stream-ordered.  The returned
 *    status covers host-side validation and launch errors only.
 *  - Device-side problems (offsets that are not monotone, a map entry out of
 *    range, a bounded wait that expired) are recorded, first error wins, in a
 *    device status word: the merge workspace's (read it with
 *    mpm_get_device_status after synchronising), or the optional
 *    `device_status` int32 of compose and gather.  Kernels never trap: a bad
 *    entry is skipped (its output row zeroed, its map entry set to -1).
 */
#ifndef MPM_H
#define MPM_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Only the entry points below are exported from libmpm.so. */
#if defined(__GNUC__)
#define MPM_API __attribute__((visibility("default")))
#else
#define MPM_API
#endif

#define MPM_ABI_VERSION 1
#define MPM_MAX_DIM 16384

typedef enum mpm_dtype {
  MPM_F32 = 0,  /* IEEE binary32 tokens */
  MPM_BF16 = 1  /* bfloat16 tokens */
} mpm_dtype;

typedef enum mpm_status {
  MPM_OK = 0,
  MPM_ERR_INVALID_ARG = 1,     /* null pointer, negative size, bad enum */
  MPM_ERR_UNSUPPORTED = 2,     /* no device of compute capability 10.3, or dim too large */
  MPM_ERR_ALIGNMENT = 3,       /* token pointer or row size not 16-byte aligned */
  MPM_ERR_WORKSPACE = 4,       /* workspace missing, too small or misaligned */
  MPM_ERR_CUDA = 5,            /* a CUDA runtime or driver call failed */
  MPM_ERR_DEVICE_CHECK = 6,    /* (device status) invalid offsets or map entry */
  MPM_ERR_DEVICE_TIMEOUT = 7,  /* (device status) a bounded wait expired */
  MPM_ERR_ALIASING = 8         /* an output buffer overlaps an input buffer */
} mpm_status;

/* Which kernel computes the nearest neighbours (Eq. 1 + arg max). */
typedef enum mpm_nn_algo {
  MPM_NN_AUTO = 0,         /* MPM_NN_TCGEN05_PAIR (both dtypes) */
  MPM_NN_SIMT = 1,         /* CUDA-core fp32 FMA tiles (any dtype) */
  MPM_NN_TCGEN05 = 2,      /* TMA + tcgen05 MMA into TMEM, every tile of X X^T (bf16) */
  MPM_NN_TCGEN05_SYM = 3,  /* as above, tiles on or above the diagonal only, each
                              feeding both its rows and its columns (bf16) */
  MPM_NN_TCGEN05_PAIR = 4  /* symmetric, 256 x 256 tiles on SM pairs with
                              tcgen05.mma.cta_group::2: bf16 products for bf16
                              tokens; for fp32 tokens three tf32 products per
                              term (x = hi + lo with hi the tf32 rounding of x:
                              hi.hi + hi.lo + lo.hi, accumulated in fp32) */
} mpm_nn_algo;

/* Version of this ABI (MPM_ABI_VERSION). */
MPM_API int32_t mpm_abi_version(void);

/* Human-readable name of a status code (static string, never NULL). */
MPM_API const char* mpm_status_string(mpm_status status);

/*
 * Bytes of device workspace that mpm_merge and mpm_nearest_neighbors need
 * for `rows` token rows and `batch` images.  Returns 0 for invalid sizes.
 * The workspace must be 256-byte aligned.  It holds per-row inverse norms,
 * packed arg-max keys, the representative list, per-image counts, sanitised
 * offsets, the work plan and the device status word; for fp32 tokens also
 * the tf32 high and low parts of the tokens (2 * rows * dim floats).
 */
MPM_API size_t mpm_merge_workspace_size(int64_t rows, int32_t batch, int32_t dim, mpm_dtype dtype);

/*
 * One MPM call on every image of a packed batch (Algorithm 1; Eq. 1-2).
 *
 *   tokens       [rows, dim] input tokens (dtype), image b at rows off[b]..
 *   offsets      int64 [batch + 1] device offsets of the input images
 *   out_tokens   [rows, dim] output capacity (dtype).  Image b's N'_b merged
 *                tokens are written at rows out_offsets[b].. in increasing
 *                order of their representative (the pair's lower index);
 *                each is (x_i + x_j) / 2 computed in fp32 and rounded to
 *                nearest even, or the unchanged token for a singleton.
 *   out_offsets  int64 [batch + 1] device, written: exclusive scan of N'_b
 *   out_map      int32 [rows] device, written for rows < off[batch]: the
 *                local output row r(i) of every input row (Algorithm 1)
 *   workspace    device scratch of mpm_merge_workspace_size(...) bytes
 *
 * The nearest neighbour of token i is the j != i of its image maximising the
 * cosine (x_i . x_j) / (|x_i| |x_j|), with norms floored at 1e-12 and ties
 * going to the lowest j; (i, j) merge when each is the other's nearest
 * neighbour (Section 3.2).  N'_b = N_b - #pairs >= ceil(N_b / 2).
 * out_tokens must not overlap tokens (MPM_ERR_ALIASING).
 */
MPM_API mpm_status mpm_merge(const void* tokens, const int64_t* offsets, int32_t batch,
                     int64_t rows, int32_t dim, mpm_dtype dtype, void* out_tokens,
                     int64_t* out_offsets, int32_t* out_map, void* workspace,
                     size_t workspace_bytes, void* stream);

/*
 * mpm_merge with per-kernel CUDA events, for profiling.  When stage_events
 * is not NULL it holds 8 cudaEvent_t handles created by the caller (timing
 * enabled); stage_events[2k] is recorded on `stream` just before kernel k
 * and stage_events[2k+1] just after it, for k = 0 row norms and work plan,
 * 1 affinity + arg max (Eq. 1, Algorithm 1 step 3), 2 mutual check and
 * left-to-right compaction scan (steps 4-6), 3 pair average (Eq. 2).
 * Otherwise identical to mpm_merge (which is this call with NULL).
 */
MPM_API mpm_status mpm_merge_timed(const void* tokens, const int64_t* offsets, int32_t batch,
                                   int64_t rows, int32_t dim, mpm_dtype dtype, void* out_tokens,
                                   int64_t* out_offsets, int32_t* out_map, void* workspace,
                                   size_t workspace_bytes, void* stream,
                                   void* const* stage_events);

/*
 * mpm_merge for callers that cannot allocate device memory.  The paper has
 * no counterpart: this is a deployment convenience.  Some callers must not
 * call cudaMalloc, for example a plug-in inside a framework that has
 * reserved the whole device memory pool, or a latency-critical loop where
 * allocation (which can block and synchronise the device) is banned.  This
 * entry point computes exactly what mpm_merge computes, with the same
 * arguments minus the workspace: its scratch is a fixed array of
 * MPM_NO_ALLOC_SCRATCH_BYTES inside the library, one per device, held until
 * the process exits.
 *  - Limit: it returns MPM_ERR_WORKSPACE when
 *    mpm_merge_workspace_size(rows, batch, dim, dtype) exceeds
 *    MPM_NO_ALLOC_SCRATCH_BYTES (8 MiB), and allocates nothing in any case.
 *    The workspace takes about 20 bytes per row for bf16 tokens, so 8 MiB
 *    holds about 400,000 rows; for fp32 tokens it also holds the two tf32
 *    split copies of the tokens, 20 + 8 * dim bytes per row: about 5,400
 *    rows at dim 192 and 1,360 rows at dim 768.  (Plus 20 bytes per image
 *    and up to 256 bytes of alignment per region either way.)
 *  - Set-up: the array's device address is looked up (cudaGetSymbolAddress,
 *    which can load the module) once per device context, by the first call
 *    on that device; make that first call before any stream capture on the
 *    device.  It is looked up again only after the device's context changed
 *    (a cudaDeviceReset between calls).
 *  - All calls on a device share the one array: calls that overlap on the
 *    GPU (different streams or host threads) race and must be serialised by
 *    the caller.  The array keeps the last call's contents; each call clears
 *    the part that must start at zero, including the device status word.
 *  - Device-detected errors (offsets that are not monotone, a bounded wait
 *    that ran out) go to the status word inside the shared array: read them
 *    with mpm_no_alloc_get_device_status, after this call and before the
 *    next one on the device.
 */
#define MPM_NO_ALLOC_SCRATCH_BYTES (8u << 20)
MPM_API mpm_status mpm_merge_no_alloc(const void* tokens, const int64_t* offsets, int32_t batch,
                                      int64_t rows, int32_t dim, mpm_dtype dtype, void* out_tokens,
                                      int64_t* out_offsets, int32_t* out_map, void* stream);

/*
 * The status word of the no-alloc scratch array on the current device, for
 * callers of mpm_merge_no_alloc (no counterpart in the paper).  Like
 * mpm_get_device_status: copies the first device-detected error of the last
 * mpm_merge_no_alloc call on this device into *host_code (0 = none;
 * otherwise MPM_ERR_DEVICE_CHECK or MPM_ERR_DEVICE_TIMEOUT), synchronising
 * `stream`, then clears the word.  Allocates nothing.
 * Errors: MPM_ERR_INVALID_ARG (host_code NULL), MPM_ERR_CUDA.
 */
MPM_API mpm_status mpm_no_alloc_get_device_status(int32_t* host_code, void* stream);

/*
 * Chunked similarity: mpm_merge with each token's nearest neighbour sought
 * only among the `chunk` consecutive tokens (raster order) of its image that
 * contain it (the last chunk of an image may be shorter).  The paper's
 * discussion proposes chunking the similarity to bound the O(N^2) cosine pass
 * at very large N (Section 5); the rest of Algorithm 1 is unchanged, so
 * pairs never cross a chunk boundary.  A token alone in its chunk has no
 * neighbour and stays a singleton.
 *
 *   chunk  0 = the whole image (exactly mpm_merge); otherwise a multiple of
 *          256 (MPM_ERR_UNSUPPORTED if not; MPM_ERR_INVALID_ARG if negative).
 * Every other argument is as for mpm_merge.  The cost of the affinity step
 * drops from N_b^2 to about N_b * chunk per image.
 */
MPM_API mpm_status mpm_merge_chunked(const void* tokens, const int64_t* offsets, int32_t batch, int64_t rows,
                                     int32_t dim, mpm_dtype dtype, int64_t chunk, void* out_tokens,
                                     int64_t* out_offsets, int32_t* out_map, void* workspace,
                                     size_t workspace_bytes, void* stream);

/*
 * Map composition across two insertions (Eq. 3): r*(p) = r2(r1(p)).
 *
 *   map1      int32 [rows0]: stage-1 map, local to image b of offsets0
 *   offsets0  int64 [batch + 1]: original images (grid rows)
 *   map2      int32 [rows1]: stage-2 map, local to image b of offsets1
 *   offsets1  int64 [batch + 1]: stage-1 output images (stage-2 inputs)
 *   out_map   int32 [rows0], written for rows < offsets0[batch]
 *   device_status  optional int32 device word (NULL = not reported); an
 *             out-of-range map1 entry writes -1 and records
 *             MPM_ERR_DEVICE_CHECK there.
 * out_map may alias map1 (in-place) but not map2.
 */
MPM_API mpm_status mpm_compose_maps(const int32_t* map1, const int64_t* offsets0, int64_t rows0,
                            const int32_t* map2, const int64_t* offsets1, int64_t rows1,
                            int32_t batch, int32_t* out_map, int32_t* device_status,
                            void* stream);

/*
 * Gather reconstruction (Eq. 4): out[g0_b + p] = merged[m0_b + map[g0_b + p]],
 * a pure copy that restores the raster order of the original grid.
 *
 *   merged          [merged_rows, dim] merged tokens (dtype)
 *   merged_offsets  int64 [batch + 1]: images of `merged`
 *   map             int32 [grid_rows]: composed map, local per image
 *   grid_offsets    int64 [batch + 1]: images of the original grid
 *   out             [grid_rows, dim] (dtype), written for rows < grid_offsets[batch]
 *   device_status   optional int32 device word; an out-of-range map entry
 *                   zeroes that output row and records MPM_ERR_DEVICE_CHECK.
 * out must not overlap merged (MPM_ERR_ALIASING).
 */
MPM_API mpm_status mpm_unmerge_gather(const void* merged, const int64_t* merged_offsets,
                              int64_t merged_rows, const int32_t* map,
                              const int64_t* grid_offsets, int64_t grid_rows, int32_t batch,
                              int32_t dim, mpm_dtype dtype, void* out,
                              int32_t* device_status, void* stream);

/*
 * Composition and gather in one pass (Eq. 3 then Eq. 4), for two
 * insertions: for every grid row p of image b,
 *   r*(p) = map2[offsets1_b + map1[p]]   and   out[p] = merged[m_b + r*(p)].
 * The result equals mpm_compose_maps followed by mpm_unmerge_gather, without
 * the separate pass over the composed map.
 *
 *   merged          [merged_rows, dim] stage-2 tokens (dtype); merged_offsets
 *                   int64 [batch + 1] their images
 *   map1, offsets0  int32 [rows0] stage-1 map and int64 [batch + 1] grid images
 *   map2, offsets1  int32 [rows1] stage-2 map and int64 [batch + 1] stage-1 images
 *   out             [rows0, dim] (dtype), written for rows < offsets0[batch]
 *   out_map         optional int32 [rows0]: receives r* (may alias map1, not
 *                   map2); NULL when the composed map is not wanted
 *   device_status   optional int32 device word; an out-of-range entry of either
 *                   map zeroes that output row, writes -1 to out_map there and
 *                   records MPM_ERR_DEVICE_CHECK.
 * out must not overlap merged (MPM_ERR_ALIASING).
 */
MPM_API mpm_status mpm_compose_gather(const void* merged, const int64_t* merged_offsets,
                              int64_t merged_rows, const int32_t* map1, const int64_t* offsets0,
                              int64_t rows0, const int32_t* map2, const int64_t* offsets1,
                              int64_t rows1, int32_t batch, int32_t dim, mpm_dtype dtype,
                              void* out, int32_t* out_map, int32_t* device_status, void* stream);

/*
 * Padded batch for dense-attention consumers.  Section 4 (Analyses) batches
 * images by padding each to the batch's longest merged sequence; a key mask
 * keeps the padding out of attention.  The paper prints no routine for this
 * step; the definition is:
 *   out[b, t]     = tokens[offsets[b] + t]  for t < min(N_b, max_len), else a zero row
 *   out_mask[b,t] = 1 for the copied rows, 0 for padding
 * with N_b = offsets[b+1] - offsets[b].
 *
 *   tokens     [rows, dim] packed (dtype), offsets int64 [batch + 1] on the device
 *   max_len    L >= 0, the padded length (e.g. the largest N_b, or the input
 *              N as a bound the host knows without reading offsets)
 *   out        [batch, L, dim] (dtype), 16-byte aligned, must not overlap tokens
 *   out_mask   optional uint8 [batch, L]
 *   out_stats  optional int64 [3]: min, max and total of N_b over the batch
 *   device_status  optional int32 device word: an image longer than L is cut
 *              to its first L rows and reported as MPM_ERR_DEVICE_CHECK
 *              (detail = image index).
 * All outputs are written on `stream`; nothing is read back to the host.
 */
MPM_API mpm_status mpm_pad_batch(const void* tokens, const int64_t* offsets, int32_t batch, int64_t rows,
                                 int32_t dim, mpm_dtype dtype, int64_t max_len, void* out,
                                 uint8_t* out_mask, int64_t* out_stats, int32_t* device_status,
                                 void* stream);

/*
 * Inverse of mpm_pad_batch: out[offsets[b] + t] = padded[b, t] for
 * t < N_b (N_b <= max_len), the packed layout the merge entry points take.
 *
 *   padded     [batch, max_len, dim] (dtype)
 *   offsets    int64 [batch + 1]: the packed images; rows = capacity of out
 *   out        [rows, dim] (dtype), written for rows < offsets[batch]; must
 *              not overlap padded
 *   device_status  optional: rows of an image longer than max_len are left
 *              untouched and reported as MPM_ERR_DEVICE_CHECK (detail = image
 *              index).
 */
MPM_API mpm_status mpm_unpad_batch(const void* padded, int32_t batch, int64_t max_len, int32_t dim,
                                   mpm_dtype dtype, const int64_t* offsets, int64_t rows, void* out,
                                   int32_t* device_status, void* stream);

/*
 * Nearest neighbours only (Eq. 1 and Algorithm 1 step 3), for testing and
 * diagnostics.  out_nn int32 [rows]: local index b(i) (-1 for a token alone
 * in its image); out_score float [rows] (may be NULL): the cosine S_{i,b(i)}
 * as computed in fp32.  `algo` selects the kernel (MPM_NN_TCGEN05 and
 * MPM_NN_TCGEN05_SYM require bf16).  Same workspace as mpm_merge.
 */
MPM_API mpm_status mpm_nearest_neighbors(const void* tokens, const int64_t* offsets, int32_t batch,
                                 int64_t rows, int32_t dim, mpm_dtype dtype,
                                 mpm_nn_algo algo, int32_t* out_nn, float* out_score,
                                 void* workspace, size_t workspace_bytes, void* stream);

/*
 * mpm_nearest_neighbors restricted to chunks, as in mpm_merge_chunked (test
 * and diagnostics hook).  `algo` must be MPM_NN_AUTO, MPM_NN_TCGEN05_PAIR or
 * MPM_NN_SIMT when chunk > 0; b(i) = -1 for a token alone in its chunk.
 */
MPM_API mpm_status mpm_nearest_neighbors_chunked(const void* tokens, const int64_t* offsets, int32_t batch,
                                                 int64_t rows, int32_t dim, mpm_dtype dtype, mpm_nn_algo algo,
                                                 int64_t chunk, int32_t* out_nn, float* out_score,
                                                 void* workspace, size_t workspace_bytes, void* stream);

/*
 * Copies the device status word of a merge workspace into *host_code
 * (synchronous on `stream`) and clears it.  Returns MPM_OK when the copy
 * worked; *host_code is then MPM_OK or the first device error.
 */
MPM_API mpm_status mpm_get_device_status(void* workspace, int32_t* host_code, void* stream);

/*
 * Self-test of the device timeout path (the paper has no counterpart).
 * Launches one block whose threads wait on an mbarrier that nothing ever
 * completes, with the bounded wait (wall-time limit plus a probe cap) that
 * the tensor-core kernels use on their pipeline barriers.  After limit_us
 * microseconds the kernel records MPM_ERR_DEVICE_TIMEOUT in
 * device_status[0] (detail 99 in device_status[1], first error wins, as in
 * every MPM kernel) and returns; the CUDA context stays usable.
 *   device_status  device int32[2], caller-owned, zeroed by the caller
 *   limit_us       1 .. 10,000,000 (else MPM_ERR_INVALID_ARG)
 * Asynchronous on `stream`.
 */
MPM_API mpm_status mpm_selftest_wait_timeout(int32_t* device_status, uint32_t limit_us, void* stream);

/*
 * Device timeline of the merge, compose and gather kernels (the paper has no
 * counterpart).  Only a library built with tracing (build(trace=True), which
 * writes libmpm_trace.so) records it; the ordinary library returns
 * MPM_ERR_UNSUPPORTED from both calls.
 *
 * For each kernel kind, the traced kernels keep three readings of the GPU
 * global timer (ns):
 *   [0] the earliest block start;
 *   [1] the earliest moment a block passed its wait for the previous
 *       kernel in the stream;
 *   [2] the latest moment one of its warps finished.
 * A kind that did not run since the last reset reads UINT64_MAX in [0] and
 * [1] and 0 in [2].  Launches of the same kind since the reset are folded
 * together, so reset between the launches you want to tell apart.
 *
 * mpm_trace_read copies MPM_TRACE_KINDS x 3 uint64 values into `out`, a
 * host array.  It is synchronous: call it after the traced work finished.
 * mpm_trace_reset is synchronous too.
 */
typedef enum {
  MPM_TRACE_PREP = 0,
  MPM_TRACE_AFFINITY = 1,
  MPM_TRACE_MUTUAL = 2,
  MPM_TRACE_PAIR_AVERAGE = 3,
  MPM_TRACE_GATHER = 4,
  MPM_TRACE_COMPOSE = 5,
  MPM_TRACE_KINDS = 6
} mpm_trace_kind;
MPM_API mpm_status mpm_trace_read(uint64_t* out);
MPM_API mpm_status mpm_trace_reset(void);

#ifdef __cplusplus
}
#endif

#endif /* MPM_H */
