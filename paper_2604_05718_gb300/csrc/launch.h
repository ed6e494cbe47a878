// Internal launchers of the MPM kernels (not part of the public ABI).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace mpm {

// Status word layout in the workspace (int32[4]):
//   [0] first device error code, [1] its detail, [2] completion counter of
//   the per-image scan kernel, [3] spare.
constexpr int kStatusWords = 4;

// Device scratch carved from the caller's workspace.
struct Workspace {
  int32_t* status;            // int32[4]
  int64_t* soff;              // int64[batch + 1] sanitised offsets
  int64_t* plan;              // int64[batch + 1] prefix of affinity work items
  int32_t* count;             // int32[batch] merged tokens per image (N'_b)
  float* inv_norm;            // float[rows] 1 / max(|x_i|, 1e-12)
  unsigned long long* keys;   // u64[rows] packed (score, lowest j) arg-max keys
  int2* reps;                 // int2[rows] (representative, partner or -1), per image
  // fp32 tokens only: x split into a tf32 high part and the fp32 remainder
  // (float[rows * dim] each), for the three-product tf32 tensor-core path.
  // Null for bf16.
  float* split_hi;
  float* split_lo;
};

// Tile of one affinity work item: rows x columns of the cosine matrix, and
// which tiles of an image's N x N matrix are computed:
//   kDense        all of them;
//   kSymmetric    those holding a rows-block at or above the diagonal
//                 (cols == 2 * rows);
//   kUpperSquare  the square tiles on or above the diagonal (rows == cols).
struct AffinityTile {
  enum Mode : int { kDense = 0, kSymmetric = 1, kUpperSquare = 2 };
  int rows;
  int cols;
  int mode;
  // Chunked similarity: tokens are compared only within runs of `chunk`
  // consecutive tokens of their image (0 = the whole image).
  int64_t chunk = 0;
};

// Inverse row norms, key reset, offsets sanitisation and the work plan.
cudaError_t launch_prep(const void* tokens, const int64_t* offsets, int batch, int64_t rows,
                        int dim, bool bf16, AffinityTile tile, const Workspace& ws, int num_sms,
                        cudaStream_t stream);

// CUDA-core affinity + arg max (any dtype).
cudaError_t launch_affinity_simt(const void* tokens, int batch, int dim, bool bf16, int64_t chunk,
                                 const Workspace& ws, int num_sms, cudaStream_t stream);
AffinityTile simt_tile();

// TMA + tcgen05 affinity + arg max (bf16), dense or symmetric tiling.
cudaError_t launch_affinity_tc(const void* tokens, int batch, int64_t rows, int dim, bool symmetric,
                               const Workspace& ws, int num_sms, cudaStream_t stream);
AffinityTile tc_tile(bool symmetric);
bool tc_available();

// Symmetric affinity + arg max on SM pairs (tcgen05.mma.cta_group::2, bf16).
// tf32: fp32 tokens through the three-product tf32 split (ws.split_hi / split_lo).
cudaError_t launch_affinity_pair(const void* tokens, int batch, int64_t rows, int dim, bool tf32, int64_t chunk,
                                 const Workspace& ws, int num_sms, cudaStream_t stream);
AffinityTile pair_tile();

// Mutual check, representative scan, per-image counts, output offsets.
cudaError_t launch_mutual_compact(int batch, int64_t chunk, const Workspace& ws, int32_t* out_map,
                                  int64_t* out_offsets, cudaStream_t stream);

// Pair average + compaction into the packed output.
cudaError_t launch_pair_average(const void* tokens, void* out_tokens, int batch, int64_t rows,
                                int dim, bool bf16, const Workspace& ws,
                                const int64_t* out_offsets, int num_sms, cudaStream_t stream);

// Keys -> nearest neighbour index and cosine.
cudaError_t launch_decode_nn(int batch, int64_t rows, const Workspace& ws, int32_t* out_nn,
                             float* out_score, int num_sms, cudaStream_t stream);

cudaError_t launch_compose(const int32_t* map1, const int64_t* off0, int64_t rows0,
                           const int32_t* map2, const int64_t* off1, int64_t rows1, int batch,
                           int32_t* out, int32_t* status, int num_sms, cudaStream_t stream);

cudaError_t launch_gather(const void* merged, const int64_t* moff, int64_t merged_rows,
                          const int32_t* map, const int64_t* goff, int64_t grid_rows, int batch,
                          int dim, bool bf16, void* out, int32_t* status, int num_sms,
                          cudaStream_t stream);

// Composition (Eq. 3) and gather (Eq. 4) in one pass over the grid rows.
cudaError_t launch_compose_gather(const void* merged, const int64_t* moff, int64_t merged_rows,
                                  const int32_t* map1, const int64_t* off0, int64_t rows0,
                                  const int32_t* map2, const int64_t* off1, int64_t rows1, int batch, int dim,
                                  bool bf16, void* out, int32_t* out_map, int32_t* status, int num_sms,
                                  cudaStream_t stream);

#ifdef MPM_TRACE
// Device timeline tables of kernels_hbm.cu and affinity_pair.cu (MPM_TRACE
// builds): copy out (reset == false) or reset.
cudaError_t trace_copy_hbm(unsigned long long* out, bool reset);
cudaError_t trace_copy_pair(unsigned long long* out, bool reset);
#endif

// Padded batch [batch, max_len, dim] + key mask + N_b statistics, and its
// inverse (kernels_pad.cu).
cudaError_t launch_pad(const void* tokens, const int64_t* offsets, int batch, int64_t rows, int64_t max_len,
                       int dim, bool bf16, void* out, uint8_t* mask, int64_t* stats, int32_t* status, int num_sms,
                       cudaStream_t stream);
cudaError_t launch_unpad(const void* padded, int batch, int64_t max_len, const int64_t* offsets, int64_t rows,
                         int dim, bool bf16, void* out, int32_t* status, int num_sms, cudaStream_t stream);

}  // namespace mpm
