// Host side of the MPM C ABI: argument validation, workspace carving and
// the launch sequence of each entry point.  No allocation happens here:
// every buffer, including the scratch workspace, belongs to the caller.
#include <cuda_runtime.h>
#include <stdint.h>

#include <nvtx3/nvToolsExt.h>

#include <atomic>

#include "mpm.h"
#include "launch.h"

namespace {

using mpm::Workspace;

// Host-side NVTX range around one launch or one entry point (a profiler
// can select an MPM stage by name; without a tool attached a range costs a
// pointer check).
struct Range {
  explicit Range(const char* name) { nvtxRangePushA(name); }
  ~Range() { nvtxRangePop(); }
  Range(const Range&) = delete;
  Range& operator=(const Range&) = delete;
};

constexpr size_t kAlign = 256;
// Chunks of the chunked similarity are whole tiles of the SM-pair kernel.
constexpr int64_t kChunkQuantum = 256;

size_t round_up(size_t v) { return (v + kAlign - 1) / kAlign * kAlign; }

int elem_size(mpm_dtype dt) { return dt == MPM_BF16 ? 2 : 4; }

bool valid_dtype(mpm_dtype dt) { return dt == MPM_F32 || dt == MPM_BF16; }

struct Layout {
  size_t status, soff, plan, count, inv_norm, keys, reps, split_hi, split_lo, total;
};

// split_elems: rows * dim for fp32 tokens (the tf32 high / low copies), 0 for bf16.
Layout layout(int64_t rows, int32_t batch, size_t split_elems) {
  Layout l{};
  size_t off = 0;
  l.status = off;
  off += round_up(sizeof(int32_t) * mpm::kStatusWords);
  l.soff = off;
  off += round_up(sizeof(int64_t) * (static_cast<size_t>(batch) + 1));
  l.plan = off;
  off += round_up(sizeof(int64_t) * (static_cast<size_t>(batch) + 1));
  l.count = off;
  off += round_up(sizeof(int32_t) * static_cast<size_t>(batch));
  l.inv_norm = off;
  off += round_up(sizeof(float) * static_cast<size_t>(rows));
  l.keys = off;
  off += round_up(sizeof(unsigned long long) * static_cast<size_t>(rows));
  l.reps = off;
  off += round_up(sizeof(int2) * static_cast<size_t>(rows));
  l.split_hi = off;
  off += round_up(sizeof(float) * split_elems);
  l.split_lo = off;
  off += round_up(sizeof(float) * split_elems);
  l.total = off;
  return l;
}

size_t split_elems(int64_t rows, int32_t dim, mpm_dtype dtype) {
  return dtype == MPM_F32 ? static_cast<size_t>(rows) * static_cast<size_t>(dim) : 0;
}

Workspace carve(void* base, int64_t rows, int32_t batch, size_t split) {
  const Layout l = layout(rows, batch, split);
  uint8_t* p = static_cast<uint8_t*>(base);
  Workspace ws;
  ws.status = reinterpret_cast<int32_t*>(p + l.status);
  ws.soff = reinterpret_cast<int64_t*>(p + l.soff);
  ws.plan = reinterpret_cast<int64_t*>(p + l.plan);
  ws.count = reinterpret_cast<int32_t*>(p + l.count);
  ws.inv_norm = reinterpret_cast<float*>(p + l.inv_norm);
  ws.keys = reinterpret_cast<unsigned long long*>(p + l.keys);
  ws.reps = reinterpret_cast<int2*>(p + l.reps);
  ws.split_hi = split > 0 ? reinterpret_cast<float*>(p + l.split_hi) : nullptr;
  ws.split_lo = split > 0 ? reinterpret_cast<float*>(p + l.split_lo) : nullptr;
  return ws;
}

bool sizes_ok(int64_t rows, int32_t batch) {
  return batch >= 1 && rows >= 0 && rows <= INT32_MAX;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

bool overlap(const void* a, size_t an, const void* b, size_t bn) {
  const uintptr_t a0 = reinterpret_cast<uintptr_t>(a), b0 = reinterpret_cast<uintptr_t>(b);
  return an > 0 && bn > 0 && a0 < b0 + bn && b0 < a0 + an;
}

// SM count of the current device (cached per device).
int num_sms() {
  static std::atomic<int> cache[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  const int slot = dev & 63;
  int v = cache[slot].load();
  if (v > 0) return v;
  if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v <= 0) return 0;
  cache[slot].store(v);
  return v;
}

mpm_status cuda_status(cudaError_t e) { return e == cudaSuccess ? MPM_OK : MPM_ERR_CUDA; }

// Shared validation of the token-matrix arguments.
mpm_status check_tokens(const void* tokens, int64_t rows, int32_t dim, mpm_dtype dtype) {
  if (!valid_dtype(dtype) || dim < 1) return MPM_ERR_INVALID_ARG;
  if (dim > MPM_MAX_DIM) return MPM_ERR_UNSUPPORTED;
  if (tokens == nullptr && rows > 0) return MPM_ERR_INVALID_ARG;
  if (!aligned16(tokens) || (static_cast<int64_t>(dim) * elem_size(dtype)) % 16 != 0) return MPM_ERR_ALIGNMENT;
  return MPM_OK;
}

// Kernel used when the caller does not choose one: the SM-pair tensor-core
// kernel, with bf16 products for bf16 tokens and three tf32 products (high
// and low parts, about fp32 accuracy) for fp32 tokens.
mpm_nn_algo default_algo(mpm_dtype) { return MPM_NN_TCGEN05_PAIR; }

// The workspace's tf32 split copies are filled only for the fp32 tensor-core path.
Workspace for_algo(Workspace ws, mpm_nn_algo algo, mpm_dtype dtype) {
  if (!(algo == MPM_NN_TCGEN05_PAIR && dtype == MPM_F32)) ws.split_hi = ws.split_lo = nullptr;
  return ws;
}

bool is_tensor_core(mpm_nn_algo a) {
  return a == MPM_NN_TCGEN05 || a == MPM_NN_TCGEN05_SYM || a == MPM_NN_TCGEN05_PAIR;
}

mpm::AffinityTile tile_of(mpm_nn_algo a, int64_t chunk) {
  mpm::AffinityTile t = a == MPM_NN_TCGEN05_PAIR                              ? mpm::pair_tile()
                        : (a == MPM_NN_TCGEN05 || a == MPM_NN_TCGEN05_SYM) ? mpm::tc_tile(a == MPM_NN_TCGEN05_SYM)
                                                                            : mpm::simt_tile();
  t.chunk = chunk;
  return t;
}

// Chunked similarity runs on the SM-pair tensor-core kernel and the fp32
// kernel, with chunks of whole 256-token tiles.
mpm_status check_chunk(mpm_nn_algo algo, int64_t chunk) {
  if (chunk < 0) return MPM_ERR_INVALID_ARG;
  if (chunk == 0) return MPM_OK;
  if (chunk % kChunkQuantum != 0) return MPM_ERR_UNSUPPORTED;
  if (algo != MPM_NN_TCGEN05_PAIR && algo != MPM_NN_SIMT) return MPM_ERR_UNSUPPORTED;
  return MPM_OK;
}

cudaError_t launch_affinity(mpm_nn_algo a, const void* tokens, int batch, int64_t rows, int dim, bool bf16,
                            int64_t chunk, const Workspace& ws, int sms, cudaStream_t s) {
  if (a == MPM_NN_TCGEN05_PAIR) return mpm::launch_affinity_pair(tokens, batch, rows, dim, !bf16, chunk, ws, sms, s);
  if (a == MPM_NN_TCGEN05 || a == MPM_NN_TCGEN05_SYM)
    return mpm::launch_affinity_tc(tokens, batch, rows, dim, a == MPM_NN_TCGEN05_SYM, ws, sms, s);
  return mpm::launch_affinity_simt(tokens, batch, dim, bf16, chunk, ws, sms, s);
}

// The affinity + arg max stage shared by the merge and nearest-neighbour
// entry points.
mpm_status run_affinity(const void* tokens, const int64_t* offsets, int32_t batch, int64_t rows, int32_t dim,
                        mpm_dtype dtype, mpm_nn_algo algo, int64_t chunk, const Workspace& ws_all,
                        cudaStream_t stream) {
  const bool bf16 = dtype == MPM_BF16;
  if (algo == MPM_NN_AUTO) algo = default_algo(dtype);
  const bool tc = is_tensor_core(algo);
  if (algo != MPM_NN_SIMT && !tc) return MPM_ERR_INVALID_ARG;
  if (tc && !bf16 && algo != MPM_NN_TCGEN05_PAIR) return MPM_ERR_UNSUPPORTED;
  const Workspace ws = for_algo(ws_all, algo, dtype);
  const mpm_status cs = check_chunk(algo, chunk);
  if (cs != MPM_OK) return cs;
  if (tc && !mpm::tc_available()) return MPM_ERR_UNSUPPORTED;
  const int sms = num_sms();
  if (sms <= 0) return MPM_ERR_CUDA;
  cudaError_t e = mpm::launch_prep(tokens, offsets, batch, rows, dim, bf16, tile_of(algo, chunk), ws, sms, stream);
  if (e != cudaSuccess) return MPM_ERR_CUDA;
  if (rows == 0) return MPM_OK;  // every image is empty: nothing to compare
  return cuda_status(launch_affinity(algo, tokens, batch, rows, dim, bf16, chunk, ws, sms, stream));
}

mpm_status nearest_neighbors_impl(const void* tokens, const int64_t* offsets, int32_t batch, int64_t rows,
                                  int32_t dim, mpm_dtype dtype, mpm_nn_algo algo, int64_t chunk, int32_t* out_nn,
                                  float* out_score, void* workspace, size_t workspace_bytes, void* stream) {
  if (!sizes_ok(rows, batch) || offsets == nullptr || out_nn == nullptr) return MPM_ERR_INVALID_ARG;
  mpm_status st = check_tokens(tokens, rows, dim, dtype);
  if (st != MPM_OK) return st;
  if (workspace == nullptr || (reinterpret_cast<uintptr_t>(workspace) % kAlign) != 0 ||
      workspace_bytes < layout(rows, batch, split_elems(rows, dim, dtype)).total)
    return MPM_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const Workspace ws = carve(workspace, rows, batch, split_elems(rows, dim, dtype));
  st = run_affinity(tokens, offsets, batch, rows, dim, dtype, algo, chunk, ws, s);
  if (st != MPM_OK) return st;
  return cuda_status(mpm::launch_decode_nn(batch, rows, ws, out_nn, out_score, num_sms(), s));
}

mpm_status merge_impl(const void* tokens, const int64_t* offsets, int32_t batch, int64_t rows, int32_t dim,
                      mpm_dtype dtype, int64_t chunk, void* out_tokens, int64_t* out_offsets, int32_t* out_map,
                      void* workspace, size_t workspace_bytes, void* stream, void* const* stage_events) {
  if (!sizes_ok(rows, batch) || offsets == nullptr || out_offsets == nullptr) return MPM_ERR_INVALID_ARG;
  if (rows > 0 && (out_tokens == nullptr || out_map == nullptr)) return MPM_ERR_INVALID_ARG;
  mpm_status st = check_tokens(tokens, rows, dim, dtype);
  if (st != MPM_OK) return st;
  if (!aligned16(out_tokens)) return MPM_ERR_ALIGNMENT;
  const size_t bytes = static_cast<size_t>(rows) * dim * elem_size(dtype);
  if (overlap(tokens, bytes, out_tokens, bytes)) return MPM_ERR_ALIASING;
  if (workspace == nullptr || (reinterpret_cast<uintptr_t>(workspace) % kAlign) != 0 ||
      workspace_bytes < layout(rows, batch, split_elems(rows, dim, dtype)).total)
    return MPM_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const bool bf16 = dtype == MPM_BF16;
  const mpm_nn_algo algo = default_algo(dtype);
  const Workspace ws = for_algo(carve(workspace, rows, batch, split_elems(rows, dim, dtype)), algo, dtype);
  st = check_chunk(algo, chunk);
  if (st != MPM_OK) return st;
  if (is_tensor_core(algo) && !mpm::tc_available()) return MPM_ERR_UNSUPPORTED;
  const int sms = num_sms();
  if (sms <= 0) return MPM_ERR_CUDA;
  // Records stage_events[idx] (if profiling) on the launch stream.
  auto mark = [&](int idx) -> bool {
    if (stage_events == nullptr) return true;
    return cudaEventRecord(static_cast<cudaEvent_t>(stage_events[idx]), s) == cudaSuccess;
  };
  const mpm::AffinityTile tile = tile_of(algo, chunk);
  cudaError_t e = cudaSuccess;
  const Range whole("mpm_merge");
  if (!mark(0)) return MPM_ERR_CUDA;
  {
    const Range r("mpm.prep");
    e = mpm::launch_prep(tokens, offsets, batch, rows, dim, bf16, tile, ws, sms, s);
  }
  if (e != cudaSuccess || !mark(1) || !mark(2)) return MPM_ERR_CUDA;
  if (rows > 0) {
    const Range r("mpm.affinity");
    e = launch_affinity(algo, tokens, batch, rows, dim, bf16, chunk, ws, sms, s);
    if (e != cudaSuccess) return MPM_ERR_CUDA;
  }
  if (!mark(3) || !mark(4)) return MPM_ERR_CUDA;
  {
    const Range r("mpm.mutual_scan");
    e = mpm::launch_mutual_compact(batch, chunk, ws, out_map, out_offsets, s);
  }
  if (e != cudaSuccess || !mark(5) || !mark(6)) return MPM_ERR_CUDA;
  if (rows > 0) {
    const Range r("mpm.pair_average");
    e = mpm::launch_pair_average(tokens, out_tokens, batch, rows, dim, bf16, ws, out_offsets, sms, s);
    if (e != cudaSuccess) return MPM_ERR_CUDA;
  }
  return mark(7) ? MPM_OK : MPM_ERR_CUDA;
}

}  // namespace

extern "C" {

int32_t mpm_abi_version(void) { return MPM_ABI_VERSION; }

const char* mpm_status_string(mpm_status status) {
  switch (status) {
    case MPM_OK: return "ok";
    case MPM_ERR_INVALID_ARG: return "invalid argument";
    case MPM_ERR_UNSUPPORTED: return "unsupported configuration";
    case MPM_ERR_ALIGNMENT: return "token buffer or row size not 16-byte aligned";
    case MPM_ERR_WORKSPACE: return "workspace missing, too small or misaligned";
    case MPM_ERR_CUDA: return "CUDA error";
    case MPM_ERR_DEVICE_CHECK: return "device check failed (offsets or map out of range)";
    case MPM_ERR_DEVICE_TIMEOUT: return "device wait timed out";
    case MPM_ERR_ALIASING: return "output overlaps input";
  }
  return "unknown status";
}

size_t mpm_merge_workspace_size(int64_t rows, int32_t batch, int32_t dim, mpm_dtype dtype) {
  if (!sizes_ok(rows, batch) || dim < 1 || !valid_dtype(dtype)) return 0;
  return layout(rows, batch, split_elems(rows, dim, dtype)).total;
}

mpm_status mpm_nearest_neighbors(const void* tokens, const int64_t* offsets, int32_t batch, int64_t rows,
                                 int32_t dim, mpm_dtype dtype, mpm_nn_algo algo, int32_t* out_nn,
                                 float* out_score, void* workspace, size_t workspace_bytes, void* stream) {
  return nearest_neighbors_impl(tokens, offsets, batch, rows, dim, dtype, algo, 0, out_nn, out_score, workspace,
                                workspace_bytes, stream);
}

mpm_status mpm_nearest_neighbors_chunked(const void* tokens, const int64_t* offsets, int32_t batch, int64_t rows,
                                         int32_t dim, mpm_dtype dtype, mpm_nn_algo algo, int64_t chunk,
                                         int32_t* out_nn, float* out_score, void* workspace,
                                         size_t workspace_bytes, void* stream) {
  return nearest_neighbors_impl(tokens, offsets, batch, rows, dim, dtype, algo, chunk, out_nn, out_score,
                                workspace, workspace_bytes, stream);
}

mpm_status mpm_merge_timed(const void* tokens, const int64_t* offsets, int32_t batch, int64_t rows,
                           int32_t dim, mpm_dtype dtype, void* out_tokens, int64_t* out_offsets,
                           int32_t* out_map, void* workspace, size_t workspace_bytes, void* stream,
                           void* const* stage_events) {
  return merge_impl(tokens, offsets, batch, rows, dim, dtype, 0, out_tokens, out_offsets, out_map, workspace,
                    workspace_bytes, stream, stage_events);
}

mpm_status mpm_merge(const void* tokens, const int64_t* offsets, int32_t batch, int64_t rows, int32_t dim,
                     mpm_dtype dtype, void* out_tokens, int64_t* out_offsets, int32_t* out_map, void* workspace,
                     size_t workspace_bytes, void* stream) {
  return merge_impl(tokens, offsets, batch, rows, dim, dtype, 0, out_tokens, out_offsets, out_map, workspace,
                    workspace_bytes, stream, nullptr);
}

mpm_status mpm_merge_chunked(const void* tokens, const int64_t* offsets, int32_t batch, int64_t rows, int32_t dim,
                             mpm_dtype dtype, int64_t chunk, void* out_tokens, int64_t* out_offsets,
                             int32_t* out_map, void* workspace, size_t workspace_bytes, void* stream) {
  return merge_impl(tokens, offsets, batch, rows, dim, dtype, chunk, out_tokens, out_offsets, out_map, workspace,
                    workspace_bytes, stream, nullptr);
}

mpm_status mpm_compose_maps(const int32_t* map1, const int64_t* offsets0, int64_t rows0, const int32_t* map2,
                            const int64_t* offsets1, int64_t rows1, int32_t batch, int32_t* out_map,
                            int32_t* device_status, void* stream) {
  const Range whole("mpm_compose_maps");
  if (!sizes_ok(rows0, batch) || !sizes_ok(rows1, batch) || offsets0 == nullptr || offsets1 == nullptr)
    return MPM_ERR_INVALID_ARG;
  if (rows0 == 0) return MPM_OK;
  if (map1 == nullptr || out_map == nullptr || (map2 == nullptr && rows1 > 0)) return MPM_ERR_INVALID_ARG;
  if (overlap(out_map, sizeof(int32_t) * rows0, map2, sizeof(int32_t) * rows1)) return MPM_ERR_ALIASING;
  const int sms = num_sms();
  if (sms <= 0) return MPM_ERR_CUDA;
  return cuda_status(mpm::launch_compose(map1, offsets0, rows0, map2, offsets1, rows1, batch, out_map,
                                         device_status, sms, static_cast<cudaStream_t>(stream)));
}

mpm_status mpm_unmerge_gather(const void* merged, const int64_t* merged_offsets, int64_t merged_rows,
                              const int32_t* map, const int64_t* grid_offsets, int64_t grid_rows, int32_t batch,
                              int32_t dim, mpm_dtype dtype, void* out, int32_t* device_status, void* stream) {
  const Range whole("mpm_unmerge_gather");
  if (!sizes_ok(merged_rows, batch) || !sizes_ok(grid_rows, batch) || merged_offsets == nullptr ||
      grid_offsets == nullptr)
    return MPM_ERR_INVALID_ARG;
  mpm_status st = check_tokens(merged, merged_rows, dim, dtype);
  if (st != MPM_OK) return st;
  if (grid_rows == 0) return MPM_OK;
  if (map == nullptr || out == nullptr) return MPM_ERR_INVALID_ARG;
  if (!aligned16(out)) return MPM_ERR_ALIGNMENT;
  const size_t row_bytes = static_cast<size_t>(dim) * elem_size(dtype);
  if (overlap(merged, row_bytes * merged_rows, out, row_bytes * grid_rows)) return MPM_ERR_ALIASING;
  const int sms = num_sms();
  if (sms <= 0) return MPM_ERR_CUDA;
  return cuda_status(mpm::launch_gather(merged, merged_offsets, merged_rows, map, grid_offsets, grid_rows, batch,
                                        dim, dtype == MPM_BF16, out, device_status, sms,
                                        static_cast<cudaStream_t>(stream)));
}

mpm_status mpm_compose_gather(const void* merged, const int64_t* merged_offsets, int64_t merged_rows,
                              const int32_t* map1, const int64_t* offsets0, int64_t rows0, const int32_t* map2,
                              const int64_t* offsets1, int64_t rows1, int32_t batch, int32_t dim, mpm_dtype dtype,
                              void* out, int32_t* out_map, int32_t* device_status, void* stream) {
  const Range whole("mpm_compose_gather");
  if (!sizes_ok(merged_rows, batch) || !sizes_ok(rows0, batch) || !sizes_ok(rows1, batch) ||
      merged_offsets == nullptr || offsets0 == nullptr || offsets1 == nullptr)
    return MPM_ERR_INVALID_ARG;
  mpm_status st = check_tokens(merged, merged_rows, dim, dtype);
  if (st != MPM_OK) return st;
  if (rows0 == 0) return MPM_OK;
  if (map1 == nullptr || out == nullptr || (map2 == nullptr && rows1 > 0)) return MPM_ERR_INVALID_ARG;
  if (!aligned16(out)) return MPM_ERR_ALIGNMENT;
  const size_t row_bytes = static_cast<size_t>(dim) * elem_size(dtype);
  if (overlap(merged, row_bytes * merged_rows, out, row_bytes * rows0)) return MPM_ERR_ALIASING;
  if (out_map != nullptr && overlap(out_map, sizeof(int32_t) * rows0, map2, sizeof(int32_t) * rows1))
    return MPM_ERR_ALIASING;
  const int sms = num_sms();
  if (sms <= 0) return MPM_ERR_CUDA;
  return cuda_status(mpm::launch_compose_gather(merged, merged_offsets, merged_rows, map1, offsets0, rows0, map2,
                                                offsets1, rows1, batch, dim, dtype == MPM_BF16, out, out_map,
                                                device_status, sms, static_cast<cudaStream_t>(stream)));
}

mpm_status mpm_pad_batch(const void* tokens, const int64_t* offsets, int32_t batch, int64_t rows, int32_t dim,
                         mpm_dtype dtype, int64_t max_len, void* out, uint8_t* out_mask, int64_t* out_stats,
                         int32_t* device_status, void* stream) {
  if (!sizes_ok(rows, batch) || offsets == nullptr || max_len < 0) return MPM_ERR_INVALID_ARG;
  mpm_status st = check_tokens(tokens, rows, dim, dtype);
  if (st != MPM_OK) return st;
  if (batch == 0) return MPM_OK;
  if (max_len > 0 && (out == nullptr || !aligned16(out))) return out == nullptr ? MPM_ERR_INVALID_ARG : MPM_ERR_ALIGNMENT;
  const size_t row_bytes = static_cast<size_t>(dim) * elem_size(dtype);
  const int64_t out_rows = static_cast<int64_t>(batch) * max_len;
  if (max_len > 0 && overlap(tokens, row_bytes * rows, out, row_bytes * out_rows)) return MPM_ERR_ALIASING;
  const int sms = num_sms();
  if (sms <= 0) return MPM_ERR_CUDA;
  return cuda_status(mpm::launch_pad(tokens, offsets, batch, rows, max_len, dim, dtype == MPM_BF16, out, out_mask,
                                     out_stats, device_status, sms, static_cast<cudaStream_t>(stream)));
}

mpm_status mpm_unpad_batch(const void* padded, int32_t batch, int64_t max_len, int32_t dim, mpm_dtype dtype,
                           const int64_t* offsets, int64_t rows, void* out, int32_t* device_status, void* stream) {
  if (!sizes_ok(rows, batch) || offsets == nullptr || max_len < 0) return MPM_ERR_INVALID_ARG;
  const int64_t in_rows = static_cast<int64_t>(batch) * max_len;
  mpm_status st = check_tokens(padded, in_rows, dim, dtype);
  if (st != MPM_OK) return st;
  if (rows == 0 || batch == 0) return MPM_OK;
  if (out == nullptr) return MPM_ERR_INVALID_ARG;
  if (!aligned16(out)) return MPM_ERR_ALIGNMENT;
  const size_t row_bytes = static_cast<size_t>(dim) * elem_size(dtype);
  if (overlap(padded, row_bytes * in_rows, out, row_bytes * rows)) return MPM_ERR_ALIASING;
  const int sms = num_sms();
  if (sms <= 0) return MPM_ERR_CUDA;
  return cuda_status(mpm::launch_unpad(padded, batch, max_len, offsets, rows, dim, dtype == MPM_BF16, out,
                                       device_status, sms, static_cast<cudaStream_t>(stream)));
}

mpm_status mpm_trace_read(uint64_t* out) {
#ifdef MPM_TRACE
  if (out == nullptr) return MPM_ERR_INVALID_ARG;
  unsigned long long a[MPM_TRACE_KINDS][3], b[MPM_TRACE_KINDS][3];
  if (cudaDeviceSynchronize() != cudaSuccess || mpm::trace_copy_hbm(&a[0][0], false) != cudaSuccess ||
      mpm::trace_copy_pair(&b[0][0], false) != cudaSuccess)
    return MPM_ERR_CUDA;
  for (int k = 0; k < MPM_TRACE_KINDS; ++k) {
    out[3 * k + 0] = a[k][0] < b[k][0] ? a[k][0] : b[k][0];
    out[3 * k + 1] = a[k][1] < b[k][1] ? a[k][1] : b[k][1];
    out[3 * k + 2] = a[k][2] > b[k][2] ? a[k][2] : b[k][2];
  }
  return MPM_OK;
#else
  (void)out;
  return MPM_ERR_UNSUPPORTED;
#endif
}

mpm_status mpm_trace_reset(void) {
#ifdef MPM_TRACE
  if (cudaDeviceSynchronize() != cudaSuccess || mpm::trace_copy_hbm(nullptr, true) != cudaSuccess ||
      mpm::trace_copy_pair(nullptr, true) != cudaSuccess)
    return MPM_ERR_CUDA;
  return MPM_OK;
#else
  return MPM_ERR_UNSUPPORTED;
#endif
}

mpm_status mpm_get_device_status(void* workspace, int32_t* host_code, void* stream) {
  if (workspace == nullptr || host_code == nullptr) return MPM_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int32_t* status = static_cast<int32_t*>(workspace);  // the status word leads the workspace
  int32_t word[2] = {0, 0};
  if (cudaMemcpyAsync(word, status, sizeof(word), cudaMemcpyDeviceToHost, s) != cudaSuccess) return MPM_ERR_CUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return MPM_ERR_CUDA;
  if (cudaMemsetAsync(status, 0, sizeof(word), s) != cudaSuccess) return MPM_ERR_CUDA;
  *host_code = word[0];
  return MPM_OK;
}

}  // extern "C"
