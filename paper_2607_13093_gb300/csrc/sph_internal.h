// Internal interfaces between the C-ABI layer (sph_api.cu) and the kernel
// translation units.  Not part of the public ABI.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>

namespace sph {

enum Epilogue : int {
  EPI_CLOUD = 0,     // +bias, optional unclipped store, clip, row |max|
  EPI_ENDPOINT = 1,  // + code * row_scale (dequantized cloud partial)
  EPI_FUSED = 2,     // endpoint that quantizes the cloud's clipped partials
                     // itself: code = Q(yc), written out as the payload,
                     // then + code * row_scale as EPI_ENDPOINT
};

enum WDtype : int { W_BF16 = 0, W_FP8 = 1 };

// Device-side error bits (OR-ed into the context's status word).
enum : unsigned int {
  ERR_TIMEOUT = 1u,     // a bounded wait gave up
  ERR_BAD_INDEX = 2u,   // reserved for an id outside its range (no kernel checks ids yet)
};

// Kernels launched by this thread (read by the tracing layer).
extern thread_local long long launch_count;

// Launch with programmatic stream serialization: the kernel may start while
// the previous kernel of the stream is still running, and must call
// griddepcontrol.wait (ptx::griddep_wait) before it touches memory that an
// earlier kernel writes or reads.  Every kernel of this library does so.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t st, Args&&... args) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  ++launch_count;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}
// launch_pdl with thread-block clusters of `cluster_x` CTAs along x
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl_cluster(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                               cudaStream_t st, int cluster_x, Args&&... args) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = (unsigned)cluster_x;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  ++launch_count;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// One gathered contraction  acc[r, j] = sum_c h[r, c] * W[ids[j], c]
// followed by an epilogue.  Pointers are device pointers.
struct GatherGemm {
  const float* h;          // [rows, K] fp32, row stride ld_h
  int64_t ld_h;
  int rows;
  const void* W;           // [V, K] bf16 or e4m3, row stride ld_w elements
  int64_t ld_w;
  int w_dtype;             // WDtype
  const float* w_scale;    // [V] (fp8 only)
  int K;
  int64_t V;               // rows of W
  const int32_t* ids;      // [n] sorted ids or nullptr (identity)
  int n;
  int act_bf16;            // round h to bf16 first
  int epilogue;            // Epilogue
  // EPI_CLOUD
  const float* bias;       // [V] or nullptr
  float clip;
  float* partial_out;      // [rows, n] unclipped, or nullptr
  float* Y;                // [rows, n] clipped (cloud) / fused z (endpoint)
  unsigned* rowmax;        // [rows] bits of max |clipped y|, zeroed by caller
  // EPI_ENDPOINT
  const int8_t* codes;     // [rows, n]
  const float* row_scale;  // [rows]
  float inv_tau;           // 1 / temperature (softmax statistics)
  int64_t ldy = 0;         // row stride of Y (z) in elements; 0: n
  // EPI_FUSED: the cloud's clipped partials and row maxima in, the payload out
  const float* yc = nullptr;            // [rows, n] clipped cloud partials
  const unsigned* rowmax_in = nullptr;  // [rows] bits of their row |max|
  int8_t* codes_out = nullptr;          // [rows, n] int8 codes (Eq. 18)
  float* scale_out = nullptr;           // [rows] row scales
  unsigned* status;        // device error word
  long long finish_wait = 1ll << 15;   // split-tile finisher poll (cycles; 0: none)
  bool no_stats = false;   // endpoint: skip the softmax statistics (Gumbel-max draw)
  // cloud GEMV in one launch: the last block to arrive (q_ticket, which it
  // resets) quantizes every row (Eq. 18) into q_codes / q_scale and clears
  // the row maxima for the next call; nullptr: the quantize pass does it
  unsigned* q_ticket = nullptr;
  int8_t* q_codes = nullptr;
  float* q_scale = nullptr;
};

// CUDA-core gathered GEMV (few rows); returns a cudaError_t.
cudaError_t launch_gemv(const GatherGemm& g, int sm_count, cudaStream_t st);
// Largest K the GEMV supports for a given row count.
int gemv_max_k();
// Hidden-state rows one GEMV launch covers (1, 2, 4 or 8).
int gemv_rows_per_launch(int rows, int K);
// Most rows x kept ids the cloud GEMV quantizes in its last block (two
// batches of eight loads a thread; measured: at 25,600 entries the one
// block took longer than a separate quantize pass over the whole grid)
constexpr int64_t kGemvQuantizeMax = 1 << 12;
// Whether the cloud GEMV can quantize in its last block (one launch covers
// the rows, at most kGemvQuantizeMax entries).
inline bool gemv_can_quantize(int64_t rows, int64_t n, int K) {
  return gemv_rows_per_launch((int)rows, K) >= rows && rows * n <= kGemvQuantizeMax;
}

// Tensor-core path (k_tc.cu): sizes, work split and scratch of one call.
struct TcPlan {
  int hilo, RB, BN, Rp, KB, Kp, NT, G, stages, whole_tiles, na, fp8;
  int pair;        // CTA pairs (clusters of two) share each 256-id tile; G counts CTAs
  int tm;          // vocabulary rows per tile: 128 or 256
  int single_acc;  // one TMEM accumulator (256-id tiles over > 128 rows)
  int nseg;        // endpoint statistics: 32-id segments per row, NT * tm / 32
  int epi_stats;   // endpoint: softmax statistics in the epilogue (else a pass over z)
  int rm;          // endpoint on CTA pairs with rows as M (256-row blocks, whole tiles)
  int epi_t;       // endpoint: the epilogue may finish through a shared-memory transpose
                   // (where rows are 2-element aligned; shared memory reserved for it)
  long long T;
  size_t hs_bytes, p_bytes, cnt_bytes, stats_bytes, scratch_bytes, smem_bytes;
  bool ok;
};
// `endpoint` reserves the per-segment softmax statistics; schedule 0/1/2 =
// automatic / whole tiles / stream-K; max_stages 0 = automatic; block_k =
// hidden elements per pipeline stage (64, 128 or 256; 0 = automatic);
// gather = the kept-id subset path (keep_ids given); fp8 = e4m3 weights;
// max_bn = most hidden-state rows per tile (0 = automatic); tile_m =
// vocabulary rows per tile (128, 256 = two M = 128 halves, 0 = automatic);
// pair_mode = CTA pairs on 256-id tiles: 0 never, 1 where the row blocks are
// long enough (bf16 weights), 2 always; max_pairs caps the pairs (0: no cap); rm_mode = the endpoint on
// pairs with rows as M: 0 where the 256-row blocks pad little, 1 always
// (where the call pairs), 2 never.
TcPlan tc_plan(int rows, int n, int K, int act_bf16, int sm_count, int endpoint,
               int schedule, int max_stages, int block_k, int gather, int fp8, int max_bn,
               int tile_m, int pair_mode = 0, int max_pairs = 0, int rm_mode = 0);
// CTA pairs of the pair kernel that can run at once on `device` (0 when the
// query fails): tc_plan's max_pairs.
int tc_pair_max_units(int device);
// Launch the operand split and the tcgen05 kernel; `scratch` holds
// plan.scratch_bytes bytes.  bf16 weights only.
cudaError_t launch_tc(const GatherGemm& g, const TcPlan& plan, void* scratch,
                      long long spin_limit, cudaStream_t st);
// Where a draw finds the fused logits of the ids it visits (the 32 ids of
// the segment it lands in): stored in Z (fp32 [rows, n]), or, with Z null,
// recomputed for just those ids from the endpoint call's own inputs (Eq. 13),
//   z[r, j] = codes[r, j] * row_scale[r] + sum_{c < K} h[r, c] * W[ids[j], c]
// with bf16 W (16-byte aligned rows), fp32 h, fp32 accumulation; codes null:
// the local part alone.
struct ZSource {
  const float* Z = nullptr;
  const float* h = nullptr;
  int64_t ld_h = 0;
  int K = 0;
  const void* W = nullptr;
  int64_t ld_w = 0;
  const int32_t* ids = nullptr;
  const int8_t* codes = nullptr;
  const float* row_scale = nullptr;
};
// One inverse-CDF draw per row after an endpoint launch_tc: from the segment
// statistics its epilogue left in `scratch` (plan.epi_stats), else from a
// statistics pass over the stored z into the same area (a z that is not
// stored needs plan.epi_stats); `cstats` receives the chunk statistics on
// the way (at most rows * (n / 1024 + 2)).
cudaError_t launch_sample_from_stats(const ZSource& zs, int rows, int n,
                                     const TcPlan& plan, const void* scratch,
                                     float2* cstats, const int32_t* ids,
                                     float inv_tau, uint64_t seed, uint64_t offset,
                                     int sm_count, int32_t* tokens, cudaStream_t st,
                                     int greedy = 0);

// codes/row_scale from the clipped partials and their row maxima
cudaError_t launch_quantize(const float* Y, const unsigned* rowmax, int rows,
                            int n, int8_t* codes, float* row_scale,
                            cudaStream_t st);

// Row kernels over fused logits Z (fp32 [rows, n]), k_rows.cu.
// Segment statistics: stats[r * nseg + s] = (max of z over the ids
// 32s..32s+31 of row r, sum of exp((z - max) * inv_tau) over them), nseg =
// seg_count(n); chunk statistics cstats[r * nchunk + c], nchunk =
// chunk_count(nseg), the same pair over the 32 segments 32c..32c+31.
int seg_count(int n);
int chunk_count(int nseg);
cudaError_t launch_seg_stats(const float* Z, int rows, int n, float inv_tau,
                             float2* stats, float2* cstats, int sm_count,
                             cudaStream_t st);
// chunk statistics from segment statistics with nseg segments per row
cudaError_t launch_chunk_stats(const float2* stats, int rows, int nseg,
                               float inv_tau, float2* cstats, int sm_count,
                               cudaStream_t st);
// Gumbel-max draw per row over Z (fp32 [rows, n]): the first index of the
// largest z * inv_tau - log(-log u) with per-(row, index) Philox uniforms.
cudaError_t launch_gumbel(const float* Z, int rows, int n, const int32_t* ids, float inv_tau,
                          uint64_t seed, uint64_t offset, int32_t* tokens, cudaStream_t st);
// One inverse-CDF draw per row from segment statistics alone (nseg per row):
// a block per row makes the chunk statistics in shared memory first.
// cudaErrorNotSupported (nothing launched) past 4096 chunks per row.
cudaError_t launch_sample_rows(const ZSource& zs, int rows, int n, const float2* stats,
                               int nseg, const int32_t* ids, float inv_tau, uint64_t seed,
                               uint64_t offset, int32_t* tokens, cudaStream_t st);
// One inverse-CDF draw per row from segment and chunk statistics with nseg
// segments per row (nseg * 32 >= n; segments past n hold zero weight);
// greedy: the first id of the row maximum (segment maxima, then the ids of
// the segment that holds it).
cudaError_t launch_sample_segments(const ZSource& zs, int rows, int n,
                                   const float2* stats, int nseg,
                                   const float2* cstats, const int32_t* ids,
                                   float inv_tau, uint64_t seed, uint64_t offset,
                                   int32_t* tokens, cudaStream_t st, int greedy = 0);
inline cudaError_t launch_sample_segments(const float* Z, int rows, int n,
                                          const float2* stats, int nseg,
                                          const float2* cstats, const int32_t* ids,
                                          float inv_tau, uint64_t seed, uint64_t offset,
                                          int32_t* tokens, cudaStream_t st, int greedy = 0) {
  ZSource zs;
  zs.Z = Z;
  return launch_sample_segments(zs, rows, n, stats, nseg, cstats, ids, inv_tau, seed, offset,
                                tokens, st, greedy);
}
int sample_max_n();
int verify_max_k();

// Speculative verification (four launches; greedy: three); `scratch` holds
// verify_scratch_bytes(sessions, k, n) bytes.
size_t verify_scratch_bytes(int sessions, int k, int n);
cudaError_t launch_verify(const float* Z, int sessions, int k, int n,
                          const int32_t* ids, int V, float inv_tau,
                          const int32_t* draft, const float* q,
                          uint64_t seed, uint64_t offset, int32_t* n_acc,
                          int32_t* next_token, void* scratch, int sm_count,
                          cudaStream_t st, int greedy = 0);

}  // namespace sph
