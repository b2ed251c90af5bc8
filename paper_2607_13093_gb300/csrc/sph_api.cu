// C-ABI layer of libsph: context, scratch arena, argument validation and
// dispatch of the split-head kernels.  Declared in include/sph.h.
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <new>
#include <string>
#include <vector>

#include "sph.h"
#include "sph_internal.h"

namespace sph {
thread_local long long launch_count = 0;
}

struct ProfPair {
  int cls;
  cudaEvent_t start, stop;
};

struct sph_ctx {
  int device = 0;
  cudaStream_t stream = nullptr;
  int sm_count = 0;
  std::string err;
  void* scratch = nullptr;          // arena for per-call temporaries
  size_t scratch_cap = 0;
  unsigned* status = nullptr;       // device error word (sph::ERR_* bits)
  int64_t tc_min_rows = 4;          // SPH_OPT_TC_MIN_ROWS
  long long spin_limit = 1ll << 34; // SPH_OPT_SPIN_LIMIT
  int tc_schedule = 0;              // SPH_OPT_TC_SCHEDULE
  int tc_stages = 0;                // SPH_OPT_TC_STAGES
  int tc_block_k = 0;               // SPH_OPT_TC_BLOCK_K
  int tc_max_bn = 0;                // SPH_OPT_TC_MAX_BN
  int tc_tile_m = 0;                // SPH_OPT_TC_TILE_M
  long long tc_finish_wait = 1ll << 15;   // SPH_OPT_TC_FINISH_WAIT
  int sampler = 0;                  // SPH_OPT_SAMPLER
  int check_ids = 0;                // SPH_OPT_CHECK_IDS
  int split_quantize = 0;           // SPH_OPT_SPLIT_QUANTIZE
  int tc_pair = 0;                  // SPH_OPT_TC_PAIR: 0 automatic, 1 always, 2 never
  int endpoint_z = 0;               // SPH_OPT_ENDPOINT_Z: 0 automatic, 1 store, 2 recompute
  int endpoint_rm = 0;              // SPH_OPT_ENDPOINT_ROWS_M: 0 automatic, 1 always, 2 never
  int gemv_quantize = 0;            // SPH_OPT_GEMV_QUANTIZE: 0 automatic, 1 never
  // the cloud GEMV's last-block quantization: row maxima [8] and the
  // arrival ticket, zero between calls (the last block resets them)
  unsigned* gemv_q = nullptr;
  int pair_units = 0;               // CTA pairs that fit at once (0: pairs unavailable)
  // chunked split steps: the endpoint's own stream (created on first use
  // when the caller passes none) and the events that order the two streams
  cudaStream_t aux_stream = nullptr;
  std::vector<cudaEvent_t> step_events;
  // sph_set_stream: orders the new stream after the old one's work
  cudaEvent_t switch_event = nullptr;
  // tracing
  bool prof = false;
  long long prof_launch0 = 0;
  sph_profile acc{};
  std::vector<ProfPair> pending;
  std::vector<cudaEvent_t> pool;
};

struct sph_buffer {
  void* ptr = nullptr;
  size_t bytes = 0;
};

namespace {

sph_status fail(sph_ctx* ctx, sph_status st, const char* fmt, ...) {
  if (ctx) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    ctx->err = buf;
  }
  return st;
}

sph_status cuda_fail(sph_ctx* ctx, cudaError_t e, const char* what) {
  return fail(ctx, SPH_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// RAII guard that makes the context's device current for one call.
struct DeviceGuard {
  int prev = -1;
  bool ok = true;
  explicit DeviceGuard(int dev) {
    if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
    if (prev != dev) ok = cudaSetDevice(dev) == cudaSuccess;
  }
  ~DeviceGuard() {
    int cur = -1;
    if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev)
      cudaSetDevice(prev);
  }
};

// Grow the scratch arena to `bytes` (outside stream capture only).
sph_status ensure_scratch(sph_ctx* ctx, size_t bytes) {
  if (bytes <= ctx->scratch_cap) return SPH_OK;
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(ctx->stream, &cap) == cudaSuccess &&
      cap != cudaStreamCaptureStatusNone)
    return fail(ctx, SPH_ERR_UNSUPPORTED,
                "scratch must grow to %zu bytes during stream capture; call "
                "sph_reserve() before capturing", bytes);
  cudaError_t e = cudaStreamSynchronize(ctx->stream);   // old arena may be in use
  if (e != cudaSuccess) return cuda_fail(ctx, e, "cudaStreamSynchronize");
  if (ctx->scratch) cudaFree(ctx->scratch);
  ctx->scratch = nullptr;
  ctx->scratch_cap = 0;
  const size_t want = align_up(bytes + bytes / 4, 1 << 20);
  e = cudaMalloc(&ctx->scratch, want);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return fail(ctx, SPH_ERR_OOM, "cudaMalloc(%zu) for scratch failed", want);
  }
  ctx->scratch_cap = want;
  return SPH_OK;
}

// Bump allocator over the arena for one call.  fits() says whether every
// piece taken so far lies inside the arena; calls check it before their
// first launch, so that a scratch plan that outgrew the arena is an error,
// never an out-of-bounds write.
struct Carve {
  char* base;
  size_t cap;
  size_t off = 0;
  Carve(void* b, size_t c) : base(static_cast<char*>(b)), cap(c) {}
  void* take(size_t bytes) {
    void* p = base ? base + off : nullptr;
    off = align_up(off + bytes, 256);
    return p;
  }
  bool fits() const { return off <= cap; }
};

bool use_tc(const sph_ctx* ctx, int64_t rows, int w_dtype) {
  (void)w_dtype;
  return rows >= ctx->tc_min_rows;
}

// tc_plan's pair mode: 0 never, 1 where it pays, 2 always
int pair_mode(const sph_ctx* ctx) {
  if (ctx->pair_units < 1 || ctx->tc_pair == 2) return 0;
  return ctx->tc_pair == 1 ? 2 : 1;
}

size_t tc_bytes(const sph_ctx* ctx, int64_t rows, int64_t n, int64_t K, int act_bf16,
                int w_dtype, int endpoint, int sm_count = 0) {
  if (!use_tc(ctx, rows, w_dtype)) return 0;
  if (sm_count <= 0) sm_count = ctx->sm_count;
  size_t b = 0;
  // the larger of the two paths, for the plan the call makes (tile height
  // as set, 0 automatic) and, with the automatic height, for both heights
  // (which smaller calls may choose)
  // (and with and without CTA pairs, which some endpoint calls leave out)
  const int pms[2] = {0, pair_mode(ctx)};
  for (int gather = 0; gather < 2; ++gather)
    for (int tm = 0; tm <= 256; tm += 128)
      for (int pi = 0; pi < (pms[1] ? 2 : 1); ++pi) {
        const int pm = pms[pi];
        if (ctx->tc_tile_m && tm != ctx->tc_tile_m) continue;
        const size_t x = sph::tc_plan((int)rows, (int)n, (int)K, act_bf16, sm_count,
                                      endpoint, ctx->tc_schedule, ctx->tc_stages,
                                      ctx->tc_block_k, gather, w_dtype == sph::W_FP8,
                                      ctx->tc_max_bn, tm, pm, ctx->pair_units,
                                      ctx->endpoint_rm)
                             .scratch_bytes;
        if (x > b) b = x;
      }
  return b;
}

size_t partial_scratch_bytes(const sph_ctx* ctx, int64_t rows, int64_t n, int64_t K,
                             int act_bf16, int w_dtype) {
  return align_up((size_t)rows * n * 4, 256) + align_up((size_t)rows * 4, 256) +
         tc_bytes(ctx, rows, n, K, act_bf16, w_dtype, 0);
}
// fused logits, then the tensor-core scratch (which holds the segment
// statistics) or, on the CUDA-core path, the segment statistics alone
size_t fuse_scratch_bytes(const sph_ctx* ctx, int64_t rows, int64_t n, int64_t K) {
  // chunk statistics: at most one per 1024 ids of the tensor-core tiling
  const size_t cstats = align_up((size_t)rows * (n / 1024 + 2) * 8, 256);
  const size_t stats = align_up((size_t)rows * sph::seg_count((int)n) * 8, 256);
  const size_t tc = tc_bytes(ctx, rows, n, K, 0, sph::W_BF16, 1);
  return align_up((size_t)rows * n * 4, 256) + cstats + (tc > stats ? tc : stats);
}
// verification over `rows` = sessions * (k + 1) target rows, for any split
size_t verify_reserve_bytes(int64_t rows, int64_t n) {
  return sph::verify_scratch_bytes((int)rows, 0, (int)n) + 2 * align_up((size_t)rows * 4, 256);
}

// SMs of the two halves of a chunked split step, in proportion to their
// cost per (row, id): the cloud's contraction over d_h in its operand
// planes (two for fp32 activations), the endpoint's over d_l in two planes
// plus its epilogue, which costs about as much as 1400 more columns
// (measured: 1024 rows x 256000 ids, cloud 3.17 ms over 4608 x 2, endpoint
// 0.82 ms over 512 x 2).  At least 4 SMs, at most half.
void split_sms(const sph_ctx* ctx, int64_t d_l, int64_t d_h, int act_bf16, int* sm_cloud,
               int* sm_end) {
  const double cloud = (double)d_h * (act_bf16 ? 1 : 2), end = 2.0 * (double)d_l + 1400.0;
  int e = (int)((double)ctx->sm_count * end / (cloud + end) + 0.5);
  if (e < 4) e = 4;
  if (e > ctx->sm_count / 2) e = ctx->sm_count / 2;
  if (e < 1) e = 1;
  *sm_end = e;
  *sm_cloud = ctx->sm_count - e > 0 ? ctx->sm_count - e : 1;
}
// Scratch of sph_split_step with chunks of L ids (L = n for one chunk), in
// the order the call carves it.
size_t split_scratch_bytes(const sph_ctx* ctx, int64_t rows, int64_t n, int64_t L, int64_t d_h,
                           int64_t d_l, int act_bf16, int w_dtype) {
  const bool chunked = L < n;
  int smc = ctx->sm_count, sme = ctx->sm_count;
  if (chunked) split_sms(ctx, d_l, d_h, act_bf16, &smc, &sme);
  const int64_t last = n - (n - 1) / L * L;
  // the larger of a chunk's plans, with the split SMs or (chunks one after
  // another on one stream) all of them
  auto plan_bytes = [&](int64_t K, int act, int wdt, int endpoint, int sm) {
    size_t x = 0;
    for (int64_t nq : {L, last})
      for (int s2 : {sm, ctx->sm_count}) {
        const size_t y = tc_bytes(ctx, rows, nq, K, act, wdt, endpoint, s2);
        if (y > x) x = y;
      }
    return x;
  };
  size_t b = align_up((size_t)rows * L * 4, 256) + align_up((size_t)rows * 4, 256);
  b += align_up(plan_bytes(d_h, act_bf16, w_dtype, 0, smc), 256);
  b += align_up((size_t)rows * n * 4, 256);                          // z
  b += align_up((size_t)rows * (n / 1024 + 2) * 8, 256);             // chunk statistics
  if (chunked) {
    b += align_up(plan_bytes(d_l, 0, sph::W_BF16, 1, sme), 256);
    b += align_up((size_t)rows * sph::seg_count((int)n) * 8, 256);   // segment statistics
  } else {
    const size_t tce = tc_bytes(ctx, rows, n, d_l, 0, sph::W_BF16, 1);
    const size_t st = (size_t)rows * sph::seg_count((int)n) * 8;
    b += align_up(tce > st ? tce : st, 256);
  }
  return b + 4096;
}

bool finite_pos(float x) { return std::isfinite(x) && x > 0.f; }
// temperature: > 0 samples from softmax(z / t); 0 is greedy decoding
bool valid_temperature(float t) { return std::isfinite(t) && t >= 0.f; }
float stats_inv_tau(float t) { return t > 0.f ? 1.0f / t : 1.0f; }

sph_status check_ids(sph_ctx* ctx, const int32_t* keep_ids, int64_t n_keep,
                     int64_t V) {
  if (V < 1 || V > INT32_MAX) return fail(ctx, SPH_ERR_INVALID_ARG, "V=%lld out of range", (long long)V);
  if (n_keep < 1 || n_keep > V)
    return fail(ctx, SPH_ERR_INVALID_ARG, "n_keep=%lld must be in [1, V=%lld]",
                (long long)n_keep, (long long)V);
  if (!keep_ids && n_keep != V)
    return fail(ctx, SPH_ERR_INVALID_ARG, "keep_ids NULL requires n_keep == V");
  return SPH_OK;
}

// SPH_OPT_CHECK_IDS: copy the device id list to the host and check it
// before anything is launched.  V < 0: the upper bound is not known (the
// verification call), only order and sign are checked.
sph_status host_check_ids(sph_ctx* ctx, const int32_t* keep_ids, int64_t n_keep, int64_t V) {
  if (!ctx->check_ids || !keep_ids) return SPH_OK;
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(ctx->stream, &cap) == cudaSuccess &&
      cap != cudaStreamCaptureStatusNone)
    return fail(ctx, SPH_ERR_UNSUPPORTED,
                "SPH_OPT_CHECK_IDS copies the ids to the host: not allowed during stream capture");
  std::vector<int32_t> ids((size_t)n_keep);
  cudaError_t e = cudaMemcpyAsync(ids.data(), keep_ids, (size_t)n_keep * 4,
                                  cudaMemcpyDeviceToHost, ctx->stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(ctx->stream);
  if (e != cudaSuccess) return cuda_fail(ctx, e, "copying keep_ids to the host");
  int64_t bad = -1;
  if (sph_check_keep_ids(ids.data(), n_keep, V < 0 ? (int64_t)INT32_MAX + 1 : V, &bad) != SPH_OK)
    return fail(ctx, SPH_ERR_INVALID_ARG,
                "keep_ids[%lld] = %d breaks the id conventions (strictly increasing, in [0, V))",
                (long long)bad, bad >= 0 ? ids[(size_t)bad] : 0);
  return SPH_OK;
}

sph_status launch_status(sph_ctx* ctx, cudaError_t e, const char* what) {
  if (e != cudaSuccess) return cuda_fail(ctx, e, what);
  return SPH_OK;
}

cudaEvent_t pooled_event(sph_ctx* ctx) {
  if (!ctx->pool.empty()) {
    cudaEvent_t ev = ctx->pool.back();
    ctx->pool.pop_back();
    return ev;
  }
  cudaEvent_t ev = nullptr;
  if (cudaEventCreate(&ev) != cudaSuccess) return nullptr;
  return ev;
}

// Run one kernel group; while tracing, bracket it with events of class cls.
template <class F>
cudaError_t traced(sph_ctx* ctx, int cls, F&& launch) {
  if (!ctx->prof) return launch();
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(ctx->stream, &cap) != cudaSuccess ||
      cap != cudaStreamCaptureStatusNone)
    return launch();                 // events are not timed inside a graph
  cudaEvent_t a = pooled_event(ctx), b = pooled_event(ctx);
  if (!a || !b) return launch();
  cudaEventRecord(a, ctx->stream);
  const cudaError_t e = launch();
  cudaEventRecord(b, ctx->stream);
  ctx->pending.push_back({cls, a, b});
  return e;
}

// traced() for a launch group that reports an sph_status
template <class F>
sph_status traced_status(sph_ctx* ctx, int cls, F&& launch) {
  sph_status st = SPH_OK;
  traced(ctx, cls, [&] {
    st = launch();
    return cudaSuccess;
  });
  return st;
}

// The endpoint half of a step on a prepared GatherGemm (EPI_ENDPOINT or
// EPI_FUSED, gg.Y = z): the local contraction with its fused epilogue, then
// the draw (S7-S11), on the context's stream.  `c` carves the rest of the
// scratch arena.  z_out: the caller asked for z (gg.Y is its buffer);
// otherwise gg.Y is scratch, and z need not be stored at all
// (SPH_OPT_ENDPOINT_Z): the epilogue then keeps only the segment
// statistics and the draw recomputes z for the segment it lands in.
sph_status endpoint_draw(sph_ctx* ctx, sph::GatherGemm& gg, Carve& c, float temperature,
                         uint64_t seed, uint64_t offset, int32_t* tokens, bool z_out) {
  const int rows = gg.rows, n_keep = gg.n;
  const int32_t* keep_ids = gg.ids;
  float* Z = gg.Y;
  float2* cstats = static_cast<float2*>(c.take((size_t)rows * (n_keep / 1024 + 2) * 8));
  gg.status = ctx->status; gg.finish_wait = ctx->tc_finish_wait;
  gg.inv_tau = stats_inv_tau(temperature);
  const int greedy = temperature == 0.f;
  // Gumbel-max draws need no softmax statistics: the epilogue skips them;
  // nor does a call without tokens (z alone, for the verification)
  const bool gumbel = ctx->sampler == 1 && !greedy;
  const bool fuse_only = tokens == nullptr;
  if (fuse_only && !z_out)
    return fail(ctx, SPH_ERR_INVALID_ARG, "a call without tokens needs fused_logits_out");
  gg.no_stats = gumbel || fuse_only;
  // z unstored (SPH_OPT_ENDPOINT_Z): automatic where the endpoint runs with
  // rows as M, whose epilogue makes each segment's statistics in its own
  // lane (measured, steps of 1024 x 256000 ids x d_l 512: 3.18 vs 3.43 ms;
  // 256 x 152064 x 1024: 0.87 vs 0.90 ms; 256 x 256000 x 512: 0.88 vs
  // 1.00 ms), not with ids as M (32 x 12000 x 256: 55 vs 49 us)
  const bool tc = use_tc(ctx, rows, sph::W_BF16);
  bool z_free = tc && !gumbel && !z_out && ctx->endpoint_z != 1;
  auto plan_of = [&](bool zf) {
    return sph::tc_plan(rows, n_keep, gg.K, 0, ctx->sm_count, zf ? 2 : 1, ctx->tc_schedule,
                        ctx->tc_stages, ctx->tc_block_k, keep_ids != nullptr, 0,
                        ctx->tc_max_bn, ctx->tc_tile_m, pair_mode(ctx), ctx->pair_units,
                        ctx->endpoint_rm);
  };
  sph::TcPlan pl{};
  if (tc) {
    pl = plan_of(z_free);
    if (z_free && ctx->endpoint_z == 0 && !pl.rm) {
      z_free = false;
      pl = plan_of(false);
    }
  }
  sph::ZSource zs;
  if (z_free) {
    gg.Y = nullptr;
    zs.h = gg.h; zs.ld_h = gg.ld_h; zs.K = gg.K; zs.W = gg.W; zs.ld_w = gg.ld_w;
    zs.ids = gg.ids;
    const bool fq = gg.epilogue == sph::EPI_FUSED;
    zs.codes = fq ? gg.codes_out : gg.codes;
    zs.row_scale = fq ? gg.scale_out : gg.row_scale;
  } else {
    zs.Z = Z;
  }
  sph_status st;
  auto draw_gumbel = [&] {
    return launch_status(ctx, traced(ctx, SPH_PROF_SAMPLE, [&] {
                           return sph::launch_gumbel(Z, rows, n_keep, keep_ids,
                                                     gg.inv_tau, seed, offset, tokens,
                                                     ctx->stream);
                         }), "sample launch");
  };
  if (tc) {
    void* tcs = c.take(pl.scratch_bytes);
    if (!c.fits())
      return fail(ctx, SPH_ERR_UNSUPPORTED, "internal: scratch plan of %zu bytes exceeds the arena of %zu",
                  c.off, ctx->scratch_cap);
    st = launch_status(ctx, traced(ctx, SPH_PROF_LOCAL_GEMM, [&] {
                         return sph::launch_tc(gg, pl, tcs, ctx->spin_limit, ctx->stream);
                       }), "tensor-core launch");
    if (st || fuse_only) return st;
    if (gumbel) return draw_gumbel();
    return launch_status(ctx, traced(ctx, SPH_PROF_SAMPLE, [&] {
                           return sph::launch_sample_from_stats(
                               zs, rows, n_keep, pl, tcs, cstats, keep_ids,
                               gg.inv_tau, seed, offset, ctx->sm_count, tokens,
                               ctx->stream, greedy);
                         }), "sample launch");
  }
  float2* stats = static_cast<float2*>(c.take((size_t)rows * sph::seg_count(n_keep) * 8));
  if (!c.fits())
    return fail(ctx, SPH_ERR_UNSUPPORTED, "internal: scratch plan of %zu bytes exceeds the arena of %zu",
                c.off, ctx->scratch_cap);
  st = launch_status(ctx, traced(ctx, SPH_PROF_LOCAL_GEMM, [&] {
                       return sph::launch_gemv(gg, ctx->sm_count, ctx->stream);
                     }), "gemv launch");
  if (st || fuse_only) return st;
  if (gumbel) return draw_gumbel();
  return launch_status(ctx, traced(ctx, SPH_PROF_SAMPLE, [&] {
                         cudaError_t e = sph::launch_seg_stats(Z, rows, n_keep,
                                                               gg.inv_tau, stats,
                                                               cstats, ctx->sm_count,
                                                               ctx->stream);
                         if (e != cudaSuccess) return e;
                         return sph::launch_sample_segments(
                             Z, rows, n_keep, stats, sph::seg_count(n_keep),
                             cstats, keep_ids, gg.inv_tau, seed, offset, tokens,
                             ctx->stream, greedy);
                       }), "sample launch");
}

}  // namespace

extern "C" {

const char* sph_status_string(sph_status s) {
  switch (s) {
    case SPH_OK: return "SPH_OK";
    case SPH_ERR_INVALID_ARG: return "SPH_ERR_INVALID_ARG";
    case SPH_ERR_UNSUPPORTED: return "SPH_ERR_UNSUPPORTED";
    case SPH_ERR_CUDA: return "SPH_ERR_CUDA";
    case SPH_ERR_TIMEOUT: return "SPH_ERR_TIMEOUT";
    case SPH_ERR_OOM: return "SPH_ERR_OOM";
  }
  return "SPH_ERR_UNKNOWN";
}

const char* sph_last_error(const sph_ctx* ctx) {
  return ctx ? ctx->err.c_str() : "null context";
}

size_t sph_payload_bytes(int64_t rows, int64_t n_keep) {
  if (rows < 0 || n_keep < 0) return 0;
  return (size_t)rows * (size_t)n_keep + 4 * (size_t)rows;
}

sph_status sph_keep_ids_from_mask(const uint8_t* mask, int64_t V,
                                  int32_t* keep_ids, int64_t* n_keep) {
  if (!mask || !keep_ids || !n_keep || V < 1 || V > INT32_MAX)
    return SPH_ERR_INVALID_ARG;
  int64_t n = 0;
  for (int64_t v = 0; v < V; ++v)
    if (mask[v >> 3] & (1u << (v & 7))) keep_ids[n++] = (int32_t)v;
  *n_keep = n;
  return n ? SPH_OK : SPH_ERR_INVALID_ARG;
}

sph_status sph_check_keep_ids(const int32_t* keep_ids, int64_t n_keep, int64_t V,
                              int64_t* bad_index) {
  if (bad_index) *bad_index = -1;
  if (!keep_ids || n_keep < 1 || V < 1) return SPH_ERR_INVALID_ARG;
  int64_t prev = -1;
  for (int64_t j = 0; j < n_keep; ++j) {
    const int64_t id = keep_ids[j];
    if (id <= prev || id >= V) {
      if (bad_index) *bad_index = j;
      return SPH_ERR_INVALID_ARG;
    }
    prev = id;
  }
  return SPH_OK;
}

sph_status sph_plan_query(sph_ctx* ctx, int call, int64_t rows, int64_t n_keep, int64_t K,
                          sph_dtype w_dtype, sph_act_mode act_mode, int gather,
                          sph_plan* out) {
  if (!ctx || !out) return SPH_ERR_INVALID_ARG;
  if ((call != 0 && call != 1) || rows < 1 || rows > (1 << 20) || n_keep < 1 ||
      n_keep > INT32_MAX || K < 1 || K > sph::gemv_max_k() ||
      (w_dtype != SPH_DTYPE_BF16 && w_dtype != SPH_DTYPE_FP8_E4M3) ||
      (act_mode != SPH_ACT_FP32 && act_mode != SPH_ACT_BF16) ||
      (call == 1 && w_dtype != SPH_DTYPE_BF16))
    return fail(ctx, SPH_ERR_INVALID_ARG, "sph_plan_query: bad arguments");
  *out = sph_plan{};
  const int wdt = w_dtype == SPH_DTYPE_BF16 ? sph::W_BF16 : sph::W_FP8;
  if (!use_tc(ctx, rows, wdt)) {
    out->gemv_rows = sph::gemv_rows_per_launch((int)rows, (int)K);
    return SPH_OK;
  }
  const sph::TcPlan pl = sph::tc_plan((int)rows, (int)n_keep, (int)K,
                                      call == 0 && act_mode == SPH_ACT_BF16, ctx->sm_count,
                                      call, ctx->tc_schedule, ctx->tc_stages, ctx->tc_block_k,
                                      gather != 0, wdt == sph::W_FP8, ctx->tc_max_bn,
                                      ctx->tc_tile_m, pair_mode(ctx), ctx->pair_units,
                                      ctx->endpoint_rm);
  out->tensor_core = 1;
  out->row_blocks = pl.RB;
  out->block_rows = pl.BN;
  out->tile_ids = pl.tm;
  out->tiles = pl.RB * pl.NT;
  out->k_blocks = pl.KB;
  out->stages = pl.stages;
  out->grid = pl.G;
  out->whole_tiles = pl.whole_tiles;
  out->planes = pl.hilo;
  out->pair = pl.pair;
  out->rows_m = pl.rm;
  out->epilogue_stats = pl.epi_stats;
  return SPH_OK;
}

sph_status sph_create(int device, void* cuda_stream, sph_ctx** out) {
  if (!out) return SPH_ERR_INVALID_ARG;
  *out = nullptr;
  int ndev = 0;
  if (cudaGetDeviceCount(&ndev) != cudaSuccess) {
    cudaGetLastError();
    return SPH_ERR_CUDA;
  }
  if (device < 0 || device >= ndev) return SPH_ERR_INVALID_ARG;
  sph_ctx* ctx = new (std::nothrow) sph_ctx();
  if (!ctx) return SPH_ERR_OOM;
  ctx->device = device;
  ctx->stream = static_cast<cudaStream_t>(cuda_stream);
  DeviceGuard g(device);
  if (!g.ok) { delete ctx; return SPH_ERR_CUDA; }
  if (cudaDeviceGetAttribute(&ctx->sm_count, cudaDevAttrMultiProcessorCount,
                             device) != cudaSuccess) {
    delete ctx;
    return SPH_ERR_CUDA;
  }
  // how many CTA pairs of the pair kernel fit at once (0: none)
  ctx->pair_units = sph::tc_pair_max_units(device);
  if (cudaMalloc(&ctx->status, sizeof(unsigned)) != cudaSuccess) {
    cudaGetLastError();
    delete ctx;
    return SPH_ERR_OOM;
  }
  if (cudaMemset(ctx->status, 0, sizeof(unsigned)) != cudaSuccess) {
    cudaFree(ctx->status);
    delete ctx;
    return SPH_ERR_CUDA;
  }
  if (cudaMalloc(&ctx->gemv_q, 16 * sizeof(unsigned)) != cudaSuccess ||
      cudaMemset(ctx->gemv_q, 0, 16 * sizeof(unsigned)) != cudaSuccess) {
    cudaGetLastError();
    if (ctx->gemv_q) cudaFree(ctx->gemv_q);
    cudaFree(ctx->status);
    delete ctx;
    return SPH_ERR_OOM;
  }
  *out = ctx;
  return SPH_OK;
}

sph_status sph_destroy(sph_ctx* ctx) {
  if (!ctx) return SPH_ERR_INVALID_ARG;
  DeviceGuard g(ctx->device);
  cudaStreamSynchronize(ctx->stream);
  if (ctx->scratch) cudaFree(ctx->scratch);
  if (ctx->status) cudaFree(ctx->status);
  if (ctx->gemv_q) cudaFree(ctx->gemv_q);
  if (ctx->aux_stream) cudaStreamDestroy(ctx->aux_stream);
  for (auto ev : ctx->step_events) cudaEventDestroy(ev);
  if (ctx->switch_event) cudaEventDestroy(ctx->switch_event);
  for (auto& p : ctx->pending) { cudaEventDestroy(p.start); cudaEventDestroy(p.stop); }
  for (auto ev : ctx->pool) cudaEventDestroy(ev);
  delete ctx;
  return SPH_OK;
}

sph_status sph_profile_enable(sph_ctx* ctx, int on) {
  if (!ctx) return SPH_ERR_INVALID_ARG;
  DeviceGuard g(ctx->device);
  if (on) {
    for (auto& p : ctx->pending) { ctx->pool.push_back(p.start); ctx->pool.push_back(p.stop); }
    ctx->pending.clear();
    ctx->acc = sph_profile{};
    ctx->prof_launch0 = sph::launch_count;
  }
  ctx->prof = on != 0;
  return SPH_OK;
}

sph_status sph_profile_read(sph_ctx* ctx, sph_profile* out) {
  if (!ctx || !out) return SPH_ERR_INVALID_ARG;
  DeviceGuard g(ctx->device);
  cudaError_t e = cudaStreamSynchronize(ctx->stream);
  if (e != cudaSuccess) return cuda_fail(ctx, e, "cudaStreamSynchronize");
  for (auto& p : ctx->pending) {
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, p.start, p.stop) == cudaSuccess) {
      ctx->acc.ms[p.cls] += ms;
      ctx->acc.calls[p.cls] += 1;
    }
    ctx->pool.push_back(p.start);
    ctx->pool.push_back(p.stop);
  }
  ctx->pending.clear();
  ctx->acc.launches = sph::launch_count - ctx->prof_launch0;
  *out = ctx->acc;
  return SPH_OK;
}

sph_status sph_set_stream(sph_ctx* ctx, void* cuda_stream) {
  if (!ctx) return SPH_ERR_INVALID_ARG;
  cudaStream_t next = static_cast<cudaStream_t>(cuda_stream);
  if (next == ctx->stream) return SPH_OK;
  DeviceGuard g(ctx->device);
  // Calls already issued on the old stream may still be using the scratch
  // (partials, row maxima, arrival counters) that the next call reuses, so
  // the new stream waits for them.  Not while either stream is being
  // captured: a capturing stream cannot wait on uncaptured work, and
  // recording on a stream outside a capture can invalidate it.  The new
  // stream is asked first, so that during a capture the old (possibly the
  // legacy default) stream is not touched at all.
  cudaStreamCaptureStatus cn = cudaStreamCaptureStatusNone, co = cudaStreamCaptureStatusNone;
  cudaError_t q = cudaStreamIsCapturing(next, &cn);
  if (q == cudaSuccess && cn == cudaStreamCaptureStatusNone)
    q = cudaStreamIsCapturing(ctx->stream, &co);
  if (q != cudaSuccess) cudaGetLastError();   // a refused query is not the caller's error
  if (q == cudaSuccess && cn == cudaStreamCaptureStatusNone &&
      co == cudaStreamCaptureStatusNone) {
    cudaError_t e = cudaSuccess;
    if (!ctx->switch_event)
      e = cudaEventCreateWithFlags(&ctx->switch_event, cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventRecord(ctx->switch_event, ctx->stream);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(next, ctx->switch_event, 0);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "ordering the new stream after the old one");
  }
  ctx->stream = next;
  return SPH_OK;
}

sph_status sph_sync(sph_ctx* ctx) {
  if (!ctx) return SPH_ERR_INVALID_ARG;
  DeviceGuard g(ctx->device);
  cudaError_t e = cudaStreamSynchronize(ctx->stream);
  if (e != cudaSuccess) return cuda_fail(ctx, e, "cudaStreamSynchronize");
  unsigned st = 0;
  e = cudaMemcpy(&st, ctx->status, sizeof st, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(ctx, e, "reading device status");
  if (st) {
    cudaMemset(ctx->status, 0, sizeof(unsigned));
    if (st & sph::ERR_TIMEOUT)
      return fail(ctx, SPH_ERR_TIMEOUT, "a device-side wait timed out (status 0x%x)", st);
    return fail(ctx, SPH_ERR_INVALID_ARG, "a kernel skipped out-of-range ids (status 0x%x)", st);
  }
  return SPH_OK;
}

sph_status sph_reserve(sph_ctx* ctx, int64_t max_rows, int64_t max_n_keep,
                       int64_t max_d) {
  if (!ctx || max_rows < 1 || max_n_keep < 1 || max_d < 1)
    return fail(ctx, SPH_ERR_INVALID_ARG, "sph_reserve: sizes must be >= 1");
  DeviceGuard g(ctx->device);
  size_t need = 0;
  for (int act = 0; act < 2; ++act) {
    const size_t a = partial_scratch_bytes(ctx, max_rows, max_n_keep, max_d, act, sph::W_BF16);
    if (a > need) need = a;
  }
  const size_t f = fuse_scratch_bytes(ctx, max_rows, max_n_keep, max_d);
  if (f > need) need = f;
  const size_t v = verify_reserve_bytes(max_rows, max_n_keep);
  if (v > need) need = v;
  for (int act = 0; act < 2; ++act) {      // a one-chunk split step
    const size_t a = split_scratch_bytes(ctx, max_rows, max_n_keep, max_n_keep, max_d, max_d,
                                         act, sph::W_BF16);
    if (a > need) need = a;
  }
  return ensure_scratch(ctx, need);
}

sph_status sph_set_option(sph_ctx* ctx, sph_option option, int64_t value) {
  if (!ctx) return SPH_ERR_INVALID_ARG;
  switch (option) {
    case SPH_OPT_TC_MIN_ROWS:
    case SPH_OPT_SPIN_LIMIT:
      if (value < 1) return fail(ctx, SPH_ERR_INVALID_ARG, "option value must be >= 1");
      if (option == SPH_OPT_TC_MIN_ROWS) ctx->tc_min_rows = value;
      else ctx->spin_limit = value;
      return SPH_OK;
    case SPH_OPT_TC_SCHEDULE:
      if (value < 0 || value > 2) return fail(ctx, SPH_ERR_INVALID_ARG, "schedule must be 0, 1 or 2");
      ctx->tc_schedule = (int)value;
      return SPH_OK;
    case SPH_OPT_TC_STAGES:
      if (value != 0 && (value < 2 || value > 12))
        return fail(ctx, SPH_ERR_INVALID_ARG, "stages must be 0 or in [2, 12]");
      ctx->tc_stages = (int)value;
      return SPH_OK;
    case SPH_OPT_TC_BLOCK_K:
      if (value != 0 && value != 64 && value != 128 && value != 256)
        return fail(ctx, SPH_ERR_INVALID_ARG, "block_k must be 0, 64, 128 or 256");
      ctx->tc_block_k = (int)value;
      return SPH_OK;
    case SPH_OPT_TC_MAX_BN:
      if (value != 0 && (value < 16 || value > 256 || value % 16))
        return fail(ctx, SPH_ERR_INVALID_ARG, "max_bn must be 0 or a multiple of 16 in [16, 256]");
      ctx->tc_max_bn = (int)value;
      return SPH_OK;
    case SPH_OPT_TC_TILE_M:
      if (value != 0 && value != 128 && value != 256)
        return fail(ctx, SPH_ERR_INVALID_ARG, "tile_m must be 0, 128 or 256");
      ctx->tc_tile_m = (int)value;
      return SPH_OK;
    case SPH_OPT_TC_FINISH_WAIT:
      if (value < 0) return fail(ctx, SPH_ERR_INVALID_ARG, "finish_wait must be >= 0");
      ctx->tc_finish_wait = value;
      return SPH_OK;
    case SPH_OPT_SAMPLER:
      if (value != 0 && value != 1) return fail(ctx, SPH_ERR_INVALID_ARG, "sampler must be 0 or 1");
      ctx->sampler = (int)value;
      return SPH_OK;
    case SPH_OPT_TC_PAIR:
      if (value < 0 || value > 2) return fail(ctx, SPH_ERR_INVALID_ARG, "tc_pair must be 0, 1 or 2");
      if (value == 1 && ctx->pair_units < 1)
        return fail(ctx, SPH_ERR_UNSUPPORTED, "CTA pairs cannot be scheduled on this device");
      ctx->tc_pair = (int)value;
      return SPH_OK;
    case SPH_OPT_SPLIT_QUANTIZE:
      if (value < 0 || value > 2) return fail(ctx, SPH_ERR_INVALID_ARG, "split_quantize must be 0, 1 or 2");
      ctx->split_quantize = (int)value;
      return SPH_OK;
    case SPH_OPT_ENDPOINT_ROWS_M:
      if (value < 0 || value > 2) return fail(ctx, SPH_ERR_INVALID_ARG, "endpoint_rows_m must be 0, 1 or 2");
      ctx->endpoint_rm = (int)value;
      return SPH_OK;
    case SPH_OPT_ENDPOINT_Z:
      if (value < 0 || value > 2) return fail(ctx, SPH_ERR_INVALID_ARG, "endpoint_z must be 0, 1 or 2");
      ctx->endpoint_z = (int)value;
      return SPH_OK;
    case SPH_OPT_CHECK_IDS:
      if (value != 0 && value != 1) return fail(ctx, SPH_ERR_INVALID_ARG, "check_ids must be 0 or 1");
      ctx->check_ids = (int)value;
      return SPH_OK;
    case SPH_OPT_GEMV_QUANTIZE:
      if (value != 0 && value != 1) return fail(ctx, SPH_ERR_INVALID_ARG, "gemv_quantize must be 0 or 1");
      ctx->gemv_quantize = (int)value;
      return SPH_OK;
  }
  return fail(ctx, SPH_ERR_INVALID_ARG, "unknown option %d", (int)option);
}

sph_status sph_buffer_alloc(sph_ctx* ctx, size_t bytes, sph_buffer** out) {
  if (!ctx || !out || bytes == 0) return fail(ctx, SPH_ERR_INVALID_ARG, "sph_buffer_alloc: bad arguments");
  DeviceGuard g(ctx->device);
  sph_buffer* b = new (std::nothrow) sph_buffer();
  if (!b) return SPH_ERR_OOM;
  if (cudaMalloc(&b->ptr, bytes) != cudaSuccess) {
    cudaGetLastError();
    delete b;
    return fail(ctx, SPH_ERR_OOM, "cudaMalloc(%zu) failed", bytes);
  }
  b->bytes = bytes;
  *out = b;
  return SPH_OK;
}

sph_status sph_buffer_free(sph_ctx* ctx, sph_buffer* buf) {
  if (!ctx || !buf) return SPH_ERR_INVALID_ARG;
  DeviceGuard g(ctx->device);
  cudaError_t e = cudaFree(buf->ptr);
  delete buf;
  return e == cudaSuccess ? SPH_OK : cuda_fail(ctx, e, "cudaFree");
}

void* sph_buffer_ptr(const sph_buffer* buf) { return buf ? buf->ptr : nullptr; }

sph_status sph_partial_logits(sph_ctx* ctx, const float* h_cloud, int64_t rows,
                              int64_t ld_h, const void* W_h, sph_dtype w_dtype,
                              int64_t V, int64_t d_h, int64_t ld_w,
                              const float* w_row_scale, const float* bias,
                              const int32_t* keep_ids, int64_t n_keep,
                              float clip, sph_act_mode act_mode, int8_t* codes,
                              float* row_scale, float* partial_out,
                              size_t* payload_bytes) {
  if (!ctx) return SPH_ERR_INVALID_ARG;
  if (!h_cloud || !W_h || !codes || !row_scale)
    return fail(ctx, SPH_ERR_INVALID_ARG, "h_cloud, W_h, codes and row_scale must be non-NULL");
  if (rows < 1 || rows > (1 << 20)) return fail(ctx, SPH_ERR_INVALID_ARG, "rows=%lld out of [1, 2^20]", (long long)rows);
  if (d_h < 1) return fail(ctx, SPH_ERR_INVALID_ARG, "d_h must be >= 1");
  if (ld_h < d_h || ld_w < d_h) return fail(ctx, SPH_ERR_INVALID_ARG, "ld_h and ld_w must be >= d_h");
  sph_status st = check_ids(ctx, keep_ids, n_keep, V);
  if (st) return st;
  if (!finite_pos(clip)) return fail(ctx, SPH_ERR_INVALID_ARG, "clip must be finite and > 0");
  if (w_dtype != SPH_DTYPE_BF16 && w_dtype != SPH_DTYPE_FP8_E4M3)
    return fail(ctx, SPH_ERR_INVALID_ARG, "unknown w_dtype %d", (int)w_dtype);
  if (act_mode != SPH_ACT_FP32 && act_mode != SPH_ACT_BF16)
    return fail(ctx, SPH_ERR_INVALID_ARG, "unknown act_mode %d", (int)act_mode);
  if (w_dtype == SPH_DTYPE_FP8_E4M3 && !w_row_scale)
    return fail(ctx, SPH_ERR_INVALID_ARG, "fp8 weights need w_row_scale");
  const int esz = w_dtype == SPH_DTYPE_BF16 ? 2 : 1;
  if (((uintptr_t)W_h & 15) || ((ld_w * esz) & 15))
    return fail(ctx, SPH_ERR_INVALID_ARG, "W_h base and row stride must be 16-byte aligned");
  if (rows * n_keep > ((int64_t)1 << 40)) return fail(ctx, SPH_ERR_UNSUPPORTED, "rows*n_keep too large");
  // the payload's consumer takes at most this many ids, and the kernels
  // index columns in 32 bits
  if (n_keep > sph::sample_max_n()) return fail(ctx, SPH_ERR_UNSUPPORTED, "n_keep above %d", sph::sample_max_n());
  if (d_h > sph::gemv_max_k()) return fail(ctx, SPH_ERR_UNSUPPORTED, "d_h=%lld above %d", (long long)d_h, sph::gemv_max_k());
  if (payload_bytes) *payload_bytes = sph_payload_bytes(rows, n_keep);

  DeviceGuard g(ctx->device);
  if (!g.ok) return fail(ctx, SPH_ERR_CUDA, "cudaSetDevice(%d) failed", ctx->device);
  st = host_check_ids(ctx, keep_ids, n_keep, V);
  if (st) return st;
  const int wdt = w_dtype == SPH_DTYPE_BF16 ? sph::W_BF16 : sph::W_FP8;
  const int act_bf16 = act_mode == SPH_ACT_BF16;
  st = ensure_scratch(ctx, partial_scratch_bytes(ctx, rows, n_keep, d_h, act_bf16, wdt));
  if (st) return st;
  Carve c(ctx->scratch, ctx->scratch_cap);
  float* Y = static_cast<float*>(c.take((size_t)rows * n_keep * 4));
  unsigned* rowmax = static_cast<unsigned*>(c.take((size_t)rows * 4));
  // few rows and a small payload: the GEMV's last block quantizes (no
  // separate pass, and its row maxima need no clearing)
  const bool gemv_q = !use_tc(ctx, rows, wdt) && ctx->gemv_quantize == 0 && ctx->gemv_q &&
                      sph::gemv_can_quantize(rows, n_keep, (int)d_h);
  if (!use_tc(ctx, rows, wdt) && !gemv_q) {   // the tensor-core path clears them itself
    cudaError_t e = cudaMemsetAsync(rowmax, 0, (size_t)rows * 4, ctx->stream);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "cudaMemsetAsync");
  }

  sph::GatherGemm gg{};
  gg.h = h_cloud; gg.ld_h = ld_h; gg.rows = (int)rows;
  gg.W = W_h; gg.ld_w = ld_w; gg.V = V;
  gg.w_dtype = wdt;
  gg.w_scale = w_row_scale; gg.K = (int)d_h;
  gg.ids = keep_ids; gg.n = (int)n_keep;
  gg.act_bf16 = act_bf16;
  gg.epilogue = sph::EPI_CLOUD;
  gg.bias = bias; gg.clip = clip; gg.partial_out = partial_out;
  gg.Y = Y; gg.rowmax = rowmax; gg.status = ctx->status; gg.finish_wait = ctx->tc_finish_wait;
  if (use_tc(ctx, rows, wdt)) {
    const sph::TcPlan pl = sph::tc_plan((int)rows, (int)n_keep, (int)d_h, act_bf16,
                                        ctx->sm_count, 0, ctx->tc_schedule, ctx->tc_stages,
                                        ctx->tc_block_k, keep_ids != nullptr,
                                        wdt == sph::W_FP8, ctx->tc_max_bn, ctx->tc_tile_m,
                                        pair_mode(ctx), ctx->pair_units);
    void* tcs = c.take(pl.scratch_bytes);
    if (!c.fits())
      return fail(ctx, SPH_ERR_UNSUPPORTED, "internal: scratch plan of %zu bytes exceeds the arena of %zu",
                  c.off, ctx->scratch_cap);
    st = launch_status(ctx, traced(ctx, SPH_PROF_CLOUD_GEMM, [&] {
                         return sph::launch_tc(gg, pl, tcs, ctx->spin_limit, ctx->stream);
                       }), "tensor-core launch");
  } else {
    if (gemv_q) {
      gg.rowmax = ctx->gemv_q;
      gg.q_ticket = ctx->gemv_q + 8;
      gg.q_codes = codes;
      gg.q_scale = row_scale;
    }
    st = launch_status(ctx, traced(ctx, SPH_PROF_CLOUD_GEMM, [&] {
                         return sph::launch_gemv(gg, ctx->sm_count, ctx->stream);
                       }), "gemv launch");
    if (st || gemv_q) return st;
  }
  if (st) return st;
  return launch_status(ctx, traced(ctx, SPH_PROF_QUANTIZE, [&] {
                         return sph::launch_quantize(Y, rowmax, (int)rows, (int)n_keep,
                                                     codes, row_scale, ctx->stream);
                       }), "quantize launch");
}

sph_status sph_fuse_sample(sph_ctx* ctx, const int8_t* codes,
                           const float* row_scale, int64_t rows,
                           const float* h_local, int64_t ld_hl,
                           const void* W_l, int64_t V, int64_t d_l,
                           int64_t ld_wl, const int32_t* keep_ids,
                           int64_t n_keep, float temperature, uint64_t seed,
                           uint64_t offset, int32_t* tokens,
                           float* fused_logits_out) {
  if (!ctx) return SPH_ERR_INVALID_ARG;
  if (!h_local || !W_l)
    return fail(ctx, SPH_ERR_INVALID_ARG, "h_local and W_l must be non-NULL");
  if (!tokens && !fused_logits_out)
    return fail(ctx, SPH_ERR_INVALID_ARG, "tokens and fused_logits_out must not both be NULL");
  if (!codes != !row_scale)
    return fail(ctx, SPH_ERR_INVALID_ARG, "codes and row_scale must both be given or both be NULL");
  if (rows < 1 || rows > (1 << 20)) return fail(ctx, SPH_ERR_INVALID_ARG, "rows=%lld out of [1, 2^20]", (long long)rows);
  if (d_l < 1) return fail(ctx, SPH_ERR_INVALID_ARG, "d_l must be >= 1");
  if (ld_hl < d_l || ld_wl < d_l) return fail(ctx, SPH_ERR_INVALID_ARG, "ld_hl and ld_wl must be >= d_l");
  sph_status st = check_ids(ctx, keep_ids, n_keep, V);
  if (st) return st;
  if (!valid_temperature(temperature)) return fail(ctx, SPH_ERR_INVALID_ARG, "temperature must be finite and >= 0");
  if (((uintptr_t)W_l & 15) || ((ld_wl * 2) & 15))
    return fail(ctx, SPH_ERR_INVALID_ARG, "W_l base and row stride must be 16-byte aligned");
  if (n_keep > sph::sample_max_n()) return fail(ctx, SPH_ERR_UNSUPPORTED, "n_keep above %d", sph::sample_max_n());
  if (d_l > sph::gemv_max_k()) return fail(ctx, SPH_ERR_UNSUPPORTED, "d_l above %d", sph::gemv_max_k());

  DeviceGuard g(ctx->device);
  if (!g.ok) return fail(ctx, SPH_ERR_CUDA, "cudaSetDevice(%d) failed", ctx->device);
  st = host_check_ids(ctx, keep_ids, n_keep, V);
  if (st) return st;
  st = ensure_scratch(ctx, fuse_scratch_bytes(ctx, rows, n_keep, d_l));
  if (st) return st;
  Carve c(ctx->scratch, ctx->scratch_cap);
  float* Z = static_cast<float*>(c.take((size_t)rows * n_keep * 4));
  if (fused_logits_out) Z = fused_logits_out;
  sph::GatherGemm gg{};
  gg.h = h_local; gg.ld_h = ld_hl; gg.rows = (int)rows;
  gg.W = W_l; gg.ld_w = ld_wl; gg.V = V; gg.w_dtype = sph::W_BF16; gg.K = (int)d_l;
  gg.ids = keep_ids; gg.n = (int)n_keep;
  gg.epilogue = sph::EPI_ENDPOINT;
  gg.Y = Z; gg.codes = codes; gg.row_scale = row_scale;
  return endpoint_draw(ctx, gg, c, temperature, seed, offset, tokens, fused_logits_out != nullptr);
}

sph_status sph_verify_draft(sph_ctx* ctx, const float* target_logits,
                            int64_t sessions, int64_t k,
                            const int32_t* keep_ids, int64_t n_keep,
                            float temperature, const int32_t* draft_tokens,
                            const float* draft_probs, uint64_t seed,
                            uint64_t offset, int32_t* n_accepted,
                            int32_t* next_token) {
  if (!ctx) return SPH_ERR_INVALID_ARG;
  if (!target_logits || !draft_tokens || !n_accepted || !next_token)
    return fail(ctx, SPH_ERR_INVALID_ARG, "target_logits, draft_tokens, n_accepted and next_token must be non-NULL");
  if (sessions < 1 || sessions > (1 << 20)) return fail(ctx, SPH_ERR_INVALID_ARG, "sessions out of [1, 2^20]");
  if (k < 1 || k > sph::verify_max_k())
    return fail(ctx, SPH_ERR_INVALID_ARG, "k must be in [1, %d]", sph::verify_max_k());
  if (sessions * (k + 1) > (1 << 20))
    return fail(ctx, SPH_ERR_INVALID_ARG, "sessions * (k + 1) above 2^20 target rows");
  if (n_keep < 1 || n_keep > INT32_MAX) return fail(ctx, SPH_ERR_INVALID_ARG, "n_keep must be >= 1");
  if (!valid_temperature(temperature)) return fail(ctx, SPH_ERR_INVALID_ARG, "temperature must be finite and >= 0");
  if (n_keep > sph::sample_max_n()) return fail(ctx, SPH_ERR_UNSUPPORTED, "n_keep above %d", sph::sample_max_n());
  DeviceGuard g(ctx->device);
  if (!g.ok) return fail(ctx, SPH_ERR_CUDA, "cudaSetDevice(%d) failed", ctx->device);
  sph_status st = host_check_ids(ctx, keep_ids, n_keep, -1);
  if (st) return st;
  st = ensure_scratch(
      ctx, sph::verify_scratch_bytes((int)sessions, (int)k, (int)n_keep));
  if (st) return st;
  // without an id list the compact index is the vocabulary id itself
  const int V = keep_ids ? INT32_MAX : (int)n_keep;
  return launch_status(ctx, traced(ctx, SPH_PROF_VERIFY, [&] {
                         return sph::launch_verify(target_logits, (int)sessions, (int)k,
                                                   (int)n_keep, keep_ids, V,
                                                   stats_inv_tau(temperature), draft_tokens,
                                                   draft_probs, seed, offset,
                                                   n_accepted, next_token, ctx->scratch,
                                                   ctx->sm_count, ctx->stream,
                                                   temperature == 0.f);
                       }), "verify launch");
}

sph_status sph_split_step(sph_ctx* ctx, const float* h, int64_t rows, int64_t ld_h,
                          int64_t d_l, int64_t d_h, const void* W_h, sph_dtype w_dtype,
                          const float* w_row_scale, int64_t ld_wh, const void* W_l,
                          int64_t ld_wl, int64_t V, const float* bias,
                          const int32_t* keep_ids, int64_t n_keep, float clip,
                          sph_act_mode act_mode, float temperature, uint64_t seed,
                          uint64_t offset, int64_t chunk, void* endpoint_stream,
                          int8_t* codes, float* scales, int32_t* tokens,
                          float* fused_logits_out, size_t* payload_bytes) {
  if (!ctx) return SPH_ERR_INVALID_ARG;
  if (!h || !W_h || !W_l || !codes || !scales || !tokens)
    return fail(ctx, SPH_ERR_INVALID_ARG, "h, W_h, W_l, codes, scales and tokens must be non-NULL");
  if (rows < 1 || rows > (1 << 20)) return fail(ctx, SPH_ERR_INVALID_ARG, "rows=%lld out of [1, 2^20]", (long long)rows);
  if (d_l < 1 || d_h < 1) return fail(ctx, SPH_ERR_INVALID_ARG, "d_l and d_h must be >= 1");
  if (ld_h < d_l + d_h || ld_wh < d_h || ld_wl < d_l)
    return fail(ctx, SPH_ERR_INVALID_ARG, "ld_h >= d_l + d_h, ld_wh >= d_h and ld_wl >= d_l are required");
  sph_status st = check_ids(ctx, keep_ids, n_keep, V);
  if (st) return st;
  if (!finite_pos(clip)) return fail(ctx, SPH_ERR_INVALID_ARG, "clip must be finite and > 0");
  if (!valid_temperature(temperature)) return fail(ctx, SPH_ERR_INVALID_ARG, "temperature must be finite and >= 0");
  if (w_dtype != SPH_DTYPE_BF16 && w_dtype != SPH_DTYPE_FP8_E4M3)
    return fail(ctx, SPH_ERR_INVALID_ARG, "unknown w_dtype %d", (int)w_dtype);
  if (act_mode != SPH_ACT_FP32 && act_mode != SPH_ACT_BF16)
    return fail(ctx, SPH_ERR_INVALID_ARG, "unknown act_mode %d", (int)act_mode);
  if (w_dtype == SPH_DTYPE_FP8_E4M3 && !w_row_scale)
    return fail(ctx, SPH_ERR_INVALID_ARG, "fp8 weights need w_row_scale");
  const int esz = w_dtype == SPH_DTYPE_BF16 ? 2 : 1;
  if (((uintptr_t)W_h & 15) || ((ld_wh * esz) & 15) || ((uintptr_t)W_l & 15) || ((ld_wl * 2) & 15))
    return fail(ctx, SPH_ERR_INVALID_ARG, "W_h and W_l base addresses and row strides must be 16-byte aligned");
  if (chunk < 0) return fail(ctx, SPH_ERR_INVALID_ARG, "chunk must be >= 0");
  if (n_keep > sph::sample_max_n()) return fail(ctx, SPH_ERR_UNSUPPORTED, "n_keep above %d", sph::sample_max_n());
  if (d_h > sph::gemv_max_k() || d_l > sph::gemv_max_k())
    return fail(ctx, SPH_ERR_UNSUPPORTED, "d_h or d_l above %d", sph::gemv_max_k());
  const int64_t L = (chunk == 0 || chunk >= n_keep) ? n_keep : chunk;
  const int64_t nchunk = (n_keep + L - 1) / L;
  if (payload_bytes) *payload_bytes = (size_t)rows * (size_t)n_keep + 4 * (size_t)rows * (size_t)nchunk;

  DeviceGuard g(ctx->device);
  if (!g.ok) return fail(ctx, SPH_ERR_CUDA, "cudaSetDevice(%d) failed", ctx->device);
  st = host_check_ids(ctx, keep_ids, n_keep, V);
  if (st) return st;
  const int wdt = w_dtype == SPH_DTYPE_BF16 ? sph::W_BF16 : sph::W_FP8;
  const int act_bf16 = act_mode == SPH_ACT_BF16;
  st = ensure_scratch(ctx, split_scratch_bytes(ctx, rows, n_keep, L, d_h, d_l, act_bf16, wdt));
  if (st) return st;
  const bool chunked = nchunk > 1;
  // the endpoint's chunks on the context's own stream: one after another,
  // each with every SM
  const bool serial = chunked && endpoint_stream == static_cast<void*>(ctx->stream);
  int sm_cloud = ctx->sm_count, sm_end = ctx->sm_count;
  if (chunked && !serial) split_sms(ctx, d_l, d_h, act_bf16, &sm_cloud, &sm_end);

  Carve c(ctx->scratch, ctx->scratch_cap);
  float* Y = static_cast<float*>(c.take((size_t)rows * L * 4));
  unsigned* rowmax = static_cast<unsigned*>(c.take((size_t)rows * 4));
  const int64_t last = n_keep - (nchunk - 1) * L;
  size_t tcc = tc_bytes(ctx, rows, L, d_h, act_bf16, wdt, 0, sm_cloud);
  const size_t tcc2 = tc_bytes(ctx, rows, last, d_h, act_bf16, wdt, 0, sm_cloud);
  if (tcc2 > tcc) tcc = tcc2;
  void* cloud_tc = c.take(tcc);
  float* Z = static_cast<float*>(c.take((size_t)rows * n_keep * 4));
  if (fused_logits_out) Z = fused_logits_out;

  // the cloud half of chunk q (S1-S4; the quantization is the caller's)
  auto cloud = [&](int64_t q, int64_t n_q, cudaStream_t s) -> sph_status {
    const int64_t j0 = q * L;
    sph::GatherGemm gg{};
    gg.h = h + d_l; gg.ld_h = ld_h; gg.rows = (int)rows;
    // the full vocabulary is cut by moving the weights' base to the chunk's
    // first row (its ids are then 0 .. n_q - 1 again); a kept-id list by
    // moving the list
    gg.W = keep_ids ? W_h : static_cast<const char*>(W_h) + j0 * ld_wh * esz;
    gg.ld_w = ld_wh; gg.V = keep_ids ? V : V - j0;
    gg.w_dtype = wdt;
    gg.w_scale = (w_row_scale && !keep_ids) ? w_row_scale + j0 : w_row_scale;
    gg.K = (int)d_h;
    gg.ids = keep_ids ? keep_ids + j0 : nullptr; gg.n = (int)n_q;
    gg.act_bf16 = act_bf16;
    gg.epilogue = sph::EPI_CLOUD;
    gg.bias = (bias && !keep_ids) ? bias + j0 : bias; gg.clip = clip;
    gg.Y = Y; gg.rowmax = rowmax; gg.status = ctx->status; gg.finish_wait = ctx->tc_finish_wait;
    if (use_tc(ctx, rows, wdt)) {
      const sph::TcPlan pl = sph::tc_plan((int)rows, (int)n_q, (int)d_h, act_bf16, sm_cloud, 0,
                                          ctx->tc_schedule, ctx->tc_stages, ctx->tc_block_k,
                                          keep_ids != nullptr, wdt == sph::W_FP8,
                                          ctx->tc_max_bn, ctx->tc_tile_m, pair_mode(ctx),
                                          ctx->pair_units);
      if (pl.scratch_bytes > tcc)
        return fail(ctx, SPH_ERR_UNSUPPORTED, "internal: cloud plan outgrew its scratch");
      return launch_status(ctx, sph::launch_tc(gg, pl, cloud_tc, ctx->spin_limit, s),
                           "tensor-core launch");
    }
    cudaError_t e = cudaMemsetAsync(rowmax, 0, (size_t)rows * 4, s);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "cudaMemsetAsync");
    return launch_status(ctx, sph::launch_gemv(gg, ctx->sm_count, s), "gemv launch");
  };

  if (!chunked) {
    // one chunk: the cloud contraction, then either the endpoint
    // contraction whose epilogue quantizes the cloud's clipped partials
    // itself and fuses them (no separate quantize launch: faster where the
    // payload is small and the launch's fixed cost weighs most), or the
    // quantize pass and the ordinary endpoint epilogue (faster for large
    // payloads, where the fused epilogue's fp32 reads are not hidden behind
    // the short endpoint contraction); then the draw.  Measured: decode (32
    // x 12000 ids) 47.4 vs 48.6 us a step fused; 32 x 60000 ids and 1024 x
    // 256000 ids slower fused.
    if (!c.fits())
      return fail(ctx, SPH_ERR_UNSUPPORTED, "internal: scratch plan of %zu bytes exceeds the arena of %zu",
                  c.off, ctx->scratch_cap);
    st = traced_status(ctx, SPH_PROF_CLOUD_GEMM, [&] { return cloud(0, n_keep, ctx->stream); });
    if (st) return st;
    const bool fuse_q = ctx->split_quantize == 1 ||
                        (ctx->split_quantize == 0 && rows * n_keep <= ((int64_t)1 << 20));
    sph::GatherGemm gg{};
    gg.h = h; gg.ld_h = ld_h; gg.rows = (int)rows;
    gg.W = W_l; gg.ld_w = ld_wl; gg.V = V; gg.w_dtype = sph::W_BF16; gg.K = (int)d_l;
    gg.ids = keep_ids; gg.n = (int)n_keep;
    gg.Y = Z;
    if (fuse_q) {
      gg.epilogue = sph::EPI_FUSED;
      gg.yc = Y; gg.rowmax_in = rowmax; gg.codes_out = codes; gg.scale_out = scales;
    } else {
      st = launch_status(ctx, traced(ctx, SPH_PROF_QUANTIZE, [&] {
                           return sph::launch_quantize(Y, rowmax, (int)rows, (int)n_keep, codes,
                                                       scales, ctx->stream);
                         }), "quantize launch");
      if (st) return st;
      gg.epilogue = sph::EPI_ENDPOINT;
      gg.codes = codes; gg.row_scale = scales;
    }
    return endpoint_draw(ctx, gg, c, temperature, seed, offset, tokens,
                         fused_logits_out != nullptr);
  }

  // chunks: the cloud emits chunk q (codes + a scale per row) on the
  // context's stream while the endpoint fuses chunk q - 1 on its own stream
  void* ecarve_tc;
  size_t tce = tc_bytes(ctx, rows, L, d_l, 0, sph::W_BF16, 1, sm_end);
  const size_t tce2 = tc_bytes(ctx, rows, last, d_l, 0, sph::W_BF16, 1, sm_end);
  if (tce2 > tce) tce = tce2;
  ecarve_tc = c.take(tce);
  float2* cstats = static_cast<float2*>(c.take((size_t)rows * (n_keep / 1024 + 2) * 8));
  float2* stats = static_cast<float2*>(c.take((size_t)rows * sph::seg_count((int)n_keep) * 8));
  if (!c.fits())
    return fail(ctx, SPH_ERR_UNSUPPORTED, "internal: scratch plan of %zu bytes exceeds the arena of %zu",
                c.off, ctx->scratch_cap);
  cudaStream_t es = static_cast<cudaStream_t>(endpoint_stream);
  if (!es && !serial) {
    if (!ctx->aux_stream) {
      cudaError_t e = cudaStreamCreateWithFlags(&ctx->aux_stream, cudaStreamNonBlocking);
      if (e != cudaSuccess) { ctx->aux_stream = nullptr; return cuda_fail(ctx, e, "cudaStreamCreate"); }
    }
    es = ctx->aux_stream;
  }
  if (serial) es = ctx->stream;
  while (!serial && ctx->step_events.size() < (size_t)nchunk + 2) {
    cudaEvent_t ev = nullptr;
    cudaError_t e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "cudaEventCreate");
    ctx->step_events.push_back(ev);
  }
  cudaEvent_t* ev = ctx->step_events.data();
  cudaError_t e = cudaSuccess;
  if (!serial) {
    e = cudaEventRecord(ev[0], ctx->stream);   // the endpoint follows earlier work
    if (e == cudaSuccess) e = cudaStreamWaitEvent(es, ev[0], 0);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "ordering the endpoint stream");
  }
  const float inv_tau = stats_inv_tau(temperature);
  for (int64_t q = 0; q < nchunk; ++q) {
    const int64_t j0 = q * L, n_q = q + 1 < nchunk ? L : last;
    int8_t* codes_q = codes + j0 * rows;         // chunk-major payload
    float* scales_q = scales + q * rows;
    st = cloud(q, n_q, ctx->stream);
    if (st) return st;
    st = launch_status(ctx, sph::launch_quantize(Y, rowmax, (int)rows, (int)n_q, codes_q,
                                                 scales_q, ctx->stream), "quantize launch");
    if (st) return st;
    if (!serial) {
      e = cudaEventRecord(ev[q + 1], ctx->stream);
      if (e == cudaSuccess) e = cudaStreamWaitEvent(es, ev[q + 1], 0);
      if (e != cudaSuccess) return cuda_fail(ctx, e, "ordering the endpoint stream");
    }
    // the endpoint half of chunk q: z[:, j0 : j0 + n_q] (S7-S8); the
    // statistics come from one pass over all of z after the last chunk
    sph::GatherGemm gg{};
    gg.h = h; gg.ld_h = ld_h; gg.rows = (int)rows;
    gg.W = keep_ids ? W_l : static_cast<const char*>(W_l) + j0 * ld_wl * 2;
    gg.ld_w = ld_wl; gg.V = keep_ids ? V : V - j0; gg.w_dtype = sph::W_BF16; gg.K = (int)d_l;
    gg.ids = keep_ids ? keep_ids + j0 : nullptr; gg.n = (int)n_q;
    gg.epilogue = sph::EPI_ENDPOINT;
    gg.codes = codes_q; gg.row_scale = scales_q;
    gg.Y = Z + j0; gg.ldy = n_keep;
    gg.status = ctx->status; gg.finish_wait = ctx->tc_finish_wait;
    gg.inv_tau = inv_tau; gg.no_stats = true;
    if (use_tc(ctx, rows, sph::W_BF16)) {
      const sph::TcPlan pl = sph::tc_plan((int)rows, (int)n_q, (int)d_l, 0, sm_end, 1,
                                          ctx->tc_schedule, ctx->tc_stages, ctx->tc_block_k,
                                          keep_ids != nullptr, 0, ctx->tc_max_bn, ctx->tc_tile_m);
      if (pl.scratch_bytes > tce)
        return fail(ctx, SPH_ERR_UNSUPPORTED, "internal: endpoint plan outgrew its scratch");
      st = launch_status(ctx, sph::launch_tc(gg, pl, ecarve_tc, ctx->spin_limit, es),
                         "tensor-core launch");
    } else {
      st = launch_status(ctx, sph::launch_gemv(gg, ctx->sm_count, es), "gemv launch");
    }
    if (st) return st;
  }
  // the draw over the whole fused row (S9-S11), on the endpoint's stream
  const int greedy = temperature == 0.f;
  if (ctx->sampler == 1 && !greedy) {
    e = sph::launch_gumbel(Z, (int)rows, (int)n_keep, keep_ids, inv_tau, seed, offset, tokens, es);
  } else {
    e = sph::launch_seg_stats(Z, (int)rows, (int)n_keep, inv_tau, stats, cstats, ctx->sm_count, es);
    if (e == cudaSuccess)
      e = sph::launch_sample_segments(Z, (int)rows, (int)n_keep, stats,
                                      sph::seg_count((int)n_keep), cstats, keep_ids, inv_tau,
                                      seed, offset, tokens, es, greedy);
  }
  if (e != cudaSuccess) return cuda_fail(ctx, e, "sample launch");
  if (serial) return SPH_OK;
  // the call ends, on the context's stream, when the endpoint's work has
  e = cudaEventRecord(ev[nchunk + 1], es);
  if (e == cudaSuccess) e = cudaStreamWaitEvent(ctx->stream, ev[nchunk + 1], 0);
  if (e != cudaSuccess) return cuda_fail(ctx, e, "joining the endpoint stream");
  return SPH_OK;
}

}  // extern "C"
