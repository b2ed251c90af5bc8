/*
 * sph.h -- C ABI of the split-head vocabulary projection library (libsph.so)
 *
 * The library computes, on one GB300 GPU (sm_103a), the data-parallel hot
 * path of the distributed vocabulary projection of "Efficient and Privacy
 * Aware Edge Cloud Collaborative Inference for Large Language Models"
 * (Sec. "Distributed Vocabulary Projection", Eqs. 9-15; Sec. "Transport
 * Protection", Eq. 18; Sec. "Endpoint Speculative Decoding and Cloud
 * Verification" with Algorithm 1):
 *
 *   cloud     y = h[:, d_l:] . W_h[V_l]^T (+ b[V_l])   -> clip -> per-row int8
 *   endpoint  z = dequant(codes) + h[:, :d_l] . W_l[V_l]^T -> mask -> softmax/tau
 *             -> sample ; speculative acceptance of k draft tokens
 *
 * Conventions shared by every call
 *   - Every function returns sph_status.  Scalar arguments and pointer
 *     presence are validated synchronously on the host; on failure nothing
 *     is launched and sph_last_error(ctx) describes the problem.
 *   - Compute calls are asynchronous on the context's stream.  Faults and
 *     device-side timeouts surface at sph_sync() (or the next call).
 *   - All tensor pointers are DEVICE pointers owned by the caller; the
 *     library never keeps them past the call.  Layouts are row-major with
 *     the stated leading dimension (in elements).  The context owns only
 *     its scratch memory (grown on demand, or pre-sized by sph_reserve()).
 *   - keep_ids is the language subset V_l: int32 vocabulary ids, strictly
 *     increasing, each in [0, V).  This is a precondition the kernels do
 *     not check: an id outside [0, V) makes them read outside W (and
 *     w_row_scale, bias).  NULL means the full vocabulary
 *     (mixed-language mode) and then n_keep must equal V.  Payloads and
 *     logits are "compacted": column j belongs to vocabulary id keep_ids[j].
 *   - A context is not thread-safe; use one per host thread.
 *   - There is no CPU fallback: a shape the kernels do not support returns
 *     SPH_ERR_UNSUPPORTED.  The hot-path calls take at most 2^20 rows (or
 *     sessions*(k+1) target rows) and at most 2^30 kept ids per row.
 */
#ifndef SPH_H_
#define SPH_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum sph_status {
  SPH_OK = 0,
  SPH_ERR_INVALID_ARG = 1,  /* bad scalar, NULL pointer, inconsistent sizes   */
  SPH_ERR_UNSUPPORTED = 2,  /* valid but outside what the kernels implement   */
  SPH_ERR_CUDA = 3,         /* a CUDA runtime call or a kernel launch failed  */
  SPH_ERR_TIMEOUT = 4,      /* a bounded device-side wait gave up             */
  SPH_ERR_OOM = 5           /* scratch memory could not be allocated          */
} sph_status;

typedef enum sph_dtype {
  SPH_DTYPE_BF16 = 0,       /* bfloat16 weights                                */
  SPH_DTYPE_FP8_E4M3 = 1    /* OCP e4m3 ('fn') weights with an fp32 scale per
                               vocabulary row: value = e4m3 * w_row_scale[v]  */
} sph_dtype;

typedef enum sph_act_mode {
  SPH_ACT_FP32 = 0,         /* hidden states used at fp32 accuracy (default)  */
  SPH_ACT_BF16 = 1          /* hidden states rounded to bf16 (RNE) first, as a
                               bf16 cloud decoder would hand them over        */
} sph_act_mode;

typedef struct sph_ctx sph_ctx;
typedef struct sph_buffer sph_buffer;

/* ---- context and memory ------------------------------------------------ */

/* Create a context on CUDA device `device` issuing work on `cuda_stream`
 * (a cudaStream_t; NULL = the legacy default stream).  *out receives the
 * handle.  Errors: INVALID_ARG (out NULL, bad device), CUDA, OOM. */
sph_status sph_create(int device, void* cuda_stream, sph_ctx** out);

/* Release the context and its scratch (waits for its stream first). */
sph_status sph_destroy(sph_ctx* ctx);

/* Issue subsequent calls on another stream of the same device.  The new
 * stream is made to wait (an event, no host synchronization) for the work
 * already issued on the old one, since the next call reuses the context's
 * scratch.  While either stream is being captured into a CUDA graph no
 * ordering is added: the caller orders the two streams itself.  The old
 * stream must not have been destroyed (as for sph_destroy and sph_sync,
 * which wait on the context's stream). */
sph_status sph_set_stream(sph_ctx* ctx, void* cuda_stream);

/* Wait for all work of the context's stream; report device-side errors
 * (SPH_ERR_TIMEOUT for a wait that gave up, SPH_ERR_CUDA for faults). */
sph_status sph_sync(sph_ctx* ctx);

/* Human-readable detail of the last error of `ctx` ("" if none). Owned by
 * the context, valid until its next call. */
const char* sph_last_error(const sph_ctx* ctx);

/* Static name of a status code. */
const char* sph_status_string(sph_status status);

/* Pre-size the context's scratch for calls up to these sizes so that later
 * calls allocate nothing (required before capturing calls into a CUDA
 * graph).  max_d is the largest of d_h and d_l. */
sph_status sph_reserve(sph_ctx* ctx, int64_t max_rows, int64_t max_n_keep,
                       int64_t max_d);

/* Tunables of a context. */
typedef enum sph_option {
  SPH_OPT_TC_MIN_ROWS = 0,  /* row count from which the tcgen05 tensor-core
                               kernels replace the CUDA-core GEMV (default 4;
                               1 forces tensor cores, a huge value forces the
                               GEMV)                                          */
  SPH_OPT_SPIN_LIMIT = 1,   /* clock cycles a device-side wait may spin before
                               it gives up and the call reports
                               SPH_ERR_TIMEOUT (default 2^34, >= 1)           */
  SPH_OPT_TC_SCHEDULE = 2,  /* tensor-core work split: 0 automatic (default),
                               1 whole vocabulary tiles per CTA, 2 contiguous
                               k-block ranges (stream-K)                      */
  SPH_OPT_TC_STAGES = 3,    /* tensor-core pipeline depth: 0 automatic
                               (default), else at most this many stages (>= 2) */
  SPH_OPT_TC_BLOCK_K = 4,   /* hidden-dimension elements each pipeline stage
                               reads per weight row: 64, 128, 256, or 0 for
                               automatic (default)                           */
  SPH_OPT_TC_MAX_BN = 5,    /* most hidden-state rows one tensor-core tile
                               covers: a multiple of 16 in [16, 256], or 0
                               for automatic (default); with
                               SPH_OPT_TC_TILE_M = 256, above 128 selects
                               256-id tiles with one accumulator            */
  SPH_OPT_TC_TILE_M = 6,    /* kept vocabulary ids one tensor-core tile
                               covers: 128, 256 (two 128-row MMAs sharing each
                               hidden-state stage), or 0 for automatic
                               (default).  A 256-id tile keeps two
                               accumulators for up to 128 hidden-state rows;
                               with SPH_OPT_TC_MAX_BN above 128 (and in the
                               automatic plan for row blocks of 129-192 rows)
                               it keeps one, for up to 256 rows (224 with fp32
                               activations)                                  */
  SPH_OPT_TC_FINISH_WAIT = 7, /* clock cycles the designated finisher of a
                               tensor-core tile split across CTAs polls for
                               the other contributors' partials (default
                               2^15, >= 0; 0: no finisher, the last
                               contributor to count in finishes the tile).
                               Results are bit-identical for every value.   */
  SPH_OPT_CHECK_IDS = 9,    /* 1: before launching anything, every hot-path
                               call copies keep_ids to the host (a
                               synchronous copy on the context's stream; not
                               allowed while the stream is being captured)
                               and checks them with sph_check_keep_ids,
                               returning SPH_ERR_INVALID_ARG for unsorted,
                               repeated or out-of-range ids.  0 (default):
                               the ids are a precondition, not checked.    */
  SPH_OPT_TC_PAIR = 11,     /* CTA pairs for the tensor-core contractions
                               (the cloud's with bf16 weights, and the
                               endpoint's; clusters of two CTAs, tcgen05
                               .cta_group::2): each 256-id tile is one M = 256
                               MMA over both CTAs' shared memory, each CTA
                               loading 128 ids of the weights and half of the
                               hidden-state rows.  0 (default): where the row
                               blocks are long (bf16 weights; >= 128 rows
                               for the cloud, >= 192 for the endpoint);
                               1: always (SPH_ERR_
                               UNSUPPORTED where pairs cannot be scheduled);
                               2: never.  The results are the fp32 sums of
                               the same products either way.               */
  SPH_OPT_SPLIT_QUANTIZE = 10, /* sph_split_step with one payload chunk: 0
                               automatic (default: in the endpoint's epilogue
                               for at most 2^20 rows x ids, else a separate
                               pass), 1 always in the endpoint contraction's
                               epilogue, 2 always a separate quantize pass.
                               The payload, z and tokens are bit-identical
                               either way.                                  */
  SPH_OPT_ENDPOINT_ROWS_M = 13, /* the endpoint contraction on CTA pairs
                               with the hidden-state rows as the MMA's M
                               dimension (256 rows over the pair, the tile's
                               256 ids as N), so that each epilogue thread
                               finishes one row's consecutive ids and makes
                               their softmax statistics itself: 0 automatic
                               (default: where the call pairs and 256-row
                               blocks pad at most 1/8 of the rows), 1 always
                               where the call pairs, 2 never.  Whole tiles
                               only (not with SPH_OPT_TC_SCHEDULE = 2).     */
  SPH_OPT_ENDPOINT_Z = 12,  /* where sph_fuse_sample and sph_split_step are
                               not asked for z (fused_logits_out NULL) and
                               run on tensor cores with the inverse-CDF or
                               greedy draw: 0 automatic (default: not stored
                               where the endpoint runs with rows as M, see
                               SPH_OPT_ENDPOINT_ROWS_M; else stored), 1 store
                               z in the scratch arena, 2 never store it.
                               Unstored, the endpoint contraction's epilogue
                               keeps the softmax statistics of every 32-id
                               segment and the draw recomputes z for the 32
                               ids of the segment it lands in (one fp32 dot
                               product of d_l per id, CUDA cores): tokens can
                               differ from the stored path's only where a
                               draw lies within fp32 rounding of a CDF step
                               (or greedy ties within it).                 */
  SPH_OPT_GEMV_QUANTIZE = 14, /* sph_partial_logits on the CUDA-core GEMV
                               (fewer rows than SPH_OPT_TC_MIN_ROWS) where
                               one launch covers every row and rows x n_keep
                               is at most 2^12: 0 (default) the GEMV's last
                               block to finish quantizes the payload itself
                               (no separate pass; the row maxima live in a
                               small buffer of the context that the call
                               leaves cleared); 1 always a separate quantize
                               pass.  Bit-identical codes and scales.      */
  SPH_OPT_SAMPLER = 8       /* the draw of sph_fuse_sample at temperature > 0:
                               0 inverse CDF (default), 1 Gumbel-max: the
                               first index j of the largest
                               z_j / temperature - log(-log u_j), u_j = word
                               j mod 4 of the Philox output for counter
                               (r, 2^31 + j / 4, offset lo, offset hi),
                               ((x >> 9) + 1/2) * 2^-23 (a draw from the same
                               softmax, with other random numbers)         */
} sph_option;

/* Set a tunable (SPH_ERR_INVALID_ARG for an unknown option or a value out of
 * range). */
sph_status sph_set_option(sph_ctx* ctx, sph_option option, int64_t value);

/* Optional device allocation helpers for callers without their own
 * allocator.  sph_buffer_ptr returns the device address (NULL for NULL). */
sph_status sph_buffer_alloc(sph_ctx* ctx, size_t bytes, sph_buffer** out);
sph_status sph_buffer_free(sph_ctx* ctx, sph_buffer* buf);
void* sph_buffer_ptr(const sph_buffer* buf);

/* ---- tracing ----------------------------------------------------------- */

/* Kernel classes whose device time the context can accumulate. */
enum {
  SPH_PROF_CLOUD_GEMM = 0,  /* gathered h_cloud . W_h contraction + epilogue */
  SPH_PROF_QUANTIZE = 1,    /* per-row int8 quantization of the partials    */
  SPH_PROF_LOCAL_GEMM = 2,  /* gathered h_local . W_l contraction + fuse     */
  SPH_PROF_SAMPLE = 3,      /* softmax / inverse-CDF draw                    */
  SPH_PROF_VERIFY = 4,      /* speculative acceptance                        */
  SPH_PROF_PREP = 5,        /* operand preparation (hidden-state splits)     */
  SPH_PROF_CLASSES = 8
};

typedef struct sph_profile {
  double ms[SPH_PROF_CLASSES];       /* summed device time per class (ms)   */
  int64_t calls[SPH_PROF_CLASSES];   /* timed launch groups per class       */
  int64_t launches;                  /* kernels launched while enabled      */
} sph_profile;

/* Start (on != 0; resets the accumulators) or stop tracing.  While on, each
 * kernel group is bracketed by CUDA events on the context's stream; groups
 * launched while the stream is being captured into a CUDA graph are not
 * timed (but are counted in `launches`). */
sph_status sph_profile_enable(sph_ctx* ctx, int on);

/* Wait for the context's stream and return the accumulated figures. */
sph_status sph_profile_read(sph_ctx* ctx, sph_profile* out);

/* ---- host helpers (no device work) ------------------------------------- */

/* Downlink payload of one cloud call (Eq. 21 with b = 8 and no tag,
 * metadata or padding): one int8 code per kept logit plus one fp32 scale
 * per row, i.e. rows*n_keep + 4*rows bytes.  Returns 0 for negative sizes. */
size_t sph_payload_bytes(int64_t rows, int64_t n_keep);

/* Turn the "compact subset mask" of Sec. "Distributed Vocabulary
 * Projection" -- a HOST bitmask of ceil(V/8) bytes, bit (v & 7) of byte
 * v >> 3 set iff id v is kept -- into the sorted HOST id list keep_ids
 * (capacity V entries).  *n_keep receives the count.  Errors: INVALID_ARG
 * (NULL pointers, V < 1, no id set). */
sph_status sph_keep_ids_from_mask(const uint8_t* mask, int64_t V,
                                  int32_t* keep_ids, int64_t* n_keep);

/* Check a HOST copy of a kept-id list against the conventions above:
 * strictly increasing, each in [0, V).  Returns SPH_OK, or
 * SPH_ERR_INVALID_ARG (NULL with n_keep > 0, n_keep < 1, V < 1, or a bad
 * id); *bad_index (if not NULL) receives the first offending position, or
 * -1.  The same check SPH_OPT_CHECK_IDS applies to device lists. */
sph_status sph_check_keep_ids(const int32_t* keep_ids, int64_t n_keep,
                              int64_t V, int64_t* bad_index);

/* The work split a context would choose for one call, without launching
 * anything (for tests and tuning).  `call`: 0 cloud (sph_partial_logits,
 * K = d_h), 1 endpoint (sph_fuse_sample, K = d_l).  gather: 1 for a kept-id
 * subset, 0 for the full vocabulary. */
typedef struct sph_plan {
  int32_t tensor_core;      /* 1: tcgen05 kernel; 0: CUDA-core GEMV        */
  int32_t row_blocks;       /* hidden-state row blocks (tensor core)       */
  int32_t block_rows;       /* rows per row block (a multiple of 16)       */
  int32_t tile_ids;         /* kept ids per vocabulary tile: 128 or 256    */
  int32_t tiles;            /* row blocks x vocabulary tiles               */
  int32_t k_blocks;         /* pipeline stages per tile (hidden dimension) */
  int32_t stages;           /* shared-memory pipeline depth                */
  int32_t grid;             /* persistent CTAs                             */
  int32_t whole_tiles;      /* 1: whole tiles per CTA; 0: stream-K ranges  */
  int32_t planes;           /* hidden-state operand planes (bf16 or e4m3)  */
  int32_t gemv_rows;        /* GEMV: rows per launch (1, 2, 4 or 8)        */
  int32_t pair;             /* 1: CTA pairs (SPH_OPT_TC_PAIR); grid counts
                               CTAs, tile_ids is per CTA (a tile is 256)   */
  int32_t rows_m;           /* endpoint: 1 = hidden-state rows as the MMA's M
                               (SPH_OPT_ENDPOINT_ROWS_M; CTA pairs, 256-row
                               blocks, 256-id tiles)                       */
  int32_t epilogue_stats;   /* endpoint: 1 = the softmax statistics of each
                               32-id segment come from the contraction's
                               epilogue, 0 = from a pass over z            */
} sph_plan;
sph_status sph_plan_query(sph_ctx* ctx, int call, int64_t rows, int64_t n_keep,
                          int64_t K, sph_dtype w_dtype, sph_act_mode act_mode,
                          int gather, sph_plan* out);

/* ---- the hot path ------------------------------------------------------ */

/* Cloud call (Eq. 12 over V_l, "after clipping, quantization" in Sec.
 * "Distributed Vocabulary Projection", Eq. 18 with b = 8, Eq. 21):
 *   y[r, j]      = sum_{c < d_h} h_cloud[r, c] * W_h[keep_ids[j], c]
 *                  (+ bias[keep_ids[j]])            fp32 accumulate
 *   yc           = min(max(y, -clip), clip)
 *   row_scale[r] = max_j |yc[r, j]| / 127   (fp32; 0 for an all-zero row)
 *   codes[r, j]  = round-half-even(yc / row_scale[r]) in [-127, 127]
 *                  (the kernels multiply yc by the correctly rounded fp32
 *                  reciprocal of row_scale[r] and round that product once,
 *                  so a code can differ by one from the exact quotient's
 *                  rounding only where that quotient lies within about
 *                  1e-5 of a half-integer)
 * Arguments
 *   h_cloud  fp32 [rows, d_h] with row stride ld_h (>= d_h); typically the
 *            slice h[:, d_l:] of the full hidden state (ld_h = d).
 *   W_h      [V, d_h] row-major, row stride ld_w (>= d_h) elements of
 *            w_dtype; vocabulary-major, i.e. W_cloud of Eq. 10 transposed.
 *            ld_w*element size and the base address must be multiples of 16
 *            bytes.
 *   w_row_scale  fp32 [V] for SPH_DTYPE_FP8_E4M3, else NULL.
 *   bias     fp32 [V] or NULL; applied once, here (Eq. 12).
 *   keep_ids int32 [n_keep] (see conventions) or NULL with n_keep == V.
 *   clip     > 0 and finite.
 *   act_mode SPH_ACT_FP32 or SPH_ACT_BF16.
 *   codes    int8 [rows, n_keep] (out), row_scale fp32 [rows] (out).
 *   partial_out  fp32 [rows, n_keep] unclipped y (out), or NULL.
 *   payload_bytes  host size_t (out) = sph_payload_bytes(rows, n_keep), or
 *            NULL.
 * Preconditions: rows >= 1, d_h >= 1, 1 <= n_keep <= V, finite inputs.
 * Errors: INVALID_ARG, UNSUPPORTED, CUDA, OOM. */
sph_status sph_partial_logits(sph_ctx* ctx,
                              const float* h_cloud, int64_t rows, int64_t ld_h,
                              const void* W_h, sph_dtype w_dtype, int64_t V,
                              int64_t d_h, int64_t ld_w,
                              const float* w_row_scale, const float* bias,
                              const int32_t* keep_ids, int64_t n_keep,
                              float clip, sph_act_mode act_mode,
                              int8_t* codes, float* row_scale,
                              float* partial_out, size_t* payload_bytes);

/* Allocation-free cloud call.  The paper has no counterpart: this is a
 * deployment variant of sph_partial_logits for callers that cannot allocate
 * device memory when they run the cloud step (an allocator owned or locked
 * by another runtime, a fixed-size memory pool, or a serving loop that must
 * never call cudaMalloc, which can synchronise the device).  Such callers
 * cannot create a context, so this call takes the device and stream
 * directly and, once set up on a device (see the first call below),
 * allocates nothing: no cudaMalloc, no cudaFree, no allocating library
 * routine.  Its scratch (clipped fp32 partials and per-row maxima) lives in
 * one fixed device array of SPH_NOALLOC_SCRATCH_BYTES inside the library,
 * which every GPU that has loaded the library's modules holds until the
 * process exits.
 *   - Same arguments, results and errors as sph_partial_logits, plus
 *     `device` (made current for the call), `cuda_stream` (a cudaStream_t,
 *     NULL = legacy default stream) and an optional host buffer err_msg of
 *     err_msg_len bytes that receives a description of any failure.
 *   - Size limit: round_up(rows*n_keep*4, 256) + round_up(rows*4, 256) must
 *     not exceed SPH_NOALLOC_SCRATCH_BYTES; larger calls return
 *     SPH_ERR_UNSUPPORTED without launching anything.
 *   - rows is at most 2^20 (INVALID_ARG beyond), as for sph_partial_logits.
 *   - The call always runs the CUDA-core GEMV, which re-reads the kept W
 *     rows once per 8 hidden-state rows: it is meant for few rows.
 *   - The first call on a device is a set-up call: it looks up the array's
 *     device address (cudaGetSymbolAddress, with that device current), and
 *     under CUDA's lazy module loading (the default) it is also the moment
 *     the library's modules -- the array among them -- are loaded onto that
 *     device, which allocates device memory and may synchronise.  Make one
 *     warm-up call per device before entering the region where nothing may
 *     allocate, and before any stream capture.  Later calls allocate
 *     nothing.
 *   - All calls share the one array and it keeps the last call's contents
 *     (the row maxima are cleared by each call).  Calls whose kernels overlap
 *     on the GPU -- on different streams or from different host threads --
 *     race and corrupt each other's results; serialise them. */
#define SPH_NOALLOC_SCRATCH_BYTES ((size_t)8 << 20)
sph_status sph_partial_logits_noalloc(int device, void* cuda_stream,
                                      const float* h_cloud, int64_t rows,
                                      int64_t ld_h, const void* W_h,
                                      sph_dtype w_dtype, int64_t V,
                                      int64_t d_h, int64_t ld_w,
                                      const float* w_row_scale,
                                      const float* bias,
                                      const int32_t* keep_ids, int64_t n_keep,
                                      float clip, sph_act_mode act_mode,
                                      int8_t* codes, float* row_scale,
                                      float* partial_out,
                                      size_t* payload_bytes, char* err_msg,
                                      size_t err_msg_len);

/* Endpoint call (Eq. 11, Eq. 13, Eq. 14, Eq. 15; Algorithm 1 "fuses partial
 * logits, applies language masking, and samples"):
 *   z[r, j]   = codes[r, j] * row_scale[r]
 *               + sum_{c < d_l} h_local[r, c] * W_l[keep_ids[j], c]
 *   p[r, :]   = softmax(z[r, :] / temperature) over the kept ids (ids
 *               outside V_l have z = -inf, i.e. probability 0)
 *   tokens[r] = keep_ids[j*], j* = the first j whose ascending-order CDF
 *               exceeds u_r, u_r = Philox4x32-10 uniform with key = seed and
 *               counter (r, 0, offset lo, offset hi), u = (x0 >> 8) * 2^-24
 *   temperature 0 is greedy decoding (the argmax decoding of Eq. 17):
 *   tokens[r] = keep_ids[j*], j* = the first j with the largest z[r, j]
 *   (the lowest kept id on ties); no uniform is drawn.
 * Arguments
 *   codes int8 [rows, n_keep], row_scale fp32 [rows]: the cloud payload;
 *   both NULL for no payload (z is the local partial alone: with the whole
 *   hidden state and head, d_l = d, this is the unsplit head of Eq. 9, the
 *   comparator of the paper's "no split projection" ablation).  Exactly one
 *   of them NULL is INVALID_ARG.
 *   h_local fp32 [rows, d_l], row stride ld_hl (the slice h[:, :d_l]).
 *   W_l bf16 [V, d_l] row-major with row stride ld_wl; the base address
 *   and ld_wl*2 must be multiples of 16 bytes.
 *   keep_ids as for sph_partial_logits.  temperature >= 0 and finite.
 *   tokens int32 [rows] (out, vocabulary ids), or NULL: z alone (fuse,
 *   Eq. 13, and mask), no softmax statistics and no draw -- the form for
 *   target rows that go to sph_verify_draft, which makes the statistics
 *   and draws the next tokens itself; fused_logits_out is then required.
 *   fused_logits_out fp32 [rows, n_keep] z before the division by
 *   temperature (out), or NULL.
 * Errors: INVALID_ARG, UNSUPPORTED, CUDA, OOM. */
sph_status sph_fuse_sample(sph_ctx* ctx,
                           const int8_t* codes, const float* row_scale,
                           int64_t rows,
                           const float* h_local, int64_t ld_hl,
                           const void* W_l, int64_t V, int64_t d_l,
                           int64_t ld_wl,
                           const int32_t* keep_ids, int64_t n_keep,
                           float temperature, uint64_t seed, uint64_t offset,
                           int32_t* tokens, float* fused_logits_out);

/* The whole split step in one call, from the full hidden state to tokens:
 * the cloud call followed by the endpoint call (Eqs. 11-15, Eq. 18;
 * Algorithm 1, the cloud's partial projection and the endpoint's fusion and
 * sampling), on one GPU, with the payload that would cross between them
 * (Eq. 21) written out.  It is the single-GPU form of the paper's split
 * projection, the counterpart of the unsplit head that sph_fuse_sample
 * computes without a payload (Sec. "Ablation Study").
 *   h        fp32 [rows, d_l + d_h], row stride ld_h: h[:, :d_l] is the
 *            endpoint's part, h[:, d_l:] the cloud's (Eq. 10).
 *   W_h, w_dtype, w_row_scale, ld_wh, bias, keep_ids, n_keep, clip,
 *   act_mode  as for sph_partial_logits;  W_l, ld_wl  as for
 *            sph_fuse_sample;  temperature, seed, offset  as there too (the
 *            draw is the same: purpose 0 of row r).
 *   chunk    kept ids per payload chunk.  0 (or >= n_keep): one chunk, the
 *            payload of sph_partial_logits (one scale per row); for small
 *            payloads the endpoint's contraction then quantizes the cloud's
 *            clipped partials in its own epilogue, so no separate
 *            quantization pass runs (SPH_OPT_SPLIT_QUANTIZE).
 *            1 <= chunk < n_keep: block streaming (the GPU form of
 *            the paper's block-wise streaming in Sec. "Device-Adaptive
 *            Feature Preparation"): chunk q holds the ids
 *            q*chunk .. min(n_keep, (q+1)*chunk) - 1 and carries its own
 *            row scales, scale[q][r] = max over the chunk of |clipped y| /
 *            127 (Eq. 18 applied per chunk); the cloud emits chunk q on the
 *            context's stream while the endpoint fuses chunk q - 1 on
 *            endpoint_stream (the SMs are divided between the two in
 *            proportion to d_l : d_h).
 *   endpoint_stream  a cudaStream_t other than the context's, or NULL for
 *            one the context creates on first use and owns; used only when
 *            there is more than one chunk.  The call's work is complete, on
 *            the context's stream, when the endpoint's is.  The context's
 *            own stream runs the chunks one after another instead, each
 *            kernel with every SM (the same results, without the overlap).
 *   codes    int8, rows * n_keep bytes (out), chunk-major: chunk q is the
 *            row-major [rows][its ids] block starting at byte
 *            q * chunk * rows.  One chunk: [rows, n_keep].
 *   scales   fp32 [nchunk][rows] (out), nchunk = ceil(n_keep / chunk).
 *   tokens   int32 [rows] (out) vocabulary ids;  fused_logits_out fp32
 *            [rows, n_keep] z (out), or NULL.
 *   payload_bytes  host (out), or NULL: rows * n_keep + 4 * rows * nchunk.
 * Errors: INVALID_ARG, UNSUPPORTED, CUDA, OOM. */
sph_status sph_split_step(sph_ctx* ctx, const float* h, int64_t rows,
                          int64_t ld_h, int64_t d_l, int64_t d_h,
                          const void* W_h, sph_dtype w_dtype,
                          const float* w_row_scale, int64_t ld_wh,
                          const void* W_l, int64_t ld_wl, int64_t V,
                          const float* bias, const int32_t* keep_ids,
                          int64_t n_keep, float clip, sph_act_mode act_mode,
                          float temperature, uint64_t seed, uint64_t offset,
                          int64_t chunk, void* endpoint_stream,
                          int8_t* codes, float* scales, int32_t* tokens,
                          float* fused_logits_out, size_t* payload_bytes);

/* Cloud verification of speculative drafts (Sec. "Endpoint Speculative
 * Decoding and Cloud Verification", Algorithm 1; standard speculative
 * sampling as in the works the paper cites).  Per session s:
 *   p_i = softmax(target_logits[s*(k+1)+i, :] / temperature), i = 0..k
 *   for i < k: accept draft x_i iff r_i * q_i(x_i) < p_i(x_i), with
 *     r_i = Philox uniform of counter (s, 1+i, offset lo, offset hi);
 *   at the first rejection draw from max(0, p_i - q_i) renormalised (p_i if
 *   that is all zero); if all k are accepted draw from p_k; the draw uses
 *   the uniform of counter (s, 1+k, ...) and the inverse CDF in ascending
 *   id order.
 *   temperature 0 is greedy verification (the limit of the rule above with
 *   ties to the lowest id): with a_i the first argmax of row i, drafts are
 *   accepted while x_i == a_i and the next token is a_i at the first
 *   mismatch, or a_k; draft_probs is not read and no uniform is drawn.
 * Arguments
 *   target_logits fp32 [sessions*(k+1), n_keep] compacted fused logits.
 *   draft_tokens int32 [sessions, k] vocabulary ids (an id outside V_l has
 *   p = q = 0 and is rejected).
 *   draft_probs fp32 [sessions, k, n_keep] compacted q, or NULL for greedy
 *   (one-hot) drafts, where q_i(x) = [x == x_i].
 *   n_accepted int32 [sessions] (out) in [0, k]; next_token int32
 *   [sessions] (out): the drawn vocabulary id.
 * Preconditions: sessions >= 1, k >= 1, temperature >= 0 and finite.
 * Errors: INVALID_ARG, UNSUPPORTED, CUDA, OOM. */
sph_status sph_verify_draft(sph_ctx* ctx,
                            const float* target_logits, int64_t sessions,
                            int64_t k,
                            const int32_t* keep_ids, int64_t n_keep,
                            float temperature,
                            const int32_t* draft_tokens,
                            const float* draft_probs,
                            uint64_t seed, uint64_t offset,
                            int32_t* n_accepted, int32_t* next_token);

#ifdef __cplusplus
}  /* extern "C" */
#endif

#endif  /* SPH_H_ */
