// Tensor-core gathered contraction for the many-row regime (Eq. 11 / Eq. 12
// over the kept vocabulary ids), tcgen05 + TMEM on sm_103a.
//
// Swap-AB: the MMA's M dimension is a block of 128 gathered vocabulary rows
// (operand A), its N dimension a block of BN hidden-state rows (operand B),
// and K runs over the hidden dimension in 128-byte atoms (64 bf16 or 128
// e4m3 elements) laid out with the 128-byte swizzle.  A tile is 128 or 256
// vocabulary rows; a 256-row tile is two M = 128 MMAs sharing every B stage.
//
// Hidden states: fp32 h is split beforehand into bf16 hi + lo planes
// (h = hi + lo + O(2^-18 |h|)) that multiply the same W tile into one fp32
// TMEM accumulator, so W is read once and the result keeps fp32 accuracy;
// bf16-activation mode uses hi alone.  With fp8 (e4m3) weights the raw e4m3
// rows are the A operand of kind::f8f6f4 MMAs against e4m3 planes of h
// under a per-row power-of-two scale (four planes: 2^-13 of |h|; two
// reproduce bf16-rounded h), all into one accumulator; the epilogue applies
// the row's scale and the weight row's scale.
//
// Operand A comes from W by TMA 2-D tile copies, one per atom:
//   full vocabulary : one box of 128 rows per atom (or one 3-D copy of all
//                     the stage's atoms when the width allows);
//   kept-id subset  : the tile's kept ids are cut into runs of consecutive
//                     vocabulary ids and every run is one box of exactly its
//                     length (one tensor map per height 1..128), written at
//                     its row of the tile; language subsets are mostly long
//                     runs, so a 128-id tile takes about two boxes.
// Operand B (the h planes, L2-resident) comes by one 3-D TMA copy per plane.
//
// Work split: the (row block, vocabulary tile, k-block) iterations -- row
// blocks outermost, so that CTA c and CTA c + G/RB work on the same W rows
// at the same time and one of the two reads them from L2 -- are cut into
// one contiguous range per persistent CTA (one CTA per SM): whole tiles, or
// stream-K ranges when that balances better.  A tile whose k-range spans
// CTAs is finished by a designated contributor (the last to reach it in
// time), which adds the others' stored fp32 partials in CTA order after a
// bounded poll for them; if the poll runs out it counts in like the others
// and the last to count in finishes the tile.  The order of the sum is fixed
// either way, so results are deterministic.
//
// Warp roles: warp 0 issues the TMA copies, warp 1 owns TMEM and issues
// tcgen05.mma (one thread), warps 2-9 drain the accumulator (double-buffered,
// or single for 256-row tiles over more than 128 rows) with tcgen05.ld and
// run the fused epilogue -- two warps per TMEM lane quadrant, so that the
// epilogue's dependent shuffle / exp chains of one warp overlap with the
// other's.  Every wait is bounded; a wait that gives up sets the context's
// error word and the CTA winds down after its copies and MMAs have landed.
//
// Epilogues: cloud = + bias, optional unclipped store, clip, store, row |max|
// (atomicMax); endpoint = + code * row_scale (Eq. 13), store z, and the
// softmax statistics (max, sum of exp((z - max)/tau)) of every 32-id segment
// of every row, which the sampler uses instead of re-reading the row.
#include <cuda.h>
#include <cuda_fp8.h>
#include <cuda_runtime.h>

#include <atomic>
#include <mutex>

#include "sm100_ptx.cuh"
#include "sph_common.cuh"
#include "sph_internal.h"

namespace sph {
namespace {

constexpr int kTileM = 128;          // vocabulary rows per MMA (M); a tile is 1 or 2 of them
constexpr int kAtomK = 64;           // bf16 elements per 128-byte swizzle atom
constexpr int kAtomBytes = kTileM * kAtomK * 2;   // one A atom: 128 rows x 128 B
constexpr int kMaxBN = 256;
constexpr int kMaxStages = 12;       // (the barriers, 2 * 12 + 5 words and two more, fit
                                     // the 512-byte area)
constexpr int kBarrierArea = 512;
// the endpoint epilogue's transpose tiles: per epilogue warp 8 rows x 32 ids
// (+4 words of padding per row, so that both the row writes and the 16-byte
// reads are free of bank conflicts)
constexpr int kTRow = 36;
constexpr float kLog2eF = 1.4426950408889634f;   // exp(d / tau) = 2^(d log2(e) / tau)
// Kernel instantiations of EPI_ENDPOINT that finish through the per-warp
// shared-memory transpose (finish_chunk_t) rather than per lane.
constexpr int EPI_ENDPOINT_T = 3;
// Rows-as-M instantiations of EPI_ENDPOINT and EPI_FUSED (CTA pairs only):
// the MMA's M dimension is the hidden-state rows (A = the h planes, 128 rows
// per CTA) and N the tile's 256 ids (B = the gathered weight rows, 128 per
// CTA), so each epilogue lane holds one row and 32 consecutive ids per
// accumulator load.
constexpr int EPI_ENDPOINT_RM = 4;
constexpr int EPI_FUSED_RM = 5;
constexpr int kTransposeBytes = 8 /* epilogue warps */ * 8 * kTRow * 4;
constexpr size_t kSmemBudget = 220 * 1024;
constexpr long long kDrainLimit = 1ll << 31;   // cycles, for in-flight copies
constexpr int kMaxDevices = 64;      // per-device launch attribute cache

constexpr int kEpiWarps = 8;         // two per TMEM lane quadrant
static_assert(kTransposeBytes == kEpiWarps * 8 * kTRow * 4, "transpose tiles per warp");
constexpr int kEpiGroups = kEpiWarps / 4;
constexpr int kThreads = 64 + 32 * kEpiWarps;       // producer, MMA, epilogue
constexpr int kAtomE8 = 128;         // e4m3 elements per 128-byte atom
constexpr int kBoxHeights = 128;     // row boxes of 1, 2, 3, ..., 128 rows (map h-1)
constexpr int kMaxBoxes = 260;       // row boxes of one tile (one per run, two per
                                     // run longer than 128 rows in a 256-row tile)

// W tensor maps: box height 2^i rows for map i (64 columns each).
struct WMaps {
  CUtensorMap m[kBoxHeights];
  CUtensorMap a3;              // full vocabulary: (element, row, atom) view, all atoms of a stage
};

struct TcParams {
  int R, n, K, KB, NT, RB, BN, Rp, stages, whole_tiles;
  int nseg;                    // endpoint statistics: 32-id segments per row (NT * TM / 32)
  int na;                      // swizzle atoms per k-block (k-block = 64 * na)
  long long T;                 // total iterations RB * NT * KB
  const int32_t* ids;          // gather path: sorted ids
  const float* h_scale;        // fp8 path: per h-row power-of-two scale of the planes
  int64_t ld_w;
  const float* w_scale;        // fp8 path: per-vocabulary-row scale
  int epilogue;
  const float* bias;
  float clip;
  float* partial_out;
  float* Y;
  unsigned* rowmax;
  const int8_t* codes;
  const float* row_scale;
  float inv_tau;
  int64_t ldy;                 // row stride of Y (endpoint: z) in elements
  const float* yc;             // fused endpoint: the cloud's clipped partials [R][n]
  const unsigned* rowmax_in;   // fused endpoint: their row |max| bits [R]
  int8_t* codes_out;           // fused endpoint: the payload codes [R][n] (out)
  float* scale_out;            // fused endpoint: the row scales [R] (out)
  float2* seg_stats;           // endpoint: [R][nseg] (max, sum exp)
  int a3d;                     // full vocabulary: A by one 3-D copy per stage
  int single_acc;              // one accumulator (no epilogue overlap): 256-id tiles of > 128 rows
  float* P;                    // split-tile partials [2 * grid][BN][TM]
  int* counters;               // [tiles][4 quadrants][epilogue groups], zero between calls
  unsigned* status;
  long long spin_limit;
  long long finish_wait;       // split-tile finisher poll bound (cycles); 0: no finisher
};

__device__ __forceinline__ long long cta_of(long long i, long long T, int G) {
  return ((i + 1) * G + T - 1) / T - 1;    // owner of iteration i (split mode)
}

// First iteration of CTA c.
__device__ __forceinline__ long long range_start(const TcParams& p, long long c, int G) {
  if (p.whole_tiles) return (c * (long long)(p.RB * p.NT) / G) * p.KB;
  return c * p.T / G;
}

// Walks the (tile, k-block range) segments of one CTA's iteration range.
struct Segments {
  long long it, end;
  int KB;
  __device__ bool next(int& tile, int& kb0, int& kb1) {
    if (it >= end) return false;
    tile = (int)(it / KB);
    kb0 = (int)(it - (long long)tile * KB);
    const long long rem = end - it;
    kb1 = (int)min((long long)KB, kb0 + rem);
    it += kb1 - kb0;
    return true;
  }
};


// Endpoint payload of one 16-row chunk at this lane's id column j: the int8
// codes of rows row0..row0+15 (as floats) and, in lane q < 16, the scale of
// row row0 + q.  The fused endpoint loads the cloud's clipped fp32 partials
// instead, and the quantizer's lift and reciprocal of the row scale.
// Addresses are clamped into the arrays and every load is issued, so the 16
// loads go out back to back and can be started a chunk ahead of their use.
struct Payload {
  float c[16];
  float s;
  float k, inv;                        // fused endpoint only
};
template <int EPI>
__device__ __forceinline__ void load_payload(const TcParams& p, int row0, int j, int lane,
                                             Payload& pl) {
  if constexpr (EPI == EPI_FUSED) {
    const float* col = p.yc + min(j, p.n - 1);
#pragma unroll
    for (int q = 0; q < 16; ++q) pl.c[q] = __ldcg(col + (int64_t)min(row0 + q, p.R - 1) * p.n);
    const RowQuant rq = row_quant(__ldcg(p.rowmax_in + min(row0 + (lane & 15), p.R - 1)));
    pl.s = rq.s;
    pl.k = rq.k;
    pl.inv = rq.inv;
    return;
  }
  if (!p.codes) {                      // no payload: z is the local partial alone
#pragma unroll
    for (int q = 0; q < 16; ++q) pl.c[q] = 0.f;
    pl.s = 0.f;
    return;
  }
  const int8_t* col = p.codes + min(j, p.n - 1);
#pragma unroll
  for (int q = 0; q < 16; ++q) pl.c[q] = (float)__ldg(col + (int64_t)min(row0 + q, p.R - 1) * p.n);
  pl.s = __ldg(p.row_scale + min(row0 + (lane & 15), p.R - 1));
}
// Warm L2 with the payload of rows row0..row0+nrows-1 at the 32 ids from j0
// (the codes, or for the fused endpoint the clipped partials).
template <int EPI>
__device__ __forceinline__ void prefetch_payload(const TcParams& p, int row0, int nrows, int j0,
                                                 int lane) {
  const int esz = EPI == EPI_FUSED ? 4 : 1;
  const char* base = EPI == EPI_FUSED ? reinterpret_cast<const char*>(p.yc)
                                      : reinterpret_cast<const char*>(p.codes);
  if (j0 >= p.n || !base) return;
  const int last = min(31, p.n - 1 - j0) * esz;
  for (int r = row0 + lane; r < min(row0 + nrows, p.R); r += 32) {
    const char* a = base + ((int64_t)r * p.n + j0) * esz;
    asm volatile("prefetch.global.L2 [%0];" ::"l"(a));
    asm volatile("prefetch.global.L2 [%0];" ::"l"(a + last));
  }
}

// Epilogue of 16 accumulator columns (hidden-state rows row0..row0+15) for
// this lane's vocabulary column j (endpoint: with the chunk's payload).
template <int EPI>
__device__ __forceinline__ void finish_chunk(const TcParams& p, const float (&v)[16],
                                             int row0, int j, bool vj, int id,
                                             int lane, int seg, const Payload& pay) {
  const int kr = (lane >> 1) & 15;               // the row this lane reduces
  if constexpr (EPI == EPI_CLOUD) {
    const float b = (vj && p.bias) ? p.bias[id] : 0.f;
    // fp8 weights: the product of raw e4m3 codes and h's scaled planes,
    // times the weight row's scale and (below) the h row's scale
    const float ws = (vj && p.w_scale) ? p.w_scale[id] : 1.0f;
    float m[16];
#pragma unroll
    for (int q = 0; q < 16; ++q) {
      const int r = row0 + q;
      m[q] = 0.f;
      if (vj && r < p.R) {
        const float y = (p.h_scale ? v[q] * __ldg(p.h_scale + r) : v[q]) * ws + b;
        const int64_t o = (int64_t)r * p.n + j;
        if (p.partial_out) p.partial_out[o] = y;
        const float yc = fminf(fmaxf(y, -p.clip), p.clip);
        p.Y[o] = yc;
        m[q] = fabsf(yc);
      }
    }
    const float mr = warp_reduce_scatter16(m, MaxOp{}, lane);
    if (!(lane & 1) && row0 + kr < p.R && mr > 0.f)
      atomicMax(&p.rowmax[row0 + kr], __float_as_uint(mr));
  } else {
    float z[16];
#pragma unroll
    for (int q = 0; q < 16; ++q) {
      const float sq = __shfl_sync(0xFFFFFFFFu, pay.s, q);
      float cq = pay.c[q];
      if constexpr (EPI == EPI_FUSED) {
        // quantize the cloud's clipped partial (Eq. 18) exactly as the
        // quantize kernel does, emit the code, and dequantize it (Eq. 13)
        const float kq = __shfl_sync(0xFFFFFFFFu, pay.k, q);
        const float iq = __shfl_sync(0xFFFFFFFFu, pay.inv, q);
        const int code = quantize_one(cq, kq, iq);
        if (vj && row0 + q < p.R) p.codes_out[(int64_t)(row0 + q) * p.n + j] = (int8_t)code;
        cq = (float)code;
      }
      z[q] = (vj && row0 + q < p.R) ? v[q] + cq * sq : -INFINITY;
    }
    if constexpr (EPI == EPI_FUSED) {
      // the warp holding the first 32 ids emits the 16 rows' scales
      if (j == lane && lane < 16 && row0 + lane < p.R) p.scale_out[row0 + lane] = pay.s;
    }
#pragma unroll
    for (int q = 0; q < 16; ++q) {
      const int r = row0 + q;
      if (p.Y && vj && r < p.R) p.Y[(int64_t)r * p.ldy + j] = z[q];
    }
    if (!p.seg_stats) return;          // statistics come from a pass over z
    // softmax statistics of this 32-id segment for each row: the maxima,
    // spread back to every lane, then the sums of exp((z - max) / tau)
    const float mk = warp_reduce_scatter16(z, MaxOp{}, lane);
    float e[16];
#pragma unroll
    for (int q = 0; q < 16; ++q) {
      const float mq = __shfl_sync(0xFFFFFFFFu, mk, 2 * q);
      e[q] = (vj && row0 + q < p.R) ? ex2_approx((z[q] - mq) * (p.inv_tau * kLog2eF)) : 0.f;
    }
    const float sk = warp_reduce_scatter16(e, SumOp{}, lane);
    if (!(lane & 1) && row0 + kr < p.R)
      p.seg_stats[(int64_t)(row0 + kr) * p.nseg + seg] = make_float2(mk, sk);
  }
}

// Endpoint epilogue through this warp's shared-memory tile `tb` [8][kTRow]
// (Eq. 13: z = code * s + local partial): the 16 rows of a chunk go in two
// halves of 8; after the transpose lane l holds row (l >> 2) of the half and
// the 8 consecutive ids 8 (l & 3) .. + 7 of the warp's 32, so its payload is
// one 8-byte load and its z two 16-byte stores (narrower where a row is less
// aligned), instead of 16 one-byte loads and 16 strided stores per lane, and
// the 32-id segment statistics of a row are a reduction over four lanes.
// Used when rows of codes (and of z, where z is stored) are 2-element
// aligned.  The payload of a chunk does not depend on the accumulator, so it
// is loaded a chunk ahead (TPay).
struct TPay {
  uint2 cw[2];     // the 8 codes of this lane's row and ids, per half
  float sc[2];     // that row's scale, per half (0 past the rows)
};
__device__ __forceinline__ void load_tpay(const TcParams& p, int row0, int j0w, int lane,
                                          TPay& t) {
  const int q = lane >> 2, seg = lane & 3;
#pragma unroll
  for (int h8 = 0; h8 < 2; ++h8) {
    t.cw[h8] = make_uint2(0u, 0u);
    t.sc[h8] = 0.f;
    const int r = row0 + h8 * 8 + q;
    const int j = j0w + 8 * seg;
    if (!p.codes || r >= p.R || j >= p.n) continue;
    t.sc[h8] = __ldg(p.row_scale + r);
    const int8_t* cp = p.codes + (int64_t)r * p.n + j;     // 2-byte aligned
    const uintptr_t ca = reinterpret_cast<uintptr_t>(cp);
    if (j + 8 <= p.n) {
      if ((ca & 7) == 0) {
        t.cw[h8] = __ldg(reinterpret_cast<const uint2*>(cp));
      } else if ((ca & 3) == 0) {
        t.cw[h8].x = __ldg(reinterpret_cast<const unsigned*>(cp));
        t.cw[h8].y = __ldg(reinterpret_cast<const unsigned*>(cp) + 1);
      } else {
        const unsigned short* hp = reinterpret_cast<const unsigned short*>(cp);
        t.cw[h8].x = (unsigned)__ldg(hp) | ((unsigned)__ldg(hp + 1) << 16);
        t.cw[h8].y = (unsigned)__ldg(hp + 2) | ((unsigned)__ldg(hp + 3) << 16);
      }
    } else {                                   // the row's last ids
      unsigned w[2] = {0u, 0u};
#pragma unroll
      for (int e = 0; e < 8; ++e)
        if (j + e < p.n) w[e >> 2] |= ((unsigned)(uint8_t)__ldg(cp + e)) << (8 * (e & 3));
      t.cw[h8] = make_uint2(w[0], w[1]);
    }
  }
}
__device__ __forceinline__ void finish_chunk_t(const TcParams& p, const float (&v)[16], int row0,
                                               int j0w, int lane, float* tb, const TPay& pay) {
  const int q = lane >> 2, seg = lane & 3;
#pragma unroll
  for (int h8 = 0; h8 < 2; ++h8) {
#pragma unroll
    for (int k = 0; k < 8; ++k) tb[k * kTRow + lane] = v[h8 * 8 + k];
    __syncwarp();
    const float4 a = *reinterpret_cast<const float4*>(tb + q * kTRow + 8 * seg);
    const float4 b = *reinterpret_cast<const float4*>(tb + q * kTRow + 8 * seg + 4);
    __syncwarp();
    const int r = row0 + h8 * 8 + q;
    const int j = j0w + 8 * seg;
    const bool rv = r < p.R;
    float x[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
    const float sc = pay.sc[h8];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      x[e] += (float)(int8_t)((pay.cw[h8].x >> (8 * e)) & 0xFF) * sc;
      x[4 + e] += (float)(int8_t)((pay.cw[h8].y >> (8 * e)) & 0xFF) * sc;
    }
    if (p.Y && rv && j < p.n) {
      float* zp = p.Y + (int64_t)r * p.ldy + j;               // 8-byte aligned
      if (j + 8 <= p.n && (reinterpret_cast<uintptr_t>(zp) & 15) == 0) {
        reinterpret_cast<float4*>(zp)[0] = make_float4(x[0], x[1], x[2], x[3]);
        reinterpret_cast<float4*>(zp)[1] = make_float4(x[4], x[5], x[6], x[7]);
      } else if (j + 8 <= p.n) {
#pragma unroll
        for (int e = 0; e < 4; ++e)
          reinterpret_cast<float2*>(zp)[e] = make_float2(x[2 * e], x[2 * e + 1]);
      } else {
#pragma unroll
        for (int e = 0; e < 8; ++e)
          if (j + e < p.n) zp[e] = x[e];
      }
    }
    if (p.seg_stats) {
      // this row's 32-id segment: (max z, sum of exp((z - max) / tau)) over
      // its ids below n, from the four lanes that hold it
#pragma unroll
      for (int e = 0; e < 8; ++e)
        if (!rv || j + e >= p.n) x[e] = -INFINITY;
      float m = fmaxf(fmaxf(fmaxf(x[0], x[1]), fmaxf(x[2], x[3])),
                      fmaxf(fmaxf(x[4], x[5]), fmaxf(x[6], x[7])));
      m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, 1));
      m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, 2));
      float sum = 0.f;
      if (m > -INFINITY) {
#pragma unroll
        for (int e = 0; e < 8; ++e) sum += ex2_approx((x[e] - m) * (p.inv_tau * kLog2eF));  // 2^-inf = 0
      }
      sum += __shfl_xor_sync(0xFFFFFFFFu, sum, 1);
      sum += __shfl_xor_sync(0xFFFFFFFFu, sum, 2);
      if (seg == 0 && rv) p.seg_stats[(int64_t)r * p.nseg + (j0w >> 5)] = make_float2(m, sum);
    }
  }
}

// ---- rows-as-M endpoint epilogue -----------------------------------------
// This lane's row r and one 32-id segment j0 .. j0 + 31 of the tile.  The
// codes of the segment (32 bytes of row r), loaded before the tile's
// accumulator is ready.
struct RPay {
  uint4 c[2];
};
__device__ __forceinline__ void load_rpay(const TcParams& p, int r, int j0, RPay& q) {
  q.c[0] = q.c[1] = make_uint4(0u, 0u, 0u, 0u);
  if (!p.codes || r >= p.R || j0 >= p.n) return;
  const int8_t* cp = p.codes + (int64_t)r * p.n + j0;
  const uintptr_t a = reinterpret_cast<uintptr_t>(cp);
  if (j0 + 32 <= p.n && (a & 15) == 0) {
    q.c[0] = __ldg(reinterpret_cast<const uint4*>(cp));
    q.c[1] = __ldg(reinterpret_cast<const uint4*>(cp) + 1);
    return;
  }
  unsigned w[8];
  if (j0 + 32 <= p.n && (a & 3) == 0) {
#pragma unroll
    for (int e = 0; e < 8; ++e) w[e] = __ldg(reinterpret_cast<const unsigned*>(cp) + e);
  } else {
    const int cnt = min(32, p.n - j0);
#pragma unroll
    for (int e = 0; e < 8; ++e) w[e] = 0u;
#pragma unroll
    for (int e = 0; e < 32; ++e)
      if (e < cnt) w[e >> 2] |= ((unsigned)(uint8_t)__ldg(cp + e)) << (8 * (e & 3));
  }
  q.c[0] = make_uint4(w[0], w[1], w[2], w[3]);
  q.c[1] = make_uint4(w[4], w[5], w[6], w[7]);
}
__device__ __forceinline__ unsigned rpay_word(const RPay& q, int w) {
  const uint4 u = q.c[w >> 2];
  return (w & 3) == 0 ? u.x : (w & 3) == 1 ? u.y : (w & 3) == 2 ? u.z : u.w;
}
// Finish the segment (Eq. 13): z = v + code * s, stored where asked; with the
// fused endpoint the codes are first quantized from the cloud's clipped
// partials (Eq. 18) and written out; the segment's softmax statistics
// (max z, sum of exp((z - max) / tau) over its ids below n) where asked.
template <int EPI>
__device__ __forceinline__ void finish_rm(const TcParams& p, float (&v)[32], int r, int j0,
                                          const RPay& q, const RowQuant& rq) {
  const bool rv = r < p.R;
  const int cnt = rv ? max(0, min(32, p.n - j0)) : 0;   // this row's ids in the segment
  const bool full = cnt == 32;
  if constexpr (EPI == EPI_FUSED_RM) {
    if (cnt > 0) {
      const float* yp = p.yc + (int64_t)r * p.n + j0;
      float y[32];
      if (full && (reinterpret_cast<uintptr_t>(yp) & 15) == 0) {
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const float4 t = __ldcg(reinterpret_cast<const float4*>(yp) + e);
          y[4 * e] = t.x; y[4 * e + 1] = t.y; y[4 * e + 2] = t.z; y[4 * e + 3] = t.w;
        }
      } else {
#pragma unroll
        for (int e = 0; e < 32; ++e) y[e] = e < cnt ? __ldcg(yp + e) : 0.f;
      }
      unsigned w[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) w[e] = 0u;
#pragma unroll
      for (int e = 0; e < 32; ++e) {
        const int code = quantize_one(y[e], rq.k, rq.inv);
        w[e >> 2] |= ((unsigned)code & 0xFFu) << (8 * (e & 3));
        v[e] = fmaf((float)code, rq.s, v[e]);
      }
      int8_t* cp = p.codes_out + (int64_t)r * p.n + j0;
      if (full && (reinterpret_cast<uintptr_t>(cp) & 15) == 0) {
        reinterpret_cast<uint4*>(cp)[0] = make_uint4(w[0], w[1], w[2], w[3]);
        reinterpret_cast<uint4*>(cp)[1] = make_uint4(w[4], w[5], w[6], w[7]);
      } else {
#pragma unroll
        for (int e = 0; e < 32; ++e)
          if (e < cnt) cp[e] = (int8_t)((w[e >> 2] >> (8 * (e & 3))) & 0xFFu);
      }
    }
  } else {
    if (p.codes) {
#pragma unroll
      for (int w = 0; w < 8; ++w) {
        const unsigned wx = rpay_word(q, w) ^ 0x80808080u;
#pragma unroll
        for (int b = 0; b < 4; ++b) v[4 * w + b] = fmaf(code_f32(wx, b), rq.s, v[4 * w + b]);
      }
    }
  }
  if (p.Y && cnt > 0) {
    float* zp = p.Y + (int64_t)r * p.ldy + j0;
    if (full && (reinterpret_cast<uintptr_t>(zp) & 15) == 0) {
#pragma unroll
      for (int e = 0; e < 8; ++e)
        reinterpret_cast<float4*>(zp)[e] =
            make_float4(v[4 * e], v[4 * e + 1], v[4 * e + 2], v[4 * e + 3]);
    } else {
#pragma unroll
      for (int e = 0; e < 32; ++e)
        if (e < cnt) zp[e] = v[e];
    }
  }
  if (p.seg_stats && rv) {
    // balanced trees (short dependency chains); ids past n count as -inf,
    // whose exponential is 0
    if (!full) {
#pragma unroll
      for (int e = 0; e < 32; ++e)
        if (e >= cnt) v[e] = -INFINITY;
    }
    float t[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) t[i] = fmaxf(v[2 * i], v[2 * i + 1]);
#pragma unroll
    for (int w = 8; w >= 1; w >>= 1)
#pragma unroll
      for (int i = 0; i < w; ++i) t[i] = fmaxf(t[2 * i], t[2 * i + 1]);
    const float m = t[0];
    float sum = 0.f;
    if (m > -INFINITY) {
      const float l2t = p.inv_tau * kLog2eF;   // exp(d / tau) = 2^(d log2(e) / tau)
#pragma unroll
      for (int i = 0; i < 16; ++i)
        t[i] = ex2_approx((v[2 * i] - m) * l2t) + ex2_approx((v[2 * i + 1] - m) * l2t);
#pragma unroll
      for (int w = 8; w >= 1; w >>= 1)
#pragma unroll
        for (int i = 0; i < w; ++i) t[i] = t[2 * i] + t[2 * i + 1];
      sum = t[0];
    }
    p.seg_stats[(int64_t)r * p.nseg + (j0 >> 5)] = make_float2(m, sum);
  }
}

// TM = vocabulary rows per tile: 128, or 256 as two M = 128 MMAs that share
// each B stage (half the B bytes per A byte; TMEM holds 2 x 2 x BN columns).
// PAIR: a cluster of two CTAs computes each 256-id tile as one M = 256
// tcgen05 MMA (.cta_group::2) issued by the even CTA: each CTA loads its own
// 128 ids of A and half (BN / 2) of the tile's hidden-state rows of B, and
// holds the accumulator of its 128 ids for all BN rows, so each SM takes in
// half the B bytes.  Both CTAs' copies of a stage complete on the even
// CTA's stage barrier (which expects both CTAs' bytes); the even CTA's
// commits arrive on both CTAs' barriers; both epilogues report to the even
// CTA.  Work is split over pairs.
template <int HILO, bool GATHER, int EPI, bool FP8, int TM, bool PAIR = false>
__global__ void __launch_bounds__(kThreads, 1)
tc_kernel(const __grid_constant__ WMaps wm,
          const __grid_constant__ CUtensorMap tmH, const TcParams p) {
  static_assert(TM == 128 || TM == 256, "tile height");
  static_assert(!PAIR || TM == 128, "a pair tile is two CTAs of 128 ids");
  // rows as M: the MMA's A operand is the h planes and B the weights (the
  // same shared-memory stages); pairs of CTAs with 256-row blocks only
  constexpr bool rm = EPI == EPI_ENDPOINT_RM || EPI == EPI_FUSED_RM;
  static_assert(!rm || (PAIR && !FP8), "rows as M: bf16 CTA pairs");
  constexpr int kAtomE = FP8 ? kAtomE8 : kAtomK;   // elements per 128-byte atom
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_addr = ptx::smem_u32(smem_raw);
  uint8_t* base = smem_raw + (((raw_addr + 1023) & ~1023u) - raw_addr);
  constexpr int kHalves = TM / 128;     // M = 128 halves of a tile
  constexpr int kGroups = TM / 32;      // 32-row lane groups of a tile
  constexpr int kTileStride = PAIR ? 256 : TM;      // ids between tiles
  const int BN = p.BN;
  const int BNc = PAIR ? BN / 2 : BN;   // hidden-state rows of B in this CTA
  const int NA = p.na;
  // A: per atom the TM tile rows at 128-byte stride (half h at h * 16 KB)
  const int atom_bytes = kHalves * kAtomBytes;
  const int a_bytes = NA * atom_bytes;
  const int b_bytes = HILO * NA * BNc * 128;
  const int stage_bytes = a_bytes + b_bytes;
  const int S = p.stages;
  uint64_t* full = reinterpret_cast<uint64_t*>(base + (size_t)S * stage_bytes);
  uint64_t* empty = full + S;
  uint64_t* tfull = empty + S;         // [2]
  uint64_t* tempty = tfull + 2;        // [2]
  uint64_t* drain = tempty + 2;        // [1]
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* s_abort = reinterpret_cast<volatile int*>(tmem_holder + 1);
  // the current tile's row boxes (subset path), after the barriers
  int2* s_box = reinterpret_cast<int2*>(base + (size_t)S * stage_bytes + kBarrierArea);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // pair: `half` = the CTA's rank in its cluster (0 issues the MMAs), the
  // work unit is the pair
  const int half = PAIR ? (int)ptx::cluster_ctarank() : 0;
  const int unit = PAIR ? (int)(blockIdx.x >> 1) : (int)blockIdx.x;
  const int G = PAIR ? (int)(gridDim.x >> 1) : (int)gridDim.x;
  const long long it0 = range_start(p, unit, G);
  const long long it1 = range_start(p, unit + 1, G);
  // producer, subset path: the ids of a segment's tile are loaded one
  // segment ahead, so that planning a tile never waits on memory; the first
  // tile's load goes out before the CTA's setup
  int nid[kGroups];
#pragma unroll
  for (int g = 0; g < kGroups; ++g) nid[g] = 0;
  auto load_ids = [&](int tl, int (&dst)[kGroups]) {
    const int j0 = (tl % p.NT) * kTileStride + half * 128;
    const int rows = min(TM, p.n - j0);
#pragma unroll
    for (int g = 0; g < kGroups; ++g) {
      const int r = 32 * g + lane;
      dst[g] = r < rows ? p.ids[j0 + r] : 0;
    }
  };
  // Subset path: plan tile t's row boxes (runs of consecutive kept ids,
  // each one box of its own height; lane l owns tile rows l, l + 32, ...)
  // into s_box, from the ids in nid, and start loading the ids of segment
  // tile next_tile (-1: none) into nid.  Returns the box count and the
  // stage's transaction bytes.  Warp-collective (producer warp).
  auto plan_tile = [&](int t, int next_tile, int& nbox, uint32_t& tx) {
    int2 box[2 * kGroups];                       // (first id, row | (rows - 1) << 8)
    unsigned bmask = 0;                          // which of box[] are in use
    const int j0 = t * kTileStride + half * 128;
    const int rows = min(TM, p.n - j0);
    int idr[kGroups];
#pragma unroll
    for (int g = 0; g < kGroups; ++g) idr[g] = nid[g];
    if (next_tile >= 0) load_ids(next_tile, nid);
    unsigned smask[kGroups];
    int prev_last = 0;
#pragma unroll
    for (int g = 0; g < kGroups; ++g) {
      const int r = 32 * g + lane;
      int prev = __shfl_up_sync(0xFFFFFFFFu, idr[g], 1);
      if (lane == 0) prev = prev_last;
      smask[g] = __ballot_sync(0xFFFFFFFFu, r < rows && (r == 0 || idr[g] != prev + 1));
      prev_last = __shfl_sync(0xFFFFFFFFu, idr[g], 31);
    }
    int covered = 0;
#pragma unroll
    for (int g = 0; g < kGroups; ++g) {
      const int r = 32 * g + lane;
      if ((smask[g] >> lane) & 1u) {
        int nxt = rows;
        const unsigned above = lane == 31 ? 0u : (smask[g] >> (lane + 1)) << (lane + 1);
        if (above) {
          nxt = 32 * g + __ffs(above) - 1;
        } else {
          for (int g2 = g + 1; g2 < kGroups; ++g2)
            if (smask[g2]) { nxt = 32 * g2 + __ffs(smask[g2]) - 1; break; }
        }
        // one box of exactly len rows (two, 128 + rest, past 128 rows)
        const int len = nxt - r;
        const int l0 = min(len, 128);
        box[2 * g] = make_int2(idr[g], r | ((l0 - 1) << 8));
        bmask |= 1u << (2 * g);
        if (len > 128) {
          box[2 * g + 1] = make_int2(idr[g] + 128, (r + 128) | ((len - 129) << 8));
          bmask |= 2u << (2 * g);
        }
        covered += len;
      }
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) covered += __shfl_xor_sync(0xFFFFFFFFu, covered, o);
    tx = (uint32_t)(covered * 128 * NA + b_bytes);
    // compact every lane's boxes into one shared list that the copy loop
    // below hands out to lanes (measured: far faster than issuing from
    // the planning registers under per-lane predicates)
    const int mine = __popc(bmask);
    int incl = mine;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(0xFFFFFFFFu, incl, o);
      if (lane >= o) incl += v;
    }
    nbox = __shfl_sync(0xFFFFFFFFu, incl, 31);
    int slot = incl - mine;
#pragma unroll
    for (int q = 0; q < 2 * kGroups; ++q)
      if ((bmask >> q) & 1u) s_box[slot++] = box[q];
    __syncwarp();
  };
  // the first tile's ids load while the CTA sets up
  if constexpr (GATHER) {
    if (warp == 0 && it0 < it1) load_ids((int)(it0 / p.KB), nid);
  }
  uint32_t ncols = 32;                 // two accumulators of kHalves x BN columns
  while (ncols < (uint32_t)((p.single_acc ? 1 : 2) * kHalves * BN)) ncols <<= 1;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      ptx::mbar_init(&full[s], 1);               // the TMA thread
      ptx::mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      ptx::mbar_init(&tfull[a], 1);
      ptx::mbar_init(&tempty[a], kEpiWarps * (PAIR ? 2 : 1));   // (pair: both epilogues)
    }
    ptx::mbar_init(drain, 1);
    *s_abort = 0;
    ptx::fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    // (the subset path's other heights are fetched on first use)
    ptx::prefetch_tmap(&wm.m[kBoxHeights - 1]);
    ptx::prefetch_tmap(&tmH);
  }
  // Only the warps that touch memory written or read by the kernels before
  // this one wait for them (griddep_wait): the producer before its first
  // copy, the epilogue before its first store.
  ptx::griddep_launch_dependents();
  // barriers initialised (pair: in both CTAs, before either signals the
  // other's)
  if constexpr (PAIR) ptx::cluster_sync();
  else __syncthreads();
  // the producer needs no tensor memory: it starts now, while warp 1
  // allocates the accumulators for itself and the other warps
  uint32_t tmem_base = 0;
  if (warp != 0) {
    if (warp == 1) {
      __syncwarp();
      if constexpr (PAIR) ptx::tmem_alloc_pair(tmem_holder, ncols);
      else ptx::tmem_alloc(tmem_holder, ncols);
    }
    ptx::tc_fence_before();
    ptx::named_bar_sync(1, (int)blockDim.x - 32);
    ptx::tc_fence_after();
    tmem_base = *tmem_holder;
  }

  const long long limit = p.spin_limit;

  auto give_up = [&]() {
    atomicOr(p.status, ERR_TIMEOUT);
    *s_abort = 1;
  };

  if (warp == 0) {
    // ------------------------------------------------------- TMA producer
    // lane 0 owns the ring.  On the subset path the warp plans each tile's
    // row boxes itself (lane l owns tile rows l, l+32, l+64, l+96): runs of
    // consecutive kept ids, each one box of its own height.
    Segments sg{it0, it1, p.KB};
    int stage = 0;
    uint32_t phase = 0;
    int tile, kb0, kb1;
    bool stop = false;
    long long issued = 0;
    // The h planes come from the operand-split kernel, the weights and ids
    // from the caller: the first segment's plan and the A copies of its
    // first stage go out before the wait for that kernel, the stage's B
    // copies right after it.
    bool waited = false;
    int rb_first = 0, kb_first = 0;
    // pair: the odd CTA's copies complete on the even CTA's stage barrier
    // (whose MMAs read both CTAs' stages)
    const uint32_t lead_full = PAIR ? ptx::mapa(ptx::smem_u32(full), 0) : 0u;
    auto load2 = [&](void* dst, const CUtensorMap* map, int x, int y, int st) {
      if (PAIR && half) ptx::tma_load_2d_pair(dst, map, x, y, lead_full + (uint32_t)(st * 8));
      else ptx::tma_load_2d(dst, map, x, y, &full[st]);
    };
    auto load3 = [&](void* dst, const CUtensorMap* map, int x, int y, int z, int st) {
      if (PAIR && half) ptx::tma_load_3d_pair(dst, map, x, y, z, lead_full + (uint32_t)(st * 8));
      else ptx::tma_load_3d(dst, map, x, y, z, &full[st]);
    };
    // the B copy of plane l of stage st (k-block kb, row block rb)
    auto issue_b = [&](int st, int kb, int rb, int l) {
      if (l >= 0 && l < HILO)
        load3(base + (size_t)st * stage_bytes + a_bytes + l * NA * BNc * 128, &tmH, 0,
              l * p.Rp + rb * BN + half * BNc, kb * NA, st);
    };
    auto finish_wait = [&]() {
      if (lane == 0) ptx::griddep_wait();
      __syncwarp();
      // the stages issued so far (0 or 1) are the first of the ring
      for (int q = lane; q < issued * HILO; q += 32)
        issue_b(q / HILO, kb_first + q / HILO, rb_first, q % HILO);
      waited = true;
    };
    while (!stop && sg.next(tile, kb0, kb1)) {
      const int rb = tile / p.NT, t = tile - rb * p.NT;
      int nbox = 0;
      uint32_t tx = (uint32_t)stage_bytes;
      if constexpr (GATHER) {
        Segments pk = sg;
        int tn = -1, a0, a1;
        if (!pk.next(tn, a0, a1)) tn = -1;
        plan_tile(t, tn, nbox, tx);
      }
      // pair: the odd CTA's bytes of each stage of this tile -- its B part,
      // and its A boxes, which cover each of its tile rows below n once (the
      // full-vocabulary path copies whole 128-row boxes)
      uint32_t tx_peer = 0;
      if constexpr (PAIR) {
        if constexpr (GATHER) {
          const int prow = max(0, min(128, p.n - (t * kTileStride + 128)));
          tx_peer = (uint32_t)(prow * 128 * NA + b_bytes);
        } else {
          tx_peer = (uint32_t)stage_bytes;
        }
      }
      for (int kb = kb0; kb < kb1; ++kb) {
        int ok = 1;
        if (lane == 0)
          ok = !*s_abort && ptx::mbar_wait(&empty[stage], phase ^ 1, limit);
        ok = __shfl_sync(0xFFFFFFFFu, ok, 0);
        if (!ok) {
          if (lane == 0 && !*s_abort) give_up();
          stop = true;
          break;
        }
        // (pair: the even CTA expects both CTAs' bytes; the odd CTA's copies
        // complete on that barrier without an arrival of their own)
        if (lane == 0 && !(PAIR && half)) ptx::mbar_expect_tx(&full[stage], tx + tx_peer);
        __syncwarp();
        // every copy of the stage goes to its own lane, so the copies are
        // issued side by side rather than one after another: A as NA x (row
        // boxes), or over the full vocabulary (when its width allows) one 3-D
        // copy of all NA atoms; B as one 3-D copy of all NA atoms per plane
        uint8_t* A = base + (size_t)stage * stage_bytes;
        const int nA = GATHER ? NA * nbox : (p.a3d ? 1 : NA * kHalves);
        if (!waited && issued == 0) { rb_first = rb; kb_first = kb; }
        for (int op = lane; op < nA + (waited ? HILO : 0); op += 32) {
          if (op < nA) {
            if constexpr (GATHER) {
              const int a = op / nbox;
              const int2 bx = s_box[op - a * nbox];
              load2(A + a * atom_bytes + (bx.y & 0xFF) * 128, &wm.m[bx.y >> 8],
                    (kb * NA + a) * kAtomE, bx.x, stage);
            } else if (p.a3d) {
              load3(A, &wm.a3, 0, t * kTileStride + half * 128, kb * NA, stage);
            } else {
              const int a = op / kHalves, hf = op - a * kHalves;
              load2(A + a * atom_bytes + hf * kAtomBytes, &wm.m[kBoxHeights - 1],
                    (kb * NA + a) * kAtomE, t * kTileStride + half * 128 + hf * 128, stage);
            }
          } else {
            issue_b(stage, kb, rb, op - nA);
          }
        }
        ++issued;
        if (++stage == S) { stage = 0; phase ^= 1; }
        if (!waited) finish_wait();
      }
    }
    // (a CTA without work, or one that stopped before its first segment's
    // stages were all issued, still sends their B copies, so that every
    // issued stage completes)
    if (!waited) finish_wait();
    if (stop && lane == 0) {
      // let the copies already issued land before the CTA winds down (the
      // odd CTA of a pair cannot wait on the even CTA's barriers: it waits
      // about 100 us, far longer than a copy takes)
      if (PAIR && half) {
        const long long t0 = clock64();
        while (clock64() - t0 < (200000ll)) __nanosleep(1000);
      } else {
        for (long long k = issued > S ? issued - S : 0; k < issued; ++k)
          ptx::mbar_wait(&full[k % S], (uint32_t)((k / S) & 1), kDrainLimit);
      }
    }
  } else if (warp == 1 && PAIR && half == 1) {
    // pair, odd CTA: the even CTA issues the MMAs for both
  } else if (warp == 1) {
    // ---------------------------------------------------------- MMA issuer
    if (lane == 0) {
      Segments sg{it0, it1, p.KB};
      int stage = 0;
      uint32_t phase = 0;
      uint32_t tph[2] = {0, 0};
      int si = 0, tile, kb0, kb1;
      constexpr int kMmaM = PAIR ? 2 * kTileM : kTileM;
      const uint32_t idesc =
          FP8 ? ptx::idesc_e4m3_f32(kMmaM, BN)
              : ptx::idesc_bf16_f32(kMmaM, rm ? kTileStride : BN);   // (rows as M: N = ids)
      auto wait_x = [&](uint64_t* bar, uint32_t parity) {
        return ptx::mbar_wait(bar, parity, limit);
      };
      // accumulator `acc`, tile half hf: TMEM columns (acc * kHalves + hf) * BN
      bool stop = false;
      while (!stop && sg.next(tile, kb0, kb1)) {
        const int acc = p.single_acc ? 0 : (si & 1);
        if (*s_abort || !wait_x(&tempty[acc], tph[acc] ^ 1)) {
          if (!*s_abort) give_up();
          break;
        }
        tph[acc] ^= 1;
        ptx::tc_fence_after();
        const uint32_t d = tmem_base + (uint32_t)(acc * kHalves * BN);
        for (int kb = kb0; kb < kb1; ++kb) {
          if (*s_abort || !wait_x(&full[stage], phase)) {
            if (!*s_abort) give_up();
            stop = true;
            break;
          }
          ptx::tc_fence_after();
          const uint32_t a0 = ptx::smem_u32(base + (size_t)stage * stage_bytes);
          const uint32_t b0 = a0 + a_bytes;
          for (int at = 0; at < NA; ++at) {
#pragma unroll
            for (int h = 0; h < HILO; ++h) {
#pragma unroll
              for (int kk = 0; kk < kAtomK / 16; ++kk) {
#pragma unroll
                for (int hf = 0; hf < kHalves; ++hf)
                {
                  // 32 bytes of K per MMA: 16 bf16 or 32 e4m3 elements
                  const uint64_t wd =
                      ptx::sdesc_k128(a0 + at * atom_bytes + hf * kAtomBytes + kk * 32);
                  const uint64_t hd = ptx::sdesc_k128(b0 + (h * NA + at) * BNc * 128 + kk * 32);
                  const uint64_t ad = rm ? hd : wd, bd = rm ? wd : hd;
                  const uint32_t accum = (kb != kb0 || at != 0 || h != 0 || kk != 0) ? 1u : 0u;
                  if constexpr (PAIR && FP8)
                    ptx::umma_f8_pair(d, ad, bd, idesc, accum);
                  else if constexpr (PAIR)
                    ptx::umma_f16_pair(d, ad, bd, idesc, accum);
                  else if constexpr (FP8)
                    ptx::umma_f8(d + (uint32_t)(hf * BN), ad, bd, idesc, accum);
                  else
                    ptx::umma_f16(d + (uint32_t)(hf * BN), ad, bd, idesc, accum);
                }
              }
            }
          }
          if constexpr (PAIR) ptx::umma_commit_pair(&empty[stage]);
          else ptx::umma_commit(&empty[stage]);
          if (++stage == S) { stage = 0; phase ^= 1; }
        }
        if (stop) break;
        if constexpr (PAIR) ptx::umma_commit_pair(&tfull[acc]);
        else ptx::umma_commit(&tfull[acc]);
        ++si;
      }
      // all issued MMAs complete before TMEM is released
      if constexpr (PAIR) {
        ptx::umma_commit_pair(drain);
        ptx::mbar_wait(drain, 0, kDrainLimit);
      } else {
        ptx::umma_commit(drain);
        ptx::mbar_wait(drain, 0, kDrainLimit);
      }
    }
  } else if (warp < 2 + kEpiWarps) {
    // ------------------------------------------------------------ epilogue
    // A warp may only read the TMEM lanes of its quadrant (warp index mod
    // 4); the two warps of a quadrant take alternate 16-column chunks.
    const int quad = warp & 3;
    const int grp = (warp - 2) >> 2;
    const int nch = BN / 16;                     // 16-column chunks per tile half
    const int nhc = kHalves * nch;               // (half, chunk) pairs, hc = hf * nch + ch
    ptx::griddep_wait();
    Segments sg{it0, it1, p.KB};
    uint32_t fph[2] = {0, 0};
    int si = 0, tile, kb0, kb1;
    while (sg.next(tile, kb0, kb1)) {
      const int acc = p.single_acc ? 0 : (si & 1);
      const int rb = tile / p.NT, t = tile - rb * p.NT;
      const bool whole = kb0 == 0 && kb1 == p.KB;
      const int segb = (t * kTileStride + half * 128) / 32;   // first 32-id segment
      // this lane's vocabulary row in each half: i = hf * 128 + quad * 32 + lane
      int jh[kHalves], idh[kHalves];
      bool vjh[kHalves];
#pragma unroll
      for (int hf = 0; hf < kHalves; ++hf) {
        jh[hf] = t * kTileStride + half * 128 + hf * 128 + quad * 32 + lane;
        vjh[hf] = jh[hf] < p.n;
        idh[hf] = vjh[hf] ? (GATHER ? p.ids[jh[hf]] : jh[hf]) : 0;
      }
      // (selects, not a runtime-indexed array, for the loops' half index)
      auto J = [&](int hf) { return (kHalves > 1 && hf) ? jh[kHalves - 1] : jh[0]; };
      auto VJ = [&](int hf) { return (kHalves > 1 && hf) ? vjh[kHalves - 1] : vjh[0]; };
      auto ID = [&](int hf) { return (kHalves > 1 && hf) ? idh[kHalves - 1] : idh[0]; };
      // the endpoint through this warp's transpose tile (no per-lane
      // payload registers then)
      constexpr bool epi_t = EPI == EPI_ENDPOINT_T;
      constexpr bool lane_pay = EPI == EPI_ENDPOINT || EPI == EPI_FUSED;
      float* tb = reinterpret_cast<float*>(base + (size_t)S * stage_bytes + kBarrierArea +
                                           kMaxBoxes * sizeof(int2)) +
                  (warp - 2) * 8 * kTRow;
      Payload pay;
      // rows as M: this lane's row, its constants, and the codes of its
      // four 32-id segments of the tile (segments grp, grp + 2, ...), all
      // loaded while the tile's MMAs run
      constexpr int kRmSeg = 8 / kEpiGroups;
      const int r_rm = rb * 256 + half * 128 + quad * 32 + lane;
      RowQuant rq_rm{0.f, 1.f, 0.f};
      RPay rp[kRmSeg];
      if constexpr (rm) {
        if (r_rm < p.R) {
          if constexpr (EPI == EPI_FUSED_RM) {
            rq_rm = row_quant(__ldcg(p.rowmax_in + r_rm));
            if (t == 0 && grp == 0) p.scale_out[r_rm] = rq_rm.s;
            // (the clipped partials are read when finishing: warm L2 now)
#pragma unroll
            for (int a = 0; a < kRmSeg; ++a) {
              const int j0 = t * 256 + (grp + a * kEpiGroups) * 32;
              if (j0 < p.n)
                asm volatile("prefetch.global.L2 [%0];" ::"l"(p.yc + (int64_t)r_rm * p.n + j0));
            }
          } else if (p.codes) {
            rq_rm.s = __ldg(p.row_scale + r_rm);
          }
        }
        if constexpr (EPI == EPI_ENDPOINT_RM) {
#pragma unroll
          for (int a = 0; a < kRmSeg; ++a)
            load_rpay(p, r_rm, t * 256 + (grp + a * kEpiGroups) * 32, rp[a]);
        }
      }
      if constexpr (EPI != EPI_CLOUD && !rm) {
        // the payload does not depend on the accumulator: start on it
        // while the tile's MMAs run
#pragma unroll
        for (int hf = 0; hf < kHalves; ++hf)
          prefetch_payload<EPI>(p, rb * BN + grp * (BN / 2), BN / 2,
                                t * kTileStride + half * 128 + hf * 128 + quad * 32, lane);
        if constexpr (lane_pay)
          if (whole && grp < nhc)
            load_payload<EPI>(p, rb * BN + (grp % nch) * 16, J(grp / nch), lane, pay);
      }
      // the transposed payload of whole tiles runs kTAhead chunks ahead of
      // the one being finished (tq[a]: chunk hc + (a + 1) kEpiGroups): a
      // chunk's work is shorter than a load's latency under the kernel's
      // own traffic
      constexpr int kTAhead = 3;
      TPay tpay, tq[kTAhead];
      if (epi_t && whole) {
#pragma unroll
        for (int a = 0; a <= kTAhead; ++a) {
          const int hn = grp + a * kEpiGroups;
          if (hn < nhc)
            load_tpay(p, rb * BN + (hn % nch) * 16, J(hn / nch) - lane, lane,
                      a == 0 ? tpay : tq[a - 1]);
        }
      }
      // (split tiles load the transposed payload right before finishing)
      auto finish = [&](const float (&vv)[16], int hf, int ch) {
        if constexpr (rm) {
          // (rows as M takes whole tiles only)
        } else if constexpr (epi_t) {
          if (!whole) load_tpay(p, rb * BN + ch * 16, J(hf) - lane, lane, tpay);
          finish_chunk_t(p, vv, rb * BN + ch * 16, J(hf) - lane, lane, tb, tpay);
        } else {
          finish_chunk<EPI>(p, vv, rb * BN + ch * 16, J(hf), VJ(hf), ID(hf), lane,
                            segb + hf * 4 + quad, pay);
        }
      };
      // Split tile: contributors c0 .. c0 + C - 1 (CTA order).  All but the
      // last end their ranges inside the tile, so they reach it at the end
      // of their work; the last one reaches it first thing (its range starts
      // inside the tile).  Contributor c0 + C - 2 is the tile's finisher: it
      // waits (briefly, bounded) until every other contributor's warp of
      // this quadrant and chunk group has stored its partial and counted
      // in, then finishes the tile from its own accumulator and their
      // partials.  The others store and count in; if the finisher gave up
      // waiting it counts in like them, and whoever counts in last finishes
      // the tile from the stored partials.
      constexpr int kMaxC = 8;
      int c0 = 0, C = 1, cnt = 0;
      bool fin = false, known_last = false, pre_ok = false;
      float pre[16];                   // two contributors: the other's first chunk
      if (!whole) {
        cnt = ((tile * 4 + quad) * kEpiGroups + grp) * (PAIR ? 2 : 1) + half;
        c0 = (int)cta_of((long long)tile * p.KB, p.T, G);
        C = (int)cta_of((long long)tile * p.KB + p.KB - 1, p.T, G) - c0 + 1;
        fin = p.finish_wait > 0 && C >= 2 && C <= kMaxC && unit == c0 + C - 2;
      }
      // the contributors' partial slots: every contributor after the first
      // starts its range inside this tile, so the tile is its first segment
      // (slot 2c); the first one holds it as its first segment only if its
      // range starts exactly at the tile (slot 2c0), else as its last
      // (slot 2c0 + 1)
      const bool c0_first = !whole && range_start(p, c0, G) == (long long)tile * p.KB;
      // (pair: each CTA of a unit keeps its own half of the partial)
      auto pslot = [&](int u) { return PAIR ? 2 * u + half : u; };
      auto slot_of = [&](int c) {
        return pslot(c == 0 ? 2 * c0 + (c0_first ? 0 : 1) : 2 * (c0 + c));
      };
      if (fin) {
        // the early contributor (the tile's last) has usually arrived
        // already: then fetch its partial while the MMAs finish
        int arrived = 0;
        if (lane == 0) arrived = ptx::ld_acquire_gpu(&p.counters[cnt]);
        known_last = __shfl_sync(0xFFFFFFFFu, arrived, 0) == C - 1;
        __syncwarp();
        // (cloud only: the endpoint epilogue's payload registers leave no
        // room, and its short hidden dimension mostly gives whole tiles)
        if (EPI == EPI_CLOUD && known_last && C == 2 && grp < nhc) {
          const int hf = grp / nch, ch = grp - hf * nch;
          const float* pc = p.P + (size_t)slot_of(1) * BN * TM + (size_t)ch * 16 * TM +
                            hf * 128 + quad * 32 + lane;
#pragma unroll
          for (int q = 0; q < 16; ++q) pre[q] = __ldcg(pc + (size_t)q * TM);
          pre_ok = true;
        }
      }
      int ok = 1;
      if (lane == 0)
        ok = !*s_abort && ptx::mbar_wait(&tfull[acc], fph[acc], limit);
      ok = __shfl_sync(0xFFFFFFFFu, ok, 0);
      if (!ok) {
        if (lane == 0 && !*s_abort) give_up();
        break;
      }
      fph[acc] ^= 1;
      if (fin && !known_last) {
        // the other contributors that end with this tile finish at about
        // the same time: poll for them, bounded (giving up only costs the
        // round trip through the partial buffer)
        int arrived = 0;
        if (lane == 0) {
          const long long t0 = clock64();
          const long long bound = limit < p.finish_wait ? limit : p.finish_wait;
          while ((arrived = ptx::ld_acquire_gpu(&p.counters[cnt])) != C - 1 &&
                 clock64() - t0 < bound)
            __nanosleep(64);
        }
        known_last = __shfl_sync(0xFFFFFFFFu, arrived, 0) == C - 1;
        __syncwarp();
      }
      ptx::tc_fence_after();
      const uint32_t taddr = tmem_base + ((uint32_t)(quad * 32) << 16) +
                             (uint32_t)(acc * kHalves * BN);
      // a CTA's split tiles can only be its first and its last segment:
      // slot 2c holds the first, 2c+1 the last ([BN][TM] each)
      float* Pt = p.P + (size_t)pslot(2 * unit + (si == 0 ? 0 : 1)) * BN * TM;
      if constexpr (rm) {
        // this lane's row: 32 consecutive columns (ids) per load
        // (two segments per accumulator wait, finished side by side)
#pragma unroll
        for (int a = 0; a < kRmSeg; a += 2) {
          const int s0 = grp + a * kEpiGroups, s1 = s0 + kEpiGroups;
          float v0[32], v1[32];
          ptx::tmem_ld32x2(taddr + (uint32_t)(s0 * 32), taddr + (uint32_t)(s1 * 32), v0, v1);
          finish_rm<EPI>(p, v0, r_rm, t * 256 + s0 * 32, rp[a], rq_rm);
          finish_rm<EPI>(p, v1, r_rm, t * 256 + s1 * 32, rp[a + 1], rq_rm);
        }
      }
      for (int hc = grp; hc < (rm ? 0 : nhc); hc += kEpiGroups) {
        const int hf = hc / nch, ch = hc - hf * nch;
        const int i = hf * 128 + quad * 32 + lane;
        float v[16];
        ptx::tmem_ld16(taddr + hf * BN + ch * 16, v);
        if (whole) {
          Payload nxt;
          const int hn = hc + kEpiGroups;
          TPay tnxt;
          if constexpr (lane_pay)
            if (hn < nhc) load_payload<EPI>(p, rb * BN + (hn % nch) * 16, J(hn / nch), lane, nxt);
          const int ht = hc + (kTAhead + 1) * kEpiGroups;
          if (epi_t && ht < nhc)
            load_tpay(p, rb * BN + (ht % nch) * 16, J(ht / nch) - lane, lane, tnxt);
          finish(v, hf, ch);
          if constexpr (lane_pay) pay = nxt;
          if constexpr (epi_t) {
            tpay = tq[0];
#pragma unroll
            for (int a = 0; a + 1 < kTAhead; ++a) tq[a] = tq[a + 1];
            tq[kTAhead - 1] = tnxt;
          }
        } else if (known_last) {
          // the partials in CTA order (the same order, and so the same
          // result, as the fix-up below), this CTA's own from registers
          if constexpr (lane_pay) load_payload<EPI>(p, rb * BN + ch * 16, J(hf), lane, pay);
          const int me = unit - c0;
          const size_t o = (size_t)ch * 16 * TM + i;
          float s[16];
          if (pre_ok && hc == grp) {       // two contributors, the other's part prefetched
#pragma unroll
            for (int q = 0; q < 16; ++q) s[q] = v[q] + pre[q];   // (me == 0)
          } else {
#pragma unroll
            for (int c = 0; c < kMaxC; ++c) {
              if (c < C) {
                const float* pc = p.P + (size_t)slot_of(c) * BN * TM + o;
#pragma unroll
                for (int q = 0; q < 16; ++q) {
                  const float x = c == me ? v[q] : __ldcg(pc + (size_t)q * TM);
                  s[q] = c == 0 ? x : s[q] + x;
                }
              }
            }
          }
          finish(s, hf, ch);
        } else {
#pragma unroll
          for (int q = 0; q < 16; ++q) Pt[(size_t)(ch * 16 + q) * TM + i] = v[q];
        }
      }
      ptx::tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (PAIR && half) ptx::mbar_arrive_remote(ptx::mapa(ptx::smem_u32(&tempty[acc]), 0));
        else ptx::mbar_arrive(&tempty[acc]);
      }
      if (known_last) {
        if (lane == 0) p.counters[cnt] = 0;
      } else if (!whole) {
        // split tile: this warp's rows x its chunks are finished by the last
        // warp (over all contributing CTAs) of the same quadrant and chunk
        // group
        __threadfence();
        int old = 0;
        if (lane == 0) old = atomicAdd(&p.counters[cnt], 1);
        old = __shfl_sync(0xFFFFFFFFu, old, 0);
        if (old == C - 1) {
          __threadfence();
          // the contributors' partials in CTA order (a fixed summation order)
          const float* ps[kMaxC];
#pragma unroll
          for (int c = 0; c < kMaxC; ++c)
            ps[c] = p.P + (size_t)slot_of(c < C ? c : 0) * BN * TM + quad * 32 + lane;
          for (int hc = grp; hc < nhc; hc += kEpiGroups) {
            const int hf = hc / nch, ch = hc - hf * nch;
            if constexpr (lane_pay) load_payload<EPI>(p, rb * BN + ch * 16, J(hf), lane, pay);
            const size_t o = (size_t)ch * 16 * TM + hf * 128;
            float v[16];
#pragma unroll
            for (int q = 0; q < 16; ++q) v[q] = __ldcg(ps[0] + o + (size_t)q * TM);
#pragma unroll
            for (int c = 1; c < kMaxC; ++c) {
              if (c < C) {
#pragma unroll
                for (int q = 0; q < 16; ++q) v[q] += __ldcg(ps[c] + o + (size_t)q * TM);
              }
            }
            for (int c = kMaxC; c < C; ++c) {    // rare: very many contributors
              const float* pc = p.P + (size_t)pslot(2 * (c0 + c)) * BN * TM + quad * 32 + lane;
#pragma unroll
              for (int q = 0; q < 16; ++q) v[q] += __ldcg(pc + o + (size_t)q * TM);
            }
            finish(v, hf, ch);
          }
          if (lane == 0) p.counters[cnt] = 0;
        }
      }
      ++si;
    }
  }

  ptx::tc_fence_before();
  // pair: neither CTA leaves (or frees its tensor memory) before the other
  // is done with its arrivals and the even CTA's MMAs have completed
  if constexpr (PAIR) ptx::cluster_sync();
  else __syncthreads();
  ptx::tc_fence_after();
  if (warp == 1) {
    __syncwarp();
    if constexpr (PAIR) ptx::tmem_dealloc_pair(tmem_base, ncols);
    else ptx::tmem_dealloc(tmem_base, ncols);
  }
}

// ---------------------------------------------------------------------------
// operand preparation: fp32 h -> bf16 hi (and lo) planes, zero padded
// ---------------------------------------------------------------------------
// ... and clear the split-tile counters and (cloud) the row maxima.
// One thread converts 8 consecutive columns of one row (Kp is a multiple of
// 64, so a group never crosses a row) and stores 16 bytes per plane.  Small
// 128-thread blocks with at most 32 registers fit beside a tensor-core CTA
// on the same SM, so that kernel starts (and issues its first weight copies)
// while this one runs.
__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<const uint32_t*>(&v);
}

// hi = bf16(x), lo = bf16(x - hi) of 8 values
__device__ __forceinline__ void split_group(const float (&x)[8], int hilo, uint4* hi, uint4* lo) {
  float r[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) r[i] = __bfloat162float(__float2bfloat16_rn(x[i]));
  *hi = make_uint4(pack_bf16x2(r[0], r[1]), pack_bf16x2(r[2], r[3]), pack_bf16x2(r[4], r[5]),
                   pack_bf16x2(r[6], r[7]));
  if (hilo == 2)
    *lo = make_uint4(pack_bf16x2(x[0] - r[0], x[1] - r[1]), pack_bf16x2(x[2] - r[2], x[3] - r[3]),
                     pack_bf16x2(x[4] - r[4], x[5] - r[5]), pack_bf16x2(x[6] - r[6], x[7] - r[7]));
}

constexpr int kSplitThreads = 128;
__global__ void __launch_bounds__(kSplitThreads, 16)
split_h_kernel(const float* __restrict__ h, int64_t ld_h, int R, int K, int Rp, int Kp,
               int hilo, __nv_bfloat16* __restrict__ Hs, int* __restrict__ counters,
               int ncounters, unsigned* __restrict__ rowmax) {
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  const int tid = blockIdx.x * blockDim.x + threadIdx.x;
  const int nth = gridDim.x * blockDim.x;
  if (rowmax)
    for (int r = tid; r < R; r += nth) rowmax[r] = 0u;
  for (int t = tid; t < ncounters; t += nth) counters[t] = 0;
  const int gpr = Kp / 8;                          // groups per row
  const int64_t groups = (int64_t)Rp * gpr;
  const int64_t total = (int64_t)Rp * Kp;
  const bool vec = (((uintptr_t)h | (uintptr_t)(ld_h * 4)) & 15) == 0;
  for (int64_t g = tid; g < groups; g += nth) {
    const int r = (int)(g / gpr), c0 = (int)(g - (int64_t)r * gpr) * 8;
    float x[8];
    const float* src = h + (int64_t)r * ld_h + c0;
    if (r < R && vec && c0 + 8 <= K) {
      const float4 a = __ldg(reinterpret_cast<const float4*>(src));
      const float4 b = __ldg(reinterpret_cast<const float4*>(src) + 1);
      x[0] = a.x; x[1] = a.y; x[2] = a.z; x[3] = a.w;
      x[4] = b.x; x[5] = b.y; x[6] = b.z; x[7] = b.w;
    } else {
#pragma unroll
      for (int i = 0; i < 8; ++i) x[i] = (r < R && c0 + i < K) ? __ldg(src + i) : 0.f;
    }
    uint4 hi, lo;
    split_group(x, hilo, &hi, &lo);
    uint4* dst = reinterpret_cast<uint4*>(Hs + g * 8);
    dst[0] = hi;
    if (hilo == 2) *reinterpret_cast<uint4*>(Hs + total + g * 8) = lo;
  }
}


// fp8 weights: h -> e4m3 planes under a per-row power-of-two scale.  One
// block per padded row: the row's max |h| fixes the scale 2^e with
// max |h| / 2^e in [128, 256) (e4m3 holds up to 448).  Plane q is the e4m3
// rounding (to nearest) of what planes 0..q-1 left of h / 2^e, so h equals
// 2^e times the sum of the planes up to the last one's rounding: 4 planes
// leave 2^-13 |h| (or 2^-10 2^e where the planes reach e4m3's subnormal
// range); 2 planes reproduce bf16-rounded h, whose 8 significant bits are
// two 4-bit halves.  Also clears the split-tile counters and row maxima.
constexpr int kSplit8Threads = 256;
__global__ void __launch_bounds__(kSplit8Threads)
split_h_e4m3_kernel(const float* __restrict__ h, int64_t ld_h, int R, int K, int Rp, int Kp,
                    int planes, uint8_t* __restrict__ Hs, float* __restrict__ h_scale,
                    int* __restrict__ counters, int ncounters, unsigned* __restrict__ rowmax,
                    int act_bf16) {
  __shared__ float s_max[kSplit8Threads / 32];
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  const int tid = blockIdx.x * blockDim.x + threadIdx.x;
  const int nth = gridDim.x * blockDim.x;
  if (rowmax)
    for (int i = tid; i < R; i += nth) rowmax[i] = 0u;
  for (int i = tid; i < ncounters; i += nth) counters[i] = 0;
  const int r = blockIdx.x;
  const float* hr = h + (int64_t)r * ld_h;
  auto value = [&](int c) {
    float x = (r < R && c < K) ? __ldg(hr + c) : 0.f;
    if (act_bf16) x = __bfloat162float(__float2bfloat16_rn(x));
    return x;
  };
  // each thread takes 4 consecutive columns at a time: one 16-byte load
  // where the row is so aligned, one 4-byte store per plane
  const bool v16 = (reinterpret_cast<uintptr_t>(hr) & 15) == 0;
  auto value4 = [&](int c, float (&x)[4]) {
    if (v16 && r < R && c + 4 <= K) {
      const float4 t = __ldg(reinterpret_cast<const float4*>(hr + c));
      x[0] = t.x; x[1] = t.y; x[2] = t.z; x[3] = t.w;
      if (act_bf16) {
#pragma unroll
        for (int e = 0; e < 4; ++e) x[e] = __bfloat162float(__float2bfloat16_rn(x[e]));
      }
    } else {
#pragma unroll
      for (int e = 0; e < 4; ++e) x[e] = value(c + e);
    }
  };
  float m = 0.f;
  for (int c = 4 * threadIdx.x; c < K; c += 4 * blockDim.x) {
    float x[4];
    value4(c, x);
    m = fmaxf(m, fmaxf(fmaxf(fabsf(x[0]), fabsf(x[1])), fmaxf(fabsf(x[2]), fabsf(x[3]))));
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
  if ((threadIdx.x & 31) == 0) s_max[threadIdx.x >> 5] = m;
  __syncthreads();
  m = 0.f;
#pragma unroll
  for (int w = 0; w < kSplit8Threads / 32; ++w) m = fmaxf(m, s_max[w]);
  // 2^e with m / 2^e in [128, 256): the exponent field of m less 7
  const int eb = (int)((__float_as_uint(m) >> 23) & 0xFF);
  const float scale = eb > 7 ? __uint_as_float((uint32_t)(eb - 7) << 23) : 1.0f;
  const float inv = eb > 7 && eb - 7 < 254 ? __uint_as_float((uint32_t)(254 - (eb - 7)) << 23)
                                           : 1.0f;
  if (threadIdx.x == 0) h_scale[r] = scale;
  const int64_t plane = (int64_t)Rp * Kp;
  // (Kp is a multiple of 128, so every 4-column group is 4-byte aligned)
  for (int c = 4 * threadIdx.x; c < Kp; c += 4 * blockDim.x) {
    float x[4];
    value4(c, x);
#pragma unroll
    for (int e = 0; e < 4; ++e) x[e] *= inv;              // exact: a power of two
    for (int q = 0; q < planes; ++q) {
      uint32_t word = 0;
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const __nv_fp8_e4m3 f(x[e]);                      // round to nearest, saturating
        word |= (uint32_t)f.__x << (8 * e);
        x[e] -= static_cast<float>(f);
      }
      *reinterpret_cast<uint32_t*>(Hs + q * plane + (int64_t)r * Kp + c) = word;
    }
  }
}


// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
using EncodeFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                              const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                              const cuuint32_t*, CUtensorMapInterleave,
                              CUtensorMapSwizzle, CUtensorMapL2promotion,
                              CUtensorMapFloatOOBfill);

EncodeFn encode_fn() {
  static EncodeFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                         cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeFn>(p);
  });
  return fn;
}

bool make_map(CUtensorMap* m, CUtensorMapDataType dt, const void* ptr,
              uint64_t inner, uint64_t outer, uint64_t row_bytes, uint32_t box_x,
              uint32_t box_y) {
  EncodeFn fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[2] = {inner, outer};
  const cuuint64_t strides[1] = {row_bytes};
  const cuuint32_t box[2] = {box_x, box_y};
  const cuuint32_t es[2] = {1, 1};
  return fn(m, dt, 2, const_cast<void*>(ptr), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 3-D view (element, row, atom) of a row-major [rows, cols] matrix, an atom
// being the `atom` elements of 128 bytes (64 bf16, 128 e4m3): strides
// row_bytes and 128 bytes; a box of (atom, box_rows, box_atoms) lands as
// box_atoms consecutive 128-byte-swizzled atom tiles of box_rows rows.  cols
// must be a multiple of atom (the view cannot mark the end of a row).
bool make_map3(CUtensorMap* m, CUtensorMapDataType dt, const void* ptr, uint64_t cols,
               uint64_t rows, uint64_t row_bytes, uint32_t box_rows, uint32_t box_atoms,
               int atom) {
  EncodeFn fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[3] = {(cuuint64_t)atom, rows, cols / atom};
  const cuuint64_t strides[2] = {row_bytes, 128};
  const cuuint32_t box[3] = {(cuuint32_t)atom, box_rows, box_atoms};
  const cuuint32_t es[3] = {1, 1, 1};
  return fn(m, dt, 3, const_cast<void*>(ptr), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

size_t align256(size_t x) { return (x + 255) / 256 * 256; }

// make_map3 with a small cache: the h-plane and full-vocabulary maps of a
// call usually repeat the previous calls' (the scratch arena and the weights
// stay put), and encoding costs more host time than the launch itself.
struct Map3Key {
  int dt;
  const void* ptr;
  uint64_t cols, rows, row_bytes;
  uint32_t box_rows, box_atoms;
  int atom;
  bool operator==(const Map3Key& o) const {
    return dt == o.dt && ptr == o.ptr && cols == o.cols && rows == o.rows &&
           row_bytes == o.row_bytes && box_rows == o.box_rows && box_atoms == o.box_atoms &&
           atom == o.atom;
  }
};
struct Map3Entry {
  Map3Key key{};
  bool valid = false;
  unsigned long long used = 0;
  CUtensorMap map;
};
std::mutex g_map3_mu;
Map3Entry g_map3[16];
unsigned long long g_map3_tick = 0;

bool cached_map3(CUtensorMap* m, CUtensorMapDataType dt, const void* ptr, uint64_t cols,
                 uint64_t rows, uint64_t row_bytes, uint32_t box_rows, uint32_t box_atoms,
                 int atom) {
  const Map3Key key{(int)dt, ptr, cols, rows, row_bytes, box_rows, box_atoms, atom};
  std::lock_guard<std::mutex> lock(g_map3_mu);
  Map3Entry* lru = &g_map3[0];
  for (Map3Entry& e : g_map3) {
    if (e.valid && e.key == key) {
      e.used = ++g_map3_tick;
      *m = e.map;
      return true;
    }
    if (!e.valid || e.used < lru->used) lru = &e;
  }
  if (!make_map3(&lru->map, dt, ptr, cols, rows, row_bytes, box_rows, box_atoms, atom)) {
    lru->valid = false;
    return false;
  }
  lru->key = key;
  lru->valid = true;
  lru->used = ++g_map3_tick;
  *m = lru->map;
  return true;
}

// W tensor maps, encoded once per weight tensor: map i copies boxes of one
// 128-byte atom (64 bf16 or 128 e4m3 columns) x (i + 1) rows of W [V rows,
// K columns], row stride ld_w (the full-vocabulary path uses only the
// 128-row map).  A few recently used
// sets are kept, since encoding 128 maps costs far more than a launch.
struct MapSet {
  const void* W = nullptr;
  int64_t V = 0, K = 0, ld = 0;
  int w_dtype = 0;
  bool gather = false;
  unsigned long long used = 0;
  WMaps maps;
};
std::mutex g_map_mu;
MapSet g_map_sets[8];
unsigned long long g_map_tick = 0;

bool w_maps(const GatherGemm& g, bool gather, WMaps& out) {
  std::lock_guard<std::mutex> lock(g_map_mu);
  MapSet* hit = nullptr;
  MapSet* lru = &g_map_sets[0];
  for (MapSet& m : g_map_sets) {
    if (m.W == g.W && m.V == g.V && m.K == g.K && m.ld == g.ld_w && m.gather == gather &&
        m.w_dtype == g.w_dtype)
      hit = &m;
    if (m.used < lru->used) lru = &m;
  }
  if (!hit) {
    hit = lru;
    hit->W = nullptr;
    for (int i = 0; i < kBoxHeights; ++i) {
      if (!gather && i != kBoxHeights - 1) {
        hit->maps.m[i] = CUtensorMap{};
        continue;
      }
      const bool e4m3 = g.w_dtype == W_FP8;
      if (!make_map(&hit->maps.m[i],
                    e4m3 ? CU_TENSOR_MAP_DATA_TYPE_UINT8 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, g.W,
                    (uint64_t)g.K, (uint64_t)g.V, (uint64_t)g.ld_w * (e4m3 ? 1 : 2),
                    e4m3 ? kAtomE8 : kAtomK, (uint32_t)(i + 1)))
        return false;
    }
    hit->W = g.W; hit->V = g.V; hit->K = g.K; hit->ld = g.ld_w; hit->gather = gather;
    hit->w_dtype = g.w_dtype;
  }
  hit->used = ++g_map_tick;
  out = hit->maps;
  return true;
}

}  // namespace

namespace {
// The plan of a CTA-pair launch: 256-id tiles, each CTA of a pair with 128
// ids of A and half of B's rows, row blocks of up to 256 rows (a multiple of
// 32, so that each CTA's half is whole 16-row groups), work split over the
// pairs (a multiple of the row-block count, as below).
TcPlan tc_plan_pair(TcPlan pl, int rows, int n, int K, int sm_count, int max_pairs,
                    int schedule, int max_stages, int block_k, int max_bn_opt, int endpoint,
                    int rm_mode) {
  // (e4m3 weights: four or two h planes; 128-row blocks keep four stages)
  int cap = pl.fp8 ? 128 : 256;
  if (max_bn_opt >= 32 && max_bn_opt < cap) cap = max_bn_opt / 32 * 32;
  pl.RB = (rows + cap - 1) / cap;
  pl.BN = ((rows + pl.RB - 1) / pl.RB + 31) / 32 * 32;
  // the endpoint with rows as M: 256-row blocks (M = 256 over the pair),
  // whole tiles; automatic where the row blocks lose at most 1/8 to padding
  // (measured on 1024 rows x 256000 ids x 512: 0.43 ms with z not stored,
  // against 0.56 ms and a 0.18 ms statistics pass with ids as M)
  const int rb256 = (rows + 255) / 256;
  pl.rm = endpoint && !pl.fp8 && schedule != 2 && rm_mode != 2 &&
          (rm_mode == 1 || (cap == 256 && 8 * (rb256 * 256 - rows) <= rb256 * 256));
  if (pl.rm) {
    pl.RB = rb256;
    pl.BN = 256;
    schedule = 1;
  }
  pl.tm = 128;
  pl.single_acc = 0;
  pl.Rp = pl.RB * pl.BN;
  // the endpoint's epilogue as on single CTAs (each CTA of a pair finishes
  // its own 128 ids for all BN rows); rows as M: the statistics of a
  // lane's 32-id segment are its own, always made in the epilogue
  pl.epi_stats = pl.rm || endpoint == 2 || (endpoint && (pl.BN < 128 || 4 * pl.BN <= K));
  pl.epi_t = !pl.rm && (endpoint == 2 || (endpoint && !pl.epi_stats));
  const int reserve = 2048 + (pl.epi_t ? kTransposeBytes : 0);
  auto stage_of = [&](int na) { return na * (kAtomBytes + pl.hilo * (pl.BN / 2) * 128); };
  // (a pair pays a cross-CTA hand-off per stage, so it prefers fewer,
  // larger stages: measured on 1024 rows x 256000 ids x 4608 with bf16
  // activations, three 128-column stages 1746 us, six 64-column 2005 us)
  pl.na = pl.fp8 ? 1 : (block_k == 64 ? 1 : (block_k == 256 ? 4 : 2));
  const int min_stages = block_k ? 2 : 3;
  while (pl.na > 1 && (int)((kSmemBudget - reserve) / stage_of(pl.na)) < min_stages) pl.na >>= 1;
  const int bk = pl.na * (pl.fp8 ? kAtomE8 : kAtomK);
  pl.KB = (K + bk - 1) / bk;
  pl.Kp = pl.KB * bk;
  pl.NT = (n + 255) / 256;
  const int tiles = pl.RB * pl.NT;
  pl.T = (long long)tiles * pl.KB;
  // pairs: as many as fit at once (the SMs of a GPU section pair up)
  int units = sm_count / 2;
  if (max_pairs > 0 && max_pairs < units) units = max_pairs;
  if (pl.RB > 1 && pl.RB <= units) units = units / pl.RB * pl.RB;
  const int g_whole = tiles < units ? tiles : units;
  const long long whole_span = (long long)((tiles + g_whole - 1) / g_whole) * pl.KB;
  const double split_span = (double)pl.T / (pl.T < units ? pl.T : units);
  pl.whole_tiles = schedule == 1 || (schedule == 0 && whole_span <= 1.1 * split_span + 2.0);
  units = pl.whole_tiles ? g_whole : (int)(pl.T < units ? pl.T : units);
  pl.G = 2 * units;
  pl.stages = (int)((kSmemBudget - reserve) / stage_of(pl.na));
  if (pl.stages > kMaxStages) pl.stages = kMaxStages;
  if (max_stages >= 2 && pl.stages > max_stages) pl.stages = max_stages;
  pl.hs_bytes = pl.fp8 ? align256((size_t)pl.hilo * pl.Rp * pl.Kp) + align256((size_t)pl.Rp * 4)
                       : align256((size_t)pl.hilo * pl.Rp * pl.Kp * 2);
  const bool splits = !pl.whole_tiles && (pl.T % units != 0 || (pl.T / units) % pl.KB != 0);
  pl.p_bytes = splits ? align256((size_t)2 * pl.G * pl.BN * 128 * 4) : 0;
  pl.cnt_bytes = align256((size_t)tiles * 4 * kEpiGroups * 2 * sizeof(int));
  pl.nseg = pl.NT * 8;
  pl.stats_bytes = endpoint ? align256((size_t)rows * pl.nseg * sizeof(float2)) : 0;
  pl.scratch_bytes = pl.hs_bytes + pl.p_bytes + pl.cnt_bytes + pl.stats_bytes;
  pl.smem_bytes = 1024 + (size_t)pl.stages * stage_of(pl.na) + kBarrierArea +
                  kMaxBoxes * sizeof(int2) + (pl.epi_t ? kTransposeBytes : 0);
  pl.ok = pl.stages >= 2;
  return pl;
}
}  // namespace

TcPlan tc_plan(int rows, int n, int K, int act_bf16, int sm_count, int endpoint,
               int schedule, int max_stages, int block_k, int gather, int fp8, int max_bn_opt,
               int tile_m, int pair_mode, int max_pairs, int rm_mode) {
  TcPlan pl{};
  // h planes: bf16 weights take one bf16 plane for bf16-rounded
  // activations (exact) and two (hi + lo) for fp32; e4m3 weights take two
  // e4m3 planes for bf16-rounded activations (exact) and four for fp32
  pl.hilo = fp8 ? (act_bf16 ? 2 : 4) : (act_bf16 ? 1 : 2);
  pl.fp8 = fp8;
  (void)gather;
  // CTA pairs: forced (pair_mode 2), or chosen (1) where their row blocks
  // are long enough that halving each SM's B bytes pays for the pair's
  // hand-offs: >= 128 rows.  Measured pair vs single: 1024 rows x 256000
  // ids x 4608 fp32 2654 vs 3191 us, bf16 (three stages) 1746 vs 2005; 256
  // rows x 256000 fp32 737 vs 897; 320 rows x 51302 x 3584 bf16 161 vs 195,
  // fp32 (160-row blocks) 182 vs 208 (with the pair hand-offs of today; 242
  // vs 223 before them); 32 rows x 12000 x 3840 38.9 vs 37.2; 64 rows x
  // 256000 x 4608 471 vs 433.
  // The endpoint (K = d_l) pairs from 192-row blocks: its B bytes per MMA
  // are most of its traffic (measured 1024 rows x 256000 ids x 512: 665 vs
  // 721 us; 256 rows: 189 vs 408), but 160-row blocks gain nothing (320
  // rows x 51302 x 512: 75.3 vs 71.6 us).
  // (an explicitly set tile height keeps single-CTA tiles unless pairs are
  // forced)
  if (pair_mode > 0 && sm_count >= 2 && (tile_m == 0 || pair_mode == 2)) {
    pl.pair = 1;
    const TcPlan pp = tc_plan_pair(pl, rows, n, K, sm_count, max_pairs, schedule, max_stages,
                                   block_k, max_bn_opt, endpoint, rm_mode);
    if (pair_mode == 2 || (!fp8 && pp.BN >= (endpoint ? 192 : 128))) return pp;
    pl.pair = 0;
  }
  const int atom = fp8 ? kAtomE8 : kAtomK;   // elements per 128-byte atom
  // e4m3: row blocks of up to 128 rows (measured on 256 rows x 152064 ids
  // x 7168, 256-id tiles: four planes 1229 / 996 / 743 us and two planes
  // 784 / 661 / 474 us at 64 / 96 / 128 rows -- fewer weight re-reads beat
  // deeper pipelines; 128-row blocks leave two 96 KB stages)
  int max_bn = fp8 ? 128 : kMaxBN;
  // two h planes: at most 224 rows, so that three stages fit (measured:
  // 1024 rows x 256k ids x 4608 runs 21 % faster in three 224-row stages
  // than in two 256-row ones)
  if (!fp8 && pl.hilo == 2 && max_bn > 224) max_bn = 224;
  if (max_bn_opt >= 16 && max_bn_opt < max_bn) max_bn = max_bn_opt;
  auto row_blocks = [&](int cap) {
    if (rows <= cap) {
      pl.RB = 1;
      pl.BN = (rows + 15) / 16 * 16;
    } else {
      pl.RB = (rows + cap - 1) / cap;
      pl.BN = ((rows + pl.RB - 1) / pl.RB + 15) / 16 * 16;
    }
  };
  row_blocks(max_bn);
  // 256-id tiles: two M = 128 MMAs share every B stage, which halves the
  // B bytes per A byte (more of the shared memory holds weights), but their
  // two double-buffered accumulators hold at most 128 hidden-state rows per
  // row block and the tiles are half as many.  Automatic: only where the
  // row blocks already have <= 128 rows, the hidden dimension is long and
  // there are >= 3/4 tiles per SM (measured over 8..256 rows, 30000..256000
  // ids, K 2048..8192: 4..44 % faster; decode's 47 tiles on 152 SMs, every
  // one split three or four ways, 10 % slower; the endpoint's short K and
  // 160..208-row blocks slower).
  // Row blocks of 129..192 rows also take 256-id tiles, with one
  // accumulator (three stages still fit; measured on 320 rows x 51302 ids x
  // 3584: 245 -> 227 us fp32 h, 233 -> 200 us bf16 h; 208-row blocks of
  // R = 1024 with two stages are slower).
  const bool wide_auto = !fp8 && pl.BN > 128 && pl.BN <= 192;
  const bool tm256_auto = tile_m == 0 && (pl.BN <= 128 || wide_auto) && K >= 2048 &&
                          4ll * pl.RB * ((n + 255) / 256) >= 3ll * sm_count;
  pl.tm = (tile_m == 256 || tm256_auto) ? 256 : 128;
  const int halves = pl.tm / 128;
  // 256-id tiles: row blocks of <= 128 rows keep two accumulators; asked
  // for with larger blocks (max_bn above 128), one accumulator holds up to
  // 256 rows and the epilogue no longer overlaps the next tile's MMAs
  pl.single_acc = 0;
  if (pl.tm == 256 && pl.BN > 128) {
    if ((tile_m == 256 && max_bn_opt > 128) || (tile_m == 0 && wide_auto)) pl.single_acc = 1;
    else row_blocks(max_bn < 128 ? max_bn : 128);
  }
  pl.Rp = pl.RB * pl.BN;
  // k-block width: as asked (automatic: 128), narrowed until the shared
  // memory holds at least min_stages pipeline stages.  The full vocabulary
  // with row blocks of at most 16 rows keeps 128 columns down to three
  // stages: one 3-D copy per stage then moves twice the bytes (measured, 8
  // rows x 256000 ids x 4608 on 256-id tiles: 383 us in three 72 KB stages
  // against 404 us in six 36 KB ones; with kept-id subsets, or 32 and 64
  // rows, the narrower stages are as fast or faster)
  pl.na = fp8 ? 1 : (block_k == 64 ? 1 : (block_k == 256 ? 4 : 2));
  const int min_stages = block_k ? 2 : ((!gather && pl.BN <= 16) ? 3 : 4);
  while (pl.na > 1 &&
         (int)((kSmemBudget - 2048) / (pl.na * (halves * kAtomBytes + pl.hilo * pl.BN * 128))) <
             min_stages)
    pl.na >>= 1;
  const int bk = pl.na * atom;
  pl.KB = (K + bk - 1) / bk;
  pl.Kp = pl.KB * bk;
  pl.NT = (n + pl.tm - 1) / pl.tm;
  const int tiles = pl.RB * pl.NT;
  pl.T = (long long)tiles * pl.KB;
  // CTAs: with several row blocks, a multiple of the row-block count, so
  // that every row block's iterations split at the same offsets and the
  // CTAs that stream the same weight tile for different row blocks run in
  // step (one reads it from DRAM, the others from L2).  Measured on 1024
  // rows x 25600 ids x 4608 in five row blocks: 152 CTAs (ranges offset by
  // 2.6 tiles between row blocks) read 5.6x the kept weights from DRAM.
  int sm_use = sm_count;
  if (pl.RB > 1 && pl.RB <= sm_count) sm_use = sm_count / pl.RB * pl.RB;
  // whole tiles per CTA unless that leaves the grid clearly unbalanced
  const int g_whole = tiles < sm_use ? tiles : sm_use;
  const long long whole_span = (long long)((tiles + g_whole - 1) / g_whole) * pl.KB;
  const double split_span = (double)pl.T / (pl.T < sm_use ? pl.T : sm_use);
  pl.whole_tiles = schedule == 1 || (schedule == 0 && whole_span <= 1.1 * split_span + 2.0);
  pl.G = pl.whole_tiles ? g_whole : (int)(pl.T < sm_use ? pl.T : sm_use);
  const int stage_bytes = pl.na * (halves * kAtomBytes + pl.hilo * pl.BN * 128);
  // endpoint: the epilogue makes the segment statistics where z is not
  // stored (endpoint == 2) or where the hidden dimension hides them (below);
  // without them, or without z, it transposes each warp's chunk through
  // shared memory (kTransposeBytes beside the stages)
  pl.epi_stats = endpoint == 2 || (endpoint && (pl.BN < 128 || 4 * pl.BN <= K));
  pl.epi_t = endpoint == 2 || (endpoint && !pl.epi_stats);
  pl.stages = (int)((kSmemBudget - 2048 - (pl.epi_t ? kTransposeBytes : 0)) / stage_bytes);
  if (pl.stages > kMaxStages) pl.stages = kMaxStages;
  if (max_stages >= 2 && pl.stages > max_stages) pl.stages = max_stages;
  // h planes (bf16 or e4m3), and with e4m3 the per-row scales after them
  pl.hs_bytes = fp8 ? align256((size_t)pl.hilo * pl.Rp * pl.Kp) + align256((size_t)pl.Rp * 4)
                    : align256((size_t)pl.hilo * pl.Rp * pl.Kp * 2);
  // split tiles exist only when a CTA's range does not cover whole tiles
  const bool splits = !pl.whole_tiles && (pl.T % pl.G != 0 || (pl.T / pl.G) % pl.KB != 0);
  pl.p_bytes = splits ? align256((size_t)2 * pl.G * pl.BN * pl.tm * 4) : 0;
  pl.cnt_bytes = align256((size_t)tiles * 4 * kEpiGroups * sizeof(int));
  pl.nseg = pl.NT * (pl.tm / 32);
  pl.stats_bytes = endpoint ? align256((size_t)rows * pl.nseg * sizeof(float2)) : 0;
  // the epilogue's statistics are latency-bound chains of shuffles and
  // exponentials per 16 rows, hidden behind the next tile's MMAs only when
  // the hidden dimension is long enough; otherwise a separate pass over z at
  // memory speed is cheaper (measured: 320 rows x 51302 ids x 512 and
  // 1024 rows x 256000 ids x 512 gain; 256 rows x 152064 ids x 1024 loses)
  pl.scratch_bytes = pl.hs_bytes + pl.p_bytes + pl.cnt_bytes + pl.stats_bytes;
  pl.smem_bytes = 1024 + (size_t)pl.stages * stage_bytes + kBarrierArea + kMaxBoxes * sizeof(int2) +
                  (pl.epi_t ? kTransposeBytes : 0);
  pl.ok = pl.stages >= 2;
  return pl;
}

template <int HILO, bool GATHER, int EPI, bool FP8 = false, int TM = 128, bool PAIR = false>
static cudaError_t launch_inst(const WMaps& mw, const CUtensorMap& mh,
                               const TcParams& prm, const TcPlan& pl,
                               cudaStream_t st) {
  auto kern = tc_kernel<HILO, GATHER, EPI, FP8, TM, PAIR>;
  // the shared-memory opt-in, raised only when a launch needs more than any
  // earlier one on this device (a host call per launch otherwise)
  static std::atomic<int> configured[kMaxDevices];
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::atomic<int>* cfg = dev >= 0 && dev < kMaxDevices ? &configured[dev] : nullptr;
  if (!cfg || cfg->load() < (int)pl.smem_bytes) {
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)pl.smem_bytes);
    if (e != cudaSuccess) return e;
    if (cfg) {
      int cur = cfg->load();
      while (cur < (int)pl.smem_bytes && !cfg->compare_exchange_weak(cur, (int)pl.smem_bytes)) {
      }
    }
  }
  if constexpr (PAIR)
    return launch_pdl_cluster(kern, dim3(pl.G), dim3(kThreads), pl.smem_bytes, st, 2,
                              mw, mh, prm);
  return launch_pdl(kern, dim3(pl.G), dim3(kThreads), pl.smem_bytes, st,
                    mw, mh, prm);
}

int tc_pair_max_units(int device) {
  static std::atomic<int> cache[kMaxDevices];
  if (device < 0 || device >= kMaxDevices) return 0;
  const int c = cache[device].load();
  if (c) return c;
  // the largest shared memory a pair launch asks for
  auto kern = tc_kernel<2, false, EPI_CLOUD, false, 128, true>;
  const int smem = (int)(kSmemBudget + 1024 + kBarrierArea + kMaxBoxes * sizeof(int2));
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) !=
      cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(2);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess || n < 1) {
    cudaGetLastError();
    return 0;
  }
  cache[device].store(n);
  return n;
}

cudaError_t launch_tc(const GatherGemm& g, const TcPlan& pl, void* scratch,
                      long long spin_limit, cudaStream_t st) {
  const bool fp8 = g.w_dtype == W_FP8;
  if (!pl.ok || (fp8 != (pl.fp8 != 0)) || (fp8 && g.epilogue != EPI_CLOUD) ||
      (pl.pair && (pl.G % 2 || pl.BN % 32)) ||
      (pl.rm && (!pl.pair || pl.BN != 256 || !pl.whole_tiles || g.epilogue == EPI_CLOUD)) ||
      (g.epilogue != EPI_CLOUD && pl.hilo != 2) ||
      (g.epilogue == EPI_FUSED && (!g.yc || !g.rowmax_in || !g.codes_out || !g.scale_out)))
    return cudaErrorNotSupported;
  char* sc = static_cast<char*>(scratch);
  auto* Hs = reinterpret_cast<__nv_bfloat16*>(sc);
  float* P = pl.p_bytes ? reinterpret_cast<float*>(sc + pl.hs_bytes) : nullptr;
  int* counters = reinterpret_cast<int*>(sc + pl.hs_bytes + pl.p_bytes);
  float2* stats = pl.stats_bytes
                      ? reinterpret_cast<float2*>(sc + pl.hs_bytes + pl.p_bytes + pl.cnt_bytes)
                      : nullptr;
  const bool gather = g.ids != nullptr;
  const int tiles = pl.RB * pl.NT;

  // e4m3 planes of h (1 byte per element) and, after them, the rows' scales
  float* h_scale = fp8 ? reinterpret_cast<float*>(
                             sc + align256((size_t)pl.hilo * pl.Rp * pl.Kp))
                       : nullptr;
  if (fp8) {
    cudaError_t e = launch_pdl(split_h_e4m3_kernel, dim3(pl.Rp), dim3(kSplit8Threads), 0, st,
                               g.h, g.ld_h, g.rows, g.K, pl.Rp, pl.Kp, pl.hilo,
                               reinterpret_cast<uint8_t*>(sc), h_scale, counters,
                               tiles * 4 * kEpiGroups * (pl.pair ? 2 : 1), g.rowmax, g.act_bf16);
    if (e != cudaSuccess) return e;
  } else {
    const int64_t groups = (int64_t)pl.Rp * pl.Kp / 8;
    int blocks = (int)((groups + kSplitThreads - 1) / kSplitThreads);
    if (blocks > 4096) blocks = 4096;
    if (blocks < 1) blocks = 1;
    cudaError_t e = launch_pdl(split_h_kernel, dim3(blocks), dim3(kSplitThreads), 0, st, g.h, g.ld_h,
                               g.rows, g.K, pl.Rp, pl.Kp, pl.hilo, Hs, counters,
                               tiles * 4 * kEpiGroups * (pl.pair ? 2 : 1),
                               g.epilogue == EPI_CLOUD ? g.rowmax : (unsigned*)nullptr);
    if (e != cudaSuccess) return e;
  }

  WMaps mw;
  alignas(64) CUtensorMap mh;
  if (!w_maps(g, gather, mw)) return cudaErrorInvalidValue;
  const CUtensorMapDataType dt =
      fp8 ? CU_TENSOR_MAP_DATA_TYPE_UINT8 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
  const int atom = fp8 ? kAtomE8 : kAtomK;
  const int esz = fp8 ? 1 : 2;
  // h planes [hilo * Rp rows, Kp columns], zero padded: all atoms of a
  // stage in one copy per plane
  // (a pair's CTAs each take half of the block's rows)
  if (!cached_map3(&mh, dt, sc, (uint64_t)pl.Kp, (uint64_t)pl.hilo * pl.Rp,
                   (uint64_t)pl.Kp * esz, (uint32_t)(pl.pair ? pl.BN / 2 : pl.BN),
                   (uint32_t)pl.na, atom))
    return cudaErrorInvalidValue;
  // full vocabulary with a width that is a multiple of the atom: A likewise
  const int a3d = (!gather && g.K % atom == 0 && g.K >= pl.na * atom) ? 1 : 0;
  mw.a3 = CUtensorMap{};
  if (a3d && !cached_map3(&mw.a3, dt, g.W, (uint64_t)g.K, (uint64_t)g.V,
                          (uint64_t)g.ld_w * esz, (uint32_t)pl.tm, (uint32_t)pl.na, atom))
    return cudaErrorInvalidValue;

  TcParams prm{};
  prm.R = g.rows; prm.n = g.n; prm.K = g.K; prm.KB = pl.KB; prm.NT = pl.NT;
  prm.RB = pl.RB; prm.BN = pl.BN; prm.Rp = pl.Rp; prm.stages = pl.stages;
  prm.whole_tiles = pl.whole_tiles; prm.T = pl.T; prm.na = pl.na; prm.nseg = pl.nseg;
  prm.ids = g.ids;
  prm.h_scale = h_scale;
  prm.ld_w = g.ld_w;
  prm.w_scale = fp8 ? g.w_scale : nullptr;
  prm.epilogue = g.epilogue; prm.bias = g.bias;
  prm.ldy = g.ldy ? g.ldy : g.n;
  prm.yc = g.yc; prm.rowmax_in = g.rowmax_in; prm.codes_out = g.codes_out;
  prm.scale_out = g.scale_out;
  prm.clip = g.clip; prm.partial_out = g.partial_out; prm.Y = g.Y;
  prm.rowmax = g.rowmax; prm.codes = g.codes; prm.row_scale = g.row_scale;
  prm.single_acc = pl.single_acc;
  prm.inv_tau = g.inv_tau; prm.seg_stats = (pl.epi_stats && !g.no_stats) ? stats : nullptr; prm.a3d = a3d;
  // (2-element-aligned rows of codes and of a stored z: n and the z stride
  // even)
  const bool et = pl.epi_t && g.epilogue == EPI_ENDPOINT && g.n % 2 == 0 &&
                 (!g.Y || (prm.ldy % 2 == 0 && (reinterpret_cast<uintptr_t>(g.Y) & 7) == 0)) &&
                 (reinterpret_cast<uintptr_t>(g.codes) & 1) == 0;
  prm.P = P; prm.counters = counters;
  prm.status = g.status; prm.spin_limit = spin_limit; prm.finish_wait = g.finish_wait;

  const bool hilo2 = pl.hilo == 2;
  if (pl.pair && fp8) {
    if (gather) return hilo2 ? launch_inst<2, true, EPI_CLOUD, true, 128, true>(mw, mh, prm, pl, st)
                             : launch_inst<4, true, EPI_CLOUD, true, 128, true>(mw, mh, prm, pl, st);
    return hilo2 ? launch_inst<2, false, EPI_CLOUD, true, 128, true>(mw, mh, prm, pl, st)
                 : launch_inst<4, false, EPI_CLOUD, true, 128, true>(mw, mh, prm, pl, st);
  }
  if (pl.rm) {
    if (g.epilogue == EPI_FUSED)
      return gather ? launch_inst<2, true, EPI_FUSED_RM, false, 128, true>(mw, mh, prm, pl, st)
                    : launch_inst<2, false, EPI_FUSED_RM, false, 128, true>(mw, mh, prm, pl, st);
    return gather ? launch_inst<2, true, EPI_ENDPOINT_RM, false, 128, true>(mw, mh, prm, pl, st)
                  : launch_inst<2, false, EPI_ENDPOINT_RM, false, 128, true>(mw, mh, prm, pl, st);
  }
  if (pl.pair) {
    if (g.epilogue == EPI_FUSED)
      return gather ? launch_inst<2, true, EPI_FUSED, false, 128, true>(mw, mh, prm, pl, st)
                    : launch_inst<2, false, EPI_FUSED, false, 128, true>(mw, mh, prm, pl, st);
    if (et)
      return gather ? launch_inst<2, true, EPI_ENDPOINT_T, false, 128, true>(mw, mh, prm, pl, st)
                    : launch_inst<2, false, EPI_ENDPOINT_T, false, 128, true>(mw, mh, prm, pl, st);
    if (g.epilogue == EPI_ENDPOINT)
      return gather ? launch_inst<2, true, EPI_ENDPOINT, false, 128, true>(mw, mh, prm, pl, st)
                    : launch_inst<2, false, EPI_ENDPOINT, false, 128, true>(mw, mh, prm, pl, st);
    if (gather) return hilo2 ? launch_inst<2, true, EPI_CLOUD, false, 128, true>(mw, mh, prm, pl, st)
                             : launch_inst<1, true, EPI_CLOUD, false, 128, true>(mw, mh, prm, pl, st);
    return hilo2 ? launch_inst<2, false, EPI_CLOUD, false, 128, true>(mw, mh, prm, pl, st)
                 : launch_inst<1, false, EPI_CLOUD, false, 128, true>(mw, mh, prm, pl, st);
  }
  if (pl.tm == 256) {
    if (fp8) {
      if (gather) return hilo2 ? launch_inst<2, true, EPI_CLOUD, true, 256>(mw, mh, prm, pl, st)
                               : launch_inst<4, true, EPI_CLOUD, true, 256>(mw, mh, prm, pl, st);
      return hilo2 ? launch_inst<2, false, EPI_CLOUD, true, 256>(mw, mh, prm, pl, st)
                   : launch_inst<4, false, EPI_CLOUD, true, 256>(mw, mh, prm, pl, st);
    }
    if (g.epilogue == EPI_CLOUD) {
      if (gather) return hilo2 ? launch_inst<2, true, EPI_CLOUD, false, 256>(mw, mh, prm, pl, st)
                               : launch_inst<1, true, EPI_CLOUD, false, 256>(mw, mh, prm, pl, st);
      return hilo2 ? launch_inst<2, false, EPI_CLOUD, false, 256>(mw, mh, prm, pl, st)
                   : launch_inst<1, false, EPI_CLOUD, false, 256>(mw, mh, prm, pl, st);
    }
    // (the endpoint's activations are always fp32-exact: two planes)
    if (g.epilogue == EPI_FUSED)
      return gather ? launch_inst<2, true, EPI_FUSED, false, 256>(mw, mh, prm, pl, st)
                    : launch_inst<2, false, EPI_FUSED, false, 256>(mw, mh, prm, pl, st);
    if (et)
      return gather ? launch_inst<2, true, EPI_ENDPOINT_T, false, 256>(mw, mh, prm, pl, st)
                    : launch_inst<2, false, EPI_ENDPOINT_T, false, 256>(mw, mh, prm, pl, st);
    return gather ? launch_inst<2, true, EPI_ENDPOINT, false, 256>(mw, mh, prm, pl, st)
                  : launch_inst<2, false, EPI_ENDPOINT, false, 256>(mw, mh, prm, pl, st);
  }
  if (fp8) {                // four e4m3 planes of h, or two for bf16-rounded h
    if (gather) return hilo2 ? launch_inst<2, true, EPI_CLOUD, true>(mw, mh, prm, pl, st)
                             : launch_inst<4, true, EPI_CLOUD, true>(mw, mh, prm, pl, st);
    return hilo2 ? launch_inst<2, false, EPI_CLOUD, true>(mw, mh, prm, pl, st)
                 : launch_inst<4, false, EPI_CLOUD, true>(mw, mh, prm, pl, st);
  }
  if (g.epilogue == EPI_CLOUD) {
    if (gather) return hilo2 ? launch_inst<2, true, EPI_CLOUD>(mw, mh, prm, pl, st)
                             : launch_inst<1, true, EPI_CLOUD>(mw, mh, prm, pl, st);
    return hilo2 ? launch_inst<2, false, EPI_CLOUD>(mw, mh, prm, pl, st)
                 : launch_inst<1, false, EPI_CLOUD>(mw, mh, prm, pl, st);
  }
  if (g.epilogue == EPI_FUSED)
    return gather ? launch_inst<2, true, EPI_FUSED>(mw, mh, prm, pl, st)
                  : launch_inst<2, false, EPI_FUSED>(mw, mh, prm, pl, st);
  if (et)
    return gather ? launch_inst<2, true, EPI_ENDPOINT_T>(mw, mh, prm, pl, st)
                  : launch_inst<2, false, EPI_ENDPOINT_T>(mw, mh, prm, pl, st);
  return gather ? launch_inst<2, true, EPI_ENDPOINT>(mw, mh, prm, pl, st)
                : launch_inst<2, false, EPI_ENDPOINT>(mw, mh, prm, pl, st);
}

cudaError_t launch_sample_from_stats(const ZSource& zs, int rows, int n, const TcPlan& pl,
                                     const void* scratch, float2* cstats,
                                     const int32_t* ids, float inv_tau, uint64_t seed,
                                     uint64_t offset, int sm_count, int32_t* tokens,
                                     cudaStream_t st, int greedy) {
  const char* sc = static_cast<const char*>(scratch);
  const float2* stats =
      reinterpret_cast<const float2*>(sc + pl.hs_bytes + pl.p_bytes + pl.cnt_bytes);
  if (!pl.epi_stats) {
    if (!zs.Z) return cudaErrorInvalidValue;
    float2* sst = const_cast<float2*>(stats);
    cudaError_t e = launch_seg_stats(zs.Z, rows, n, inv_tau, sst, cstats, sm_count, st);
    if (e != cudaSuccess) return e;
    return launch_sample_segments(zs, rows, n, sst, seg_count(n), cstats, ids, inv_tau, seed,
                                  offset, tokens, st, greedy);
  }
  const int nseg = pl.nseg;
  if (greedy)   // the segment maxima are all greedy decoding needs
    return launch_sample_segments(zs, rows, n, stats, nseg, nullptr, ids, inv_tau, seed, offset,
                                  tokens, st, 1);
  if (chunk_count(nseg) <= 4096)
    return launch_sample_rows(zs, rows, n, stats, nseg, ids, inv_tau, seed, offset, tokens, st);
  cudaError_t e = launch_chunk_stats(stats, rows, nseg, inv_tau, cstats, sm_count, st);
  if (e != cudaSuccess) return e;
  return launch_sample_segments(zs, rows, n, stats, nseg, cstats, ids, inv_tau, seed, offset,
                                tokens, st);
}

}  // namespace sph
