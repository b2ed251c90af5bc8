// Row-wise softmax statistics, inverse-CDF draws and speculative
// verification over fused logits z (fp32 [rows, n], ascending compact ids).
//
//   seg_stats : per 32-id segment of every row, (max z, sum exp((z - max)/tau))
//   sample    : Eq. 14-15, one Philox uniform per row, inverse CDF
//   verify    : standard speculative acceptance of k drafts per session with
//               a residual draw at the first rejection (Sec. "Endpoint
//               Speculative Decoding and Cloud Verification", Algorithm 1)
//
// Every pass is spread over the whole GPU: the statistics pass reads each
// logit once (the only HBM-sized pass), the row reductions and draws work on
// the 32x smaller segment statistics.  A draw is a three-level search in
// ascending id order -- 1024-id chunks, 32-id segments, ids -- whose CDF is
// the oracle's up to fp32 rounding.
#include <climits>

#include "sm100_ptx.cuh"
#include "sph_common.cuh"
#include "sph_internal.h"

namespace sph {
namespace {

constexpr int kSeg = 32;                // ids per segment (one per lane)
constexpr int kGroup = 16;              // segments per half chunk (one reduce-scatter)
constexpr int kWarps = 8;               // warps per CTA
constexpr int kMaxN = 1 << 30;          // ids per row
constexpr int kMaxK = 64;               // drafts per session

// exp(d / tau) for the per-logit passes, as 2^(d * (log2(e) / tau)): the
// scale is one fp32 rounding of log2(e) / tau (relative 2^-24, so an error of
// at most |d / tau| * 6e-8 in the exponent), and 2^x is the special-function
// unit's approximation (ex2_approx).
constexpr float kLog2e = 1.4426950408889634f;
__device__ __forceinline__ float exp_tau(float d, float log2e_inv_tau) {
  return ex2_approx(d * log2e_inv_tau);
}

__device__ __forceinline__ float seg_weight(float2 st, float M, float inv_tau) {
  return st.y > 0.f ? st.y * expf((st.x - M) * inv_tau) : 0.f;
}

// ---------------------------------------------------------------------------
// statistics: a warp takes one 1024-id chunk (32 segments) of one row, a
// lane one 32-id segment
// ---------------------------------------------------------------------------
// The warp reads the chunk with coalesced loads (16-byte where the row is so
// aligned) into its shared-memory tile, segment s at words 36 s .. 36 s + 31
// (the padding keeps the stores and the lanes' 16-byte reads free of bank
// conflicts), then each lane reduces its segment's max and sum of exp in
// registers as balanced trees.  That is a handful of instructions per logit
// where the warp-wide reduce-scatter it replaces spent about eight (issue-
// bound at 45 % of HBM); a lane reading its own 128 bytes straight from
// global memory instead made every load touch 32 lines (47.6 us against
// 22.5 us on the spec workload's 66 MB).
constexpr int kSegRow = 36;             // words per segment in the tile
__global__ void __launch_bounds__(kWarps * 32)
seg_stats_kernel(const float* __restrict__ Z, int rows, int n, int nseg, int nchunk,
                 float inv_tau, float2* __restrict__ stats, float2* __restrict__ cstats) {
  __shared__ __align__(16) float tile[kWarps][kSeg * kSegRow];
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  const int lane = threadIdx.x & 31;
  float* tb = tile[threadIdx.x >> 5];
  const float l2t = inv_tau * kLog2e;
  const long long total = (long long)nchunk * rows;
  const long long nwarps = (long long)gridDim.x * kWarps;
  const bool narrow = total <= INT_MAX;
  for (long long g = (long long)blockIdx.x * kWarps + (threadIdx.x >> 5); g < total;
       g += nwarps) {
    long long r;
    int c;
    if (narrow) {
      const unsigned rr = (unsigned)g / (unsigned)nchunk;
      r = rr;
      c = (int)((unsigned)g - rr * (unsigned)nchunk);
    } else {
      r = g / nchunk;
      c = (int)(g - r * nchunk);
    }
    const int j0 = c * kSeg * kSeg;             // the chunk's first id
    const float* z = Z + r * n + j0;
    const int left = n - j0;                    // ids of the row from j0 on
    __syncwarp();                               // (the previous item's reads)
    if (left >= kSeg * kSeg && ((reinterpret_cast<uintptr_t>(z) & 15) == 0)) {
#pragma unroll
      for (int q = 0; q < kSeg / 4; ++q) {
        const float4 t = __ldcs(reinterpret_cast<const float4*>(z) + q * 32 + lane);
        *reinterpret_cast<float4*>(tb + (q * 4 + (lane >> 3)) * kSegRow + 4 * (lane & 7)) = t;
      }
    } else {
#pragma unroll 8
      for (int q = 0; q < kSeg; ++q) {
        const int e = q * 32 + lane;
        tb[q * kSegRow + lane] = e < left ? __ldcs(z + e) : -INFINITY;
      }
    }
    __syncwarp();
    float v[kSeg];
#pragma unroll
    for (int m = 0; m < kSeg / 4; ++m) {
      const float4 t = *reinterpret_cast<const float4*>(tb + lane * kSegRow + 4 * m);
      v[4 * m] = t.x; v[4 * m + 1] = t.y; v[4 * m + 2] = t.z; v[4 * m + 3] = t.w;
    }
    const int sg = c * kSeg + lane;             // this lane's segment
    float t[kSeg / 2];
#pragma unroll
    for (int q = 0; q < kSeg / 2; ++q) t[q] = fmaxf(v[2 * q], v[2 * q + 1]);
#pragma unroll
    for (int w = kSeg / 4; w >= 1; w >>= 1)
#pragma unroll
      for (int q = 0; q < w; ++q) t[q] = fmaxf(t[2 * q], t[2 * q + 1]);
    const float m = t[0];
    float sum = 0.f;
    if (m > -INFINITY) {
      // exp of -inf (ids past n) is 0
#pragma unroll
      for (int q = 0; q < kSeg / 2; ++q)
        t[q] = exp_tau(v[2 * q] - m, l2t) + exp_tau(v[2 * q + 1] - m, l2t);
#pragma unroll
      for (int w = kSeg / 4; w >= 1; w >>= 1)
#pragma unroll
        for (int q = 0; q < w; ++q) t[q] = t[2 * q] + t[2 * q + 1];
      sum = t[0];
    }
    if (sg < nseg) stats[r * nseg + sg] = make_float2(m, sum);
    const float Mc = warp_max(m);
    const float Sc = warp_sum(seg_weight(make_float2(m, sum), Mc, inv_tau));
    if (lane == 0) cstats[r * nchunk + c] = make_float2(Mc, Sc);
  }
}

// Chunk statistics from segment statistics (rows of `nseg` entries): a warp
// per chunk.
__global__ void __launch_bounds__(kWarps * 32)
chunk_stats_kernel(const float2* __restrict__ stats, int rows, int nseg, int nchunk,
                   float inv_tau, float2* __restrict__ cstats) {
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  const int lane = threadIdx.x & 31;
  const long long total = (long long)nchunk * rows;
  const long long nwarps = (long long)gridDim.x * kWarps;
  for (long long g = (long long)blockIdx.x * kWarps + (threadIdx.x >> 5); g < total;
       g += nwarps) {
    const long long r = g / nchunk;
    const int c = (int)(g - r * nchunk);
    const int sg = c * kSeg + lane;
    const float2 st = sg < nseg ? stats[r * nseg + sg] : make_float2(-INFINITY, 0.f);
    const float Mc = warp_max(st.x);
    const float Sc = warp_sum(seg_weight(st, Mc, inv_tau));
    if (lane == 0) cstats[r * nchunk + c] = make_float2(Mc, Sc);
  }
}

// ---------------------------------------------------------------------------
// warp-level inverse CDF over three levels: chunks, segments, ids
// ---------------------------------------------------------------------------
__device__ __forceinline__ float warp_incl_scan(float x, int lane) {
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const float t = __shfl_up_sync(0xFFFFFFFFu, x, o);
    if (lane >= o) x += t;
  }
  return x;
}

// Within 32 consecutive weights w (one per lane) find the first lane whose
// running sum from `before` exceeds target; the last lane with weight if
// rounding leaves none; lane 0 if all are zero.  Updates `before`.
__device__ __forceinline__ int scan_pick(float w, float target, float& before, int lane) {
  const float incl = warp_incl_scan(w, lane);
  const unsigned hit = __ballot_sync(0xFFFFFFFFu, w > 0.f && target < before + incl);
  const unsigned nz = __ballot_sync(0xFFFFFFFFu, w > 0.f);
  const int l = hit ? __ffs(hit) - 1 : (nz ? 31 - __clz(nz) : 0);
  before += __shfl_sync(0xFFFFFFFFu, incl - w, l);
  return l;
}

// Draw with chunk weights cw(c) (c < nchunk), segment weights sw(s)
// (s < nseg) and id weights ew(j) (j < n): the first id, in ascending order,
// at which the running weight sum exceeds u * total.  Each lane first sums
// a contiguous run of chunks; the warp then scans the run that holds the
// target 32 chunks at a time, then that chunk's segments, then the
// segment's ids.  Returns the total weight (the draw is void if it is 0);
// all lanes receive the same j.  warp_draw_segment stops after the segment
// (the target and the weight before the segment in target/before), for
// callers that make the segment's id weights themselves.
template <class CW, class SW>
__device__ __forceinline__ float warp_draw_segment(int nchunk, int nseg, const CW& cw,
                                                   const SW& sw, float u, int lane,
                                                   int& seg_out, float& target_out,
                                                   float& before_out) {
  const int per = (nchunk + 31) / 32;
  const int c0 = min(nchunk, lane * per), c1 = min(nchunk, c0 + per);
  float local = 0.f;
  int c = c0;
  for (; c + 4 <= c1; c += 4) {
    const float a0 = cw(c), a1 = cw(c + 1), a2 = cw(c + 2), a3 = cw(c + 3);
    local += a0; local += a1; local += a2; local += a3;
  }
  for (; c < c1; ++c) local += cw(c);
  const float incl = warp_incl_scan(local, lane);
  const float total = __shfl_sync(0xFFFFFFFFu, incl, 31);
  const float target = u * total;
  const unsigned hit = __ballot_sync(0xFFFFFFFFu, local > 0.f && target < incl);
  const unsigned nz = __ballot_sync(0xFFFFFFFFu, local > 0.f);
  const int owner = hit ? __ffs(hit) - 1 : (nz ? 31 - __clz(nz) : 0);
  float before = __shfl_sync(0xFFFFFFFFu, incl - local, owner);
  const int o0 = __shfl_sync(0xFFFFFFFFu, c0, owner);
  const int o1 = __shfl_sync(0xFFFFFFFFu, c1, owner);
  int chunk = -1, last_chunk = o0;
  float before_last = before;
  for (int b0 = o0; b0 < o1 && chunk < 0; b0 += 32) {
    const int cc = b0 + lane;
    const float w = cc < o1 ? cw(cc) : 0.f;
    const float inc = warp_incl_scan(w, lane);
    const unsigned h2 = __ballot_sync(0xFFFFFFFFu, w > 0.f && target < before + inc);
    const unsigned z2 = __ballot_sync(0xFFFFFFFFu, w > 0.f);
    if (h2) {
      const int l = __ffs(h2) - 1;
      chunk = b0 + l;
      before += __shfl_sync(0xFFFFFFFFu, inc - w, l);
    } else {
      if (z2) {
        const int l = 31 - __clz(z2);
        last_chunk = b0 + l;
        before_last = before + __shfl_sync(0xFFFFFFFFu, inc - w, l);
      }
      before += __shfl_sync(0xFFFFFFFFu, inc, 31);
    }
  }
  if (chunk < 0) { chunk = last_chunk; before = before_last; }
  const int s = chunk * kSeg + lane;
  const int ls = scan_pick(s < nseg ? sw(s) : 0.f, target, before, lane);
  seg_out = chunk * kSeg + ls;
  target_out = target;
  before_out = before;
  return total;
}
template <class CW, class SW, class EW>
__device__ __forceinline__ float warp_draw(int nchunk, int nseg, int n, const CW& cw,
                                           const SW& sw, const EW& ew, float u, int lane,
                                           int& j_out) {
  int seg;
  float target, before;
  const float total = warp_draw_segment(nchunk, nseg, cw, sw, u, lane, seg, target, before);
  const int j = seg * kSeg + lane;
  const int lj = scan_pick(j < n ? ew(j) : 0.f, target, before, lane);
  j_out = min(seg * kSeg + lj, n - 1);
  return total;
}

struct StatsWeight {                    // chunk or segment weight relative to M
  const float2* st;
  float M, inv_tau;
  __device__ float operator()(int s) const { return seg_weight(st[s], M, inv_tau); }
};
// A row of fused logits as the draws read it (z(j) for j < n): stored, or
// recomputed id by id from the endpoint's inputs (ZSource).  A draw reads
// the 32 ids of one segment, one per lane, so a recomputing lane takes one
// K-long dot product: the z a draw needs cost 32 weight rows per row
// instead of a store and a reload of all n.
struct ZRowStored {
  const float* z;
  __device__ float operator()(int j) const { return z[j]; }
};
struct ZRowRecomputed {
  const float* h;          // the row's hidden state, K values
  int K;
  const uint16_t* W;       // bf16 weight rows, ld_w elements apart (16-byte aligned)
  int64_t ld_w;
  const int32_t* ids;      // compact index -> weight row (nullptr: identity)
  const int8_t* c;         // the row's codes, or nullptr (no payload)
  float s;                 // the row's scale
  bool h16;                // h is 16-byte aligned
  __device__ void dot8(const uint4& wv, int k, float (&a)[4]) const {
    float x[8];
    if (h16) {
      const float4 x0 = __ldg(reinterpret_cast<const float4*>(h + k));
      const float4 x1 = __ldg(reinterpret_cast<const float4*>(h + k) + 1);
      x[0] = x0.x; x[1] = x0.y; x[2] = x0.z; x[3] = x0.w;
      x[4] = x1.x; x[5] = x1.y; x[6] = x1.z; x[7] = x1.w;
    } else {
#pragma unroll
      for (int e = 0; e < 8; ++e) x[e] = __ldg(h + k + e);
    }
    const unsigned u[4] = {wv.x, wv.y, wv.z, wv.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {     // element 2e in the low half, 2e + 1 in the high
      a[e] = fmaf(x[2 * e], __uint_as_float(u[e] << 16), a[e]);
      a[e] = fmaf(x[2 * e + 1], __uint_as_float(u[e] & 0xFFFF0000u), a[e]);
    }
  }
  __device__ float operator()(int j) const {
    const int id = ids ? __ldg(ids + j) : j;
    const uint16_t* w = W + (int64_t)id * ld_w;
    float a[4] = {0.f, 0.f, 0.f, 0.f};
    int k = 0;
    // the draw is latency-bound: eight 16-byte loads of the row in flight
#pragma unroll 1
    for (; k + 64 <= K; k += 64) {
      uint4 wv[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) wv[q] = __ldg(reinterpret_cast<const uint4*>(w + k) + q);
#pragma unroll
      for (int q = 0; q < 8; ++q) dot8(wv[q], k + 8 * q, a);
    }
#pragma unroll 1
    for (; k + 8 <= K; k += 8) dot8(__ldg(reinterpret_cast<const uint4*>(w + k)), k, a);
    for (; k < K; ++k) a[0] = fmaf(__ldg(h + k), __uint_as_float((unsigned)w[k] << 16), a[0]);
    const float z = (a[0] + a[1]) + (a[2] + a[3]);
    return c ? fmaf((float)__ldg(c + j), s, z) : z;
  }
  // The same z by the whole warp (every lane gets it): lane l takes the
  // 8-element pieces l, l + 32, ... of the row, then a warp sum.
  __device__ float coop(int j, int lane) const {
    const int id = ids ? __ldg(ids + j) : j;
    const uint16_t* w = W + (int64_t)id * ld_w;
    float a[4] = {0.f, 0.f, 0.f, 0.f};
    const int K8 = K & ~7;
    for (int k = 8 * lane; k < K8; k += 256) dot8(__ldg(reinterpret_cast<const uint4*>(w + k)), k, a);
    for (int k = K8 + lane; k < K; k += 32)
      a[0] = fmaf(__ldg(h + k), __uint_as_float((unsigned)w[k] << 16), a[0]);
    const float z = warp_sum((a[0] + a[1]) + (a[2] + a[3]));
    return c ? fmaf((float)__ldg(c + j), s, z) : z;
  }
};
struct ZRowsStored {
  static constexpr bool kRecompute = false;
  const float* Z;
  int n;
  __device__ ZRowStored row(int64_t r) const { return ZRowStored{Z + r * n}; }
};
struct ZRowsRecomputed {
  static constexpr bool kRecompute = true;
  ZSource zs;
  int n;
  __device__ ZRowRecomputed row(int64_t r) const {
    const float* hr = zs.h + r * zs.ld_h;
    return ZRowRecomputed{hr, zs.K, static_cast<const uint16_t*>(zs.W), zs.ld_w,
                          zs.ids, zs.codes ? zs.codes + r * n : nullptr,
                          zs.codes ? __ldg(zs.row_scale + r) : 0.f,
                          (reinterpret_cast<uintptr_t>(hr) & 15) == 0};
  }
};

template <class ZR>
struct ExpWeightOf {                    // exp((z_j - M) / tau)
  ZR z;
  float M, inv_tau;
  __device__ float operator()(int j) const { return expf((z(j) - M) * inv_tau); }
};
using ExpWeight = ExpWeightOf<ZRowStored>;
// Residual weight of the rejected position: max(0, p_j - q_j), or with
// greedy drafts (q == nullptr) p_j with the draft id xi removed.
struct ResidualWeight {
  const float* z;
  const float* q;
  float M, l2t, inv_S;                  // l2t = log2(e) / tau
  int xi;
  __device__ float operator()(int j) const {
    const float p = exp_tau(z[j] - M, l2t) * inv_S;
    if (q) return fmaxf(0.f, p - q[j]);
    return j == xi ? 0.f : p;
  }
};
struct ArrayWeight {
  const float* w;
  __device__ float operator()(int s) const { return w[s]; }
};

// row maximum from the chunk statistics
__device__ __forceinline__ float stats_max(const float2* cst, int nchunk, int lane) {
  float M = -INFINITY;
  int c = lane;
  for (; c + 96 < nchunk; c += 128)
    M = fmaxf(fmaxf(M, fmaxf(cst[c].x, cst[c + 32].x)), fmaxf(cst[c + 64].x, cst[c + 96].x));
  for (; c < nchunk; c += 32) M = fmaxf(M, cst[c].x);
  return warp_max(M);
}

// ---------------------------------------------------------------------------
// sampling: one warp per row
// ---------------------------------------------------------------------------
template <class ZRows>
__global__ void __launch_bounds__(kWarps * 32)
sample_seg_kernel(const ZRows zr, int rows, int n,
                  const float2* __restrict__ stats, int nseg,
                  const float2* __restrict__ cstats, const int32_t* __restrict__ ids,
                  float inv_tau, uint64_t seed, uint64_t offset,
                  int32_t* __restrict__ tokens) {
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  const int lane = threadIdx.x & 31;
  const int r = blockIdx.x * kWarps + (threadIdx.x >> 5);
  if (r >= rows) return;
  const int nchunk = (nseg + kSeg - 1) / kSeg;
  const float2* cst = cstats + (int64_t)r * nchunk;
  const float M = stats_max(cst, nchunk, lane);
  const StatsWeight cw{cst, M, inv_tau};
  const StatsWeight sw{stats + (int64_t)r * nseg, M, inv_tau};
  const ExpWeightOf<decltype(zr.row(0))> ew{zr.row(r), M, inv_tau};
  const float u = philox_uniform(seed, (uint32_t)r, 0u, offset);
  int j;
  warp_draw(nchunk, nseg, n, cw, sw, ew, u, lane, j);
  if (lane == 0) tokens[r] = ids ? ids[j] : j;
}

// Sampling with the chunk statistics made in the same block (one block per
// row, 4..32 warps as the chunk count asks): the warps reduce the row's
// segment statistics to chunk statistics in shared memory -- the same
// reductions, and so the same values, as the chunk-statistics kernel --
// then warp 0 draws.  Saves that kernel's launch on the step's critical
// path.
constexpr int kMaxFusedChunks = 4096;   // shared memory: 8 bytes per chunk
constexpr int kFusedU = 4;              // chunks in flight per warp
template <class ZRows>
__global__ void __launch_bounds__(1024)
sample_rows_kernel(const ZRows zr, int n, const float2* __restrict__ stats,
                   int nseg, const int32_t* __restrict__ ids, float inv_tau, uint64_t seed,
                   uint64_t offset, int32_t* __restrict__ tokens) {
  extern __shared__ float2 s_cst[];
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  const int r = blockIdx.x;
  const int nchunk = (nseg + kSeg - 1) / kSeg;
  const float2* srow = stats + (int64_t)r * nseg;
  constexpr int kU = kFusedU;
  for (int cb = warp; cb < nchunk; cb += nw * kU) {
    float2 st[kU];
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int c = cb + u * nw, sg = c * kSeg + lane;
      st[u] = (c < nchunk && sg < nseg) ? srow[sg] : make_float2(-INFINITY, 0.f);
    }
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int c = cb + u * nw;
      if (c < nchunk) {
        const float Mc = warp_max(st[u].x);
        const float Sc = warp_sum(seg_weight(st[u], Mc, inv_tau));
        if (lane == 0) s_cst[c] = make_float2(Mc, Sc);
      }
    }
  }
  __syncthreads();
  if constexpr (ZRows::kRecompute) {
    // warp 0 finds the segment; all warps recompute its 32 logits (a warp
    // per id, lanes across the hidden dimension); warp 0 draws the id
    __shared__ int s_seg;
    __shared__ float s_par[3];
    __shared__ float s_z[kSeg];
    if (warp == 0) {
      const float M = stats_max(s_cst, nchunk, lane);
      const StatsWeight cw{s_cst, M, inv_tau};
      const StatsWeight sw{srow, M, inv_tau};
      const float u = philox_uniform(seed, (uint32_t)r, 0u, offset);
      int seg;
      float target, before;
      warp_draw_segment(nchunk, nseg, cw, sw, u, lane, seg, target, before);
      if (lane == 0) {
        s_seg = seg;
        s_par[0] = M; s_par[1] = target; s_par[2] = before;
      }
    }
    __syncthreads();
    const int seg = s_seg;
    const auto zrow = zr.row(r);
    for (int i = warp; i < kSeg; i += nw) {
      const int j = seg * kSeg + i;
      const float z = j < n ? zrow.coop(j, lane) : -INFINITY;
      if (lane == 0) s_z[i] = z;
    }
    __syncthreads();
    if (warp != 0) return;
    const float M = s_par[0];
    float before = s_par[2];
    const int j = seg * kSeg + lane;
    const float wj = j < n ? expf((s_z[lane] - M) * inv_tau) : 0.f;
    const int lj = scan_pick(wj, s_par[1], before, lane);
    const int jj = min(seg * kSeg + lj, n - 1);
    if (lane == 0) tokens[r] = ids ? ids[jj] : jj;
  } else {
    if (warp != 0) return;
    const float M = stats_max(s_cst, nchunk, lane);
    const StatsWeight cw{s_cst, M, inv_tau};
    const StatsWeight sw{srow, M, inv_tau};
    const ExpWeightOf<decltype(zr.row(0))> ew{zr.row(r), M, inv_tau};
    const float u = philox_uniform(seed, (uint32_t)r, 0u, offset);
    int j;
    warp_draw(nchunk, nseg, n, cw, sw, ew, u, lane, j);
    if (lane == 0) tokens[r] = ids ? ids[j] : j;
  }
}

// ---------------------------------------------------------------------------
// Gumbel-max sampling (the alternative single-pass sampler): the first index
// of the largest z_j / tau - log(-log u_j) is a draw from softmax(z / tau).
// Index j of row r takes word j mod 4 of the Philox output for counter
// (r, 2^31 + j / 4, offset lo, offset hi), u = ((x >> 9) + 1/2) * 2^-23,
// strictly inside (0, 1).  A block per row; no softmax statistics needed.
// ---------------------------------------------------------------------------
constexpr uint32_t kGumbelTag = 0x80000000u;
constexpr int kGumbelThreads = 256;
__global__ void __launch_bounds__(kGumbelThreads)
gumbel_rows_kernel(const float* __restrict__ Z, int n, const int32_t* __restrict__ ids,
                   float inv_tau, uint64_t seed, uint64_t offset,
                   int32_t* __restrict__ tokens) {
  __shared__ float s_key[kGumbelThreads / 32];
  __shared__ int s_idx[kGumbelThreads / 32];
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  const int r = blockIdx.x, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const float* z = Z + (int64_t)r * n;
  const uint2 key = make_uint2((uint32_t)seed, (uint32_t)(seed >> 32));
  float best = -INFINITY;
  int bj = INT_MAX;
  const int groups = (n + 3) >> 2;
  for (int q = threadIdx.x; q < groups; q += blockDim.x) {
    const uint4 x = philox4x32_10(
        make_uint4((uint32_t)r, kGumbelTag | (uint32_t)q, (uint32_t)offset,
                   (uint32_t)(offset >> 32)), key);
    const uint32_t w[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      const int j = 4 * q + t;
      if (j < n) {
        const float u = ((float)(w[t] >> 9) + 0.5f) * 1.1920928955078125e-07f;  // 2^-23
        const float k = z[j] * inv_tau - logf(-logf(u));
        if (k > best) { best = k; bj = j; }    // a thread's j ascend: ties keep the first
      }
    }
  }
  // the largest key, the lowest index among equal keys
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    const float ob = __shfl_xor_sync(0xFFFFFFFFu, best, o);
    const int oj = __shfl_xor_sync(0xFFFFFFFFu, bj, o);
    if (ob > best || (ob == best && oj < bj)) { best = ob; bj = oj; }
  }
  if (lane == 0) { s_key[warp] = best; s_idx[warp] = bj; }
  __syncthreads();
  if (warp == 0) {
    const int nw = blockDim.x >> 5;
    best = lane < nw ? s_key[lane] : -INFINITY;
    bj = lane < nw ? s_idx[lane] : INT_MAX;
#pragma unroll
    for (int o = 16; o; o >>= 1) {
      const float ob = __shfl_xor_sync(0xFFFFFFFFu, best, o);
      const int oj = __shfl_xor_sync(0xFFFFFFFFu, bj, o);
      if (ob > best || (ob == best && oj < bj)) { best = ob; bj = oj; }
    }
    if (lane == 0) {
      const int j = bj < n ? bj : 0;
      tokens[r] = ids ? ids[j] : j;
    }
  }
}

// ---------------------------------------------------------------------------
// greedy decoding (temperature 0): the first id of the row maximum
// ---------------------------------------------------------------------------
__device__ __forceinline__ int warp_min_int(int v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v = min(v, __shfl_xor_sync(0xFFFFFFFFu, v, o));
  return v;
}

// The lowest segment holding the row maximum (from its statistics), then the
// lowest id in it whose z equals the segment's largest z (the maximum
// itself where z is stored); all lanes return it.
template <class ZR>
__device__ __forceinline__ int warp_argmax(const ZR& z, int n, const float2* st, int nseg,
                                           int lane) {
  float M = -INFINITY;
  int sb = nseg;
  for (int s = lane; s < nseg; s += 32) {
    const float m = st[s].x;
    if (m > M) { M = m; sb = s; }
  }
  const float Mw = warp_max(M);
  if (!(Mw > -INFINITY)) return 0;
  const int seg = warp_min_int(M == Mw ? sb : nseg);
  const int j = seg * kSeg + lane;
  const float zj = j < n ? z(j) : -INFINITY;
  const float mz = warp_max(zj);
  const unsigned hit = __ballot_sync(0xFFFFFFFFu, j < n && zj == mz);
  return hit ? seg * kSeg + __ffs(hit) - 1 : min(seg * kSeg, n - 1);
}

// One warp per row: vocabulary ids into tokens and/or compact indices.
template <class ZRows>
__global__ void __launch_bounds__(kWarps * 32)
greedy_kernel(const ZRows zr, int rows, int n, const float2* __restrict__ stats,
              int nseg, const int32_t* __restrict__ ids, int32_t* __restrict__ tokens,
              int32_t* __restrict__ compact) {
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  const int lane = threadIdx.x & 31;
  const int r = blockIdx.x * kWarps + (threadIdx.x >> 5);
  if (r >= rows) return;
  const int j = warp_argmax(zr.row(r), n, stats + (int64_t)r * nseg, nseg, lane);
  if (lane == 0) {
    if (tokens) tokens[r] = ids ? ids[j] : j;
    if (compact) compact[r] = j;
  }
}

// ---------------------------------------------------------------------------
// verification
// ---------------------------------------------------------------------------
__device__ int find_compact(const int32_t* ids, int n, int V, int x) {
  if (!ids) return (x >= 0 && x < n && x < V) ? x : -1;
  int lo = 0, hi = n;                   // first position with ids[pos] >= x
  while (lo < hi) {
    const int mid = (lo + hi) >> 1;
    if (ids[mid] < x) lo = mid + 1; else hi = mid;
  }
  return (lo < n && ids[lo] == x) ? lo : -1;
}

// First rejected draft of session s (k if all were accepted).
__device__ __forceinline__ int first_rejection(const int32_t* acc, int s, int k, int lane) {
  for (int i0 = 0; i0 < k; i0 += 32) {
    const int i = i0 + lane;
    const unsigned rej = __ballot_sync(0xFFFFFFFFu, i < k && !acc[(int64_t)s * k + i]);
    if (rej) return i0 + __ffs(rej) - 1;
  }
  return k;
}

// One warp per target row: the row's softmax maximum and normaliser and,
// for a draft position, the acceptance test r_i * q_i(x_i) < p_i(x_i).
__global__ void __launch_bounds__(kWarps * 32)
verify_rows_kernel(const float* __restrict__ Z, const float2* __restrict__ cstats,
                   int nchunk, int n, int sessions, int k, const int32_t* __restrict__ ids,
                   int V, float inv_tau, const int32_t* __restrict__ draft,
                   const float* __restrict__ q, uint64_t seed, uint64_t offset,
                   float2* __restrict__ rowMS, int32_t* __restrict__ acc,
                   int32_t* __restrict__ xis) {
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  const int lane = threadIdx.x & 31;
  const int64_t r = (int64_t)blockIdx.x * kWarps + (threadIdx.x >> 5);
  if (r >= (int64_t)sessions * (k + 1)) return;
  const int s = (int)(r / (k + 1)), i = (int)(r - (int64_t)s * (k + 1));
  const float2* cst = cstats + r * nchunk;
  const float M = stats_max(cst, nchunk, lane);
  float S = 0.f;
  for (int t = lane; t < nchunk; t += 32) S += seg_weight(cst[t], M, inv_tau);
  S = warp_sum(S);
  if (lane == 0) {
    rowMS[r] = make_float2(M, S);
    if (i < k) {
      const int64_t di = (int64_t)s * k + i;
      const int xi = find_compact(ids, n, V, draft[di]);
      const float px = xi >= 0 ? expf((Z[r * n + xi] - M) * inv_tau) / S : 0.f;
      const float qx = xi >= 0 ? (q ? q[di * n + xi] : 1.f) : 0.f;
      const float rr = philox_uniform(seed, (uint32_t)s, (uint32_t)(1 + i), offset);
      acc[di] = rr * qx < px ? 1 : 0;
      xis[di] = xi;
    }
  }
}

// Segment and chunk weights of the residual distribution at each session's
// first rejection: a warp per (session, chunk).
__global__ void __launch_bounds__(kWarps * 32)
verify_residual_kernel(const float* __restrict__ Z, int n, int nseg, int nchunk,
                       int sessions, int k, const float* __restrict__ q, float inv_tau,
                       const float2* __restrict__ rowMS, const int32_t* __restrict__ acc,
                       const int32_t* __restrict__ xis, float* __restrict__ resw,
                       float* __restrict__ resc) {
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  const int lane = threadIdx.x & 31;
  const int kr = (lane >> 1) & 15;
  const long long total = (long long)nchunk * sessions;
  const long long nwarps = (long long)gridDim.x * kWarps;
  for (long long g = (long long)blockIdx.x * kWarps + (threadIdx.x >> 5); g < total;
       g += nwarps) {
    const int s = (int)(g / nchunk);
    const int c = (int)(g - (long long)s * nchunk);
    const int i = first_rejection(acc, s, k, lane);
    if (i == k) continue;               // the bonus draw uses the statistics
    const int64_t r = (int64_t)s * (k + 1) + i;
    const int64_t di = (int64_t)s * k + i;
    const float2 ms = rowMS[r];
    const ResidualWeight rw{Z + r * n, q ? q + di * n : nullptr, ms.x, inv_tau * kLog2e,
                            1.f / ms.y, xis[di]};
    float csum = 0.f;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      float v[kGroup];
#pragma unroll
      for (int t = 0; t < kGroup; ++t) {
        const int sg = c * kSeg + h * kGroup + t;
        const int j = sg * kSeg + lane;
        v[t] = (sg < nseg && j < n) ? rw(j) : 0.f;
      }
      const float w = warp_reduce_scatter16(v, SumOp{}, lane);
      const int sg = c * kSeg + h * kGroup + kr;
      if (!(lane & 1) && sg < nseg) resw[(int64_t)s * nseg + sg] = w;
      if (!(lane & 1)) csum += w;
    }
    csum = warp_sum(csum);
    if (lane == 0) resc[(int64_t)s * nchunk + c] = csum;
  }
}

// Greedy verification, one thread per session: accept while the draft is
// the target's argmax; the next token is the argmax at the first mismatch,
// or at the bonus position.
__global__ void greedy_verify_kernel(const int32_t* __restrict__ amax, int sessions, int k,
                                     int n, const int32_t* __restrict__ ids, int V,
                                     const int32_t* __restrict__ draft,
                                     int32_t* __restrict__ n_acc,
                                     int32_t* __restrict__ next_token) {
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  const int s = blockIdx.x * blockDim.x + threadIdx.x;
  if (s >= sessions) return;
  const int32_t* a = amax + (int64_t)s * (k + 1);
  int i = 0;
  while (i < k && find_compact(ids, n, V, draft[(int64_t)s * k + i]) == a[i]) ++i;
  n_acc[s] = i;
  next_token[s] = ids ? ids[a[i]] : a[i];
}

// One warp per session: the draw, from the residual (or, if that is all
// zero, from p_i) at the first rejection, else the bonus draw from p_k.
__global__ void __launch_bounds__(kWarps * 32)
verify_draw_kernel(const float* __restrict__ Z, int n, const float2* __restrict__ stats,
                   const float2* __restrict__ cstats, int nseg, int nchunk, int sessions,
                   int k, const int32_t* __restrict__ ids, const float* __restrict__ q,
                   float inv_tau, uint64_t seed, uint64_t offset,
                   const float2* __restrict__ rowMS, const int32_t* __restrict__ acc,
                   const int32_t* __restrict__ xis, const float* __restrict__ resw,
                   const float* __restrict__ resc, int32_t* __restrict__ n_acc,
                   int32_t* __restrict__ next_token) {
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  const int lane = threadIdx.x & 31;
  const int s = blockIdx.x * kWarps + (threadIdx.x >> 5);
  if (s >= sessions) return;
  const int i = first_rejection(acc, s, k, lane);
  const int64_t r = (int64_t)s * (k + 1) + i;
  const float2 ms = rowMS[r];
  const float u = philox_uniform(seed, (uint32_t)s, (uint32_t)(1 + k), offset);
  int j = 0;
  float tot = 0.f;
  if (i < k) {
    const int64_t di = (int64_t)s * k + i;
    const ArrayWeight cw{resc + (int64_t)s * nchunk};
    const ArrayWeight sw{resw + (int64_t)s * nseg};
    const ResidualWeight rw{Z + r * n, q ? q + di * n : nullptr, ms.x, inv_tau * kLog2e,
                            1.f / ms.y, xis[di]};
    tot = warp_draw(nchunk, nseg, n, cw, sw, rw, u, lane, j);
  }
  if (!(tot > 0.f)) {
    const StatsWeight cw{cstats + r * nchunk, ms.x, inv_tau};
    const StatsWeight sw{stats + r * nseg, ms.x, inv_tau};
    const ExpWeight ew{ZRowStored{Z + r * n}, ms.x, inv_tau};
    warp_draw(nchunk, nseg, n, cw, sw, ew, u, lane, j);
  }
  if (lane == 0) {
    n_acc[s] = i;
    next_token[s] = ids ? ids[j] : j;
  }
}

int stats_grid(long long warps_of_work, int sm_count) {
  long long b = (warps_of_work + kWarps - 1) / kWarps;
  const long long cap = (long long)(sm_count > 0 ? sm_count : 148) * 8;
  if (b > cap) b = cap;
  return (int)(b < 1 ? 1 : b);
}

size_t align256(size_t x) { return (x + 255) / 256 * 256; }

}  // namespace

int sample_max_n() { return kMaxN; }
int verify_max_k() { return kMaxK; }
int seg_count(int n) { return (n + kSeg - 1) / kSeg; }
int chunk_count(int nseg) { return (nseg + kSeg - 1) / kSeg; }

cudaError_t launch_seg_stats(const float* Z, int rows, int n, float inv_tau,
                             float2* stats, float2* cstats, int sm_count,
                             cudaStream_t st) {
  const int nseg = seg_count(n), nchunk = chunk_count(nseg);
  return launch_pdl(seg_stats_kernel,
                    dim3(stats_grid((long long)rows * nchunk, sm_count)),
                    dim3(kWarps * 32), 0, st, Z, rows, n, nseg, nchunk, inv_tau, stats,
                    cstats);
}

cudaError_t launch_chunk_stats(const float2* stats, int rows, int nseg, float inv_tau,
                               float2* cstats, int sm_count, cudaStream_t st) {
  const int nchunk = chunk_count(nseg);
  return launch_pdl(chunk_stats_kernel,
                    dim3(stats_grid((long long)rows * nchunk, sm_count)),
                    dim3(kWarps * 32), 0, st, stats, rows, nseg, nchunk, inv_tau, cstats);
}

namespace {
template <class ZRows>
cudaError_t sample_segments_with(const ZRows& zr, int rows, int n, const float2* stats,
                                 int nseg, const float2* cstats, const int32_t* ids,
                                 float inv_tau, uint64_t seed, uint64_t offset,
                                 int32_t* tokens, cudaStream_t st, int greedy) {
  if (greedy)
    return launch_pdl(greedy_kernel<ZRows>, dim3((rows + kWarps - 1) / kWarps),
                      dim3(kWarps * 32), 0, st, zr, rows, n, stats, nseg, ids, tokens,
                      (int32_t*)nullptr);
  return launch_pdl(sample_seg_kernel<ZRows>, dim3((rows + kWarps - 1) / kWarps),
                    dim3(kWarps * 32), 0, st, zr, rows, n, stats, nseg, cstats, ids, inv_tau,
                    seed, offset, tokens);
}
template <class ZRows>
cudaError_t sample_rows_with(const ZRows& zr, int rows, int n, const float2* stats, int nseg,
                             const int32_t* ids, float inv_tau, uint64_t seed, uint64_t offset,
                             int32_t* tokens, cudaStream_t st) {
  const int nchunk = chunk_count(nseg);
  if (rows < 1 || nchunk > kMaxFusedChunks) return cudaErrorNotSupported;
  int warps = (nchunk + kFusedU - 1) / kFusedU;
  // (z recomputed: at most 8 warps, so that more rows run at once -- the
  // draw is a chain of dependent loads per row; measured on 1024 rows x
  // 256000 ids: 54 us with 8, 61 with 16, 71 with 32)
  const int cap = ZRows::kRecompute ? 8 : 32;
  warps = warps < 4 ? 4 : (warps > cap ? cap : warps);
  return launch_pdl(sample_rows_kernel<ZRows>, dim3(rows), dim3(warps * 32),
                    (size_t)nchunk * sizeof(float2), st, zr, n, stats, nseg, ids, inv_tau, seed,
                    offset, tokens);
}
}  // namespace

cudaError_t launch_sample_segments(const ZSource& zs, int rows, int n, const float2* stats,
                                   int nseg, const float2* cstats, const int32_t* ids,
                                   float inv_tau, uint64_t seed, uint64_t offset,
                                   int32_t* tokens, cudaStream_t st, int greedy) {
  if (zs.Z)
    return sample_segments_with(ZRowsStored{zs.Z, n}, rows, n, stats, nseg, cstats, ids,
                                inv_tau, seed, offset, tokens, st, greedy);
  if (!zs.h || !zs.W || zs.K < 1 || (zs.codes && !zs.row_scale)) return cudaErrorInvalidValue;
  return sample_segments_with(ZRowsRecomputed{zs, n}, rows, n, stats, nseg, cstats, ids,
                              inv_tau, seed, offset, tokens, st, greedy);
}

cudaError_t launch_gumbel(const float* Z, int rows, int n, const int32_t* ids, float inv_tau,
                          uint64_t seed, uint64_t offset, int32_t* tokens, cudaStream_t st) {
  if (rows < 1) return cudaErrorInvalidValue;
  return launch_pdl(gumbel_rows_kernel, dim3(rows), dim3(kGumbelThreads), 0, st, Z, n, ids,
                    inv_tau, seed, offset, tokens);
}

cudaError_t launch_sample_rows(const ZSource& zs, int rows, int n, const float2* stats,
                               int nseg, const int32_t* ids, float inv_tau, uint64_t seed,
                               uint64_t offset, int32_t* tokens, cudaStream_t st) {
  if (zs.Z)
    return sample_rows_with(ZRowsStored{zs.Z, n}, rows, n, stats, nseg, ids, inv_tau, seed,
                            offset, tokens, st);
  if (!zs.h || !zs.W || zs.K < 1 || (zs.codes && !zs.row_scale)) return cudaErrorInvalidValue;
  return sample_rows_with(ZRowsRecomputed{zs, n}, rows, n, stats, nseg, ids, inv_tau, seed,
                          offset, tokens, st);
}

// Scratch: stats [R][nseg] float2 | chunk stats [R][nchunk] float2 | rowMS
// [R] float2 | acc, xis [S*k] int32 | residual segment weights [S][nseg] |
// residual chunk weights [S][nchunk], with R = S * (k + 1).
size_t verify_scratch_bytes(int sessions, int k, int n) {
  const size_t R = (size_t)sessions * (k + 1), nseg = (size_t)seg_count(n),
               nchunk = (size_t)chunk_count((int)nseg);
  return align256(R * nseg * 8) + align256(R * nchunk * 8) + align256(R * 8) +
         2 * align256((size_t)sessions * k * 4) + align256((size_t)sessions * nseg * 4) +
         align256((size_t)sessions * nchunk * 4);
}

cudaError_t launch_verify(const float* Z, int sessions, int k, int n, const int32_t* ids,
                          int V, float inv_tau, const int32_t* draft, const float* q,
                          uint64_t seed, uint64_t offset, int32_t* n_acc,
                          int32_t* next_token, void* scratch, int sm_count,
                          cudaStream_t st, int greedy) {
  const int R = sessions * (k + 1), nseg = seg_count(n), nchunk = chunk_count(nseg);
  char* p = static_cast<char*>(scratch);
  float2* stats = reinterpret_cast<float2*>(p);
  p += align256((size_t)R * nseg * 8);
  float2* cstats = reinterpret_cast<float2*>(p);
  p += align256((size_t)R * nchunk * 8);
  float2* rowMS = reinterpret_cast<float2*>(p);
  p += align256((size_t)R * 8);
  int32_t* acc = reinterpret_cast<int32_t*>(p);
  p += align256((size_t)sessions * k * 4);
  int32_t* xis = reinterpret_cast<int32_t*>(p);
  p += align256((size_t)sessions * k * 4);
  float* resw = reinterpret_cast<float*>(p);
  p += align256((size_t)sessions * nseg * 4);
  float* resc = reinterpret_cast<float*>(p);
  cudaError_t e = launch_seg_stats(Z, R, n, inv_tau, stats, cstats, sm_count, st);
  if (greedy) {
    // the row maxima only: argmax per target row (into the normaliser
    // area), then one thread per session
    int32_t* amax = reinterpret_cast<int32_t*>(rowMS);
    if (e == cudaSuccess)
      e = launch_pdl(greedy_kernel<ZRowsStored>, dim3((R + kWarps - 1) / kWarps),
                     dim3(kWarps * 32), 0, st, ZRowsStored{Z, n}, R, n, (const float2*)stats,
                     nseg, ids, (int32_t*)nullptr, amax);
    if (e == cudaSuccess)
      e = launch_pdl(greedy_verify_kernel, dim3((sessions + 127) / 128), dim3(128), 0, st,
                     (const int32_t*)amax, sessions, k, n, ids, V, draft, n_acc, next_token);
    return e;
  }
  if (e == cudaSuccess)
    e = launch_pdl(verify_rows_kernel, dim3((R + kWarps - 1) / kWarps), dim3(kWarps * 32), 0,
                   st, Z, (const float2*)cstats, nchunk, n, sessions, k, ids, V, inv_tau,
                   draft, q, seed, offset, rowMS, acc, xis);
  if (e == cudaSuccess)
    e = launch_pdl(verify_residual_kernel,
                   dim3(stats_grid((long long)sessions * nchunk, sm_count)),
                   dim3(kWarps * 32), 0, st, Z, n, nseg, nchunk, sessions, k, q, inv_tau,
                   (const float2*)rowMS, (const int32_t*)acc, (const int32_t*)xis, resw,
                   resc);
  if (e == cudaSuccess)
    e = launch_pdl(verify_draw_kernel, dim3((sessions + kWarps - 1) / kWarps),
                   dim3(kWarps * 32), 0, st, Z, n, (const float2*)stats,
                   (const float2*)cstats, nseg, nchunk, sessions, k, ids, q, inv_tau, seed,
                   offset, (const float2*)rowMS, (const int32_t*)acc, (const int32_t*)xis,
                   (const float*)resw, (const float*)resc, n_acc, next_token);
  return e;
}

}  // namespace sph
