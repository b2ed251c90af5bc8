// Tensor-core gathered contraction for the many-row regime (Eq. 11 / Eq. 12
// over the kept vocabulary ids), tcgen05 + TMEM + TMA on sm_103a.
//
// Swap-AB: the MMA's M dimension is a tile of 128 gathered vocabulary rows
// (operand A, fetched from W by TMA tile::gather4, four rows per
// instruction), its N dimension is a block of BN hidden-state rows (operand
// B), and K runs over the hidden dimension in 64-element (128-byte) blocks,
// 128-byte swizzled.  fp32 hidden states are split on the fly into bf16
// hi + lo parts (h = hi + lo + O(2^-18 |h|)); both parts multiply the same
// W tile into one fp32 TMEM accumulator, so W is read once and the result
// keeps fp32 accuracy.  In bf16-activation mode only the hi part is used.
//
// Work is split stream-K style: the (row block, vocabulary tile, k-block)
// iterations are cut into one contiguous range per CTA (one persistent CTA
// per SM).  A tile whose k-range spans several CTAs is finished by the last
// CTA to arrive: every contributor stores its fp32 partial tile, counts in,
// and the last one adds the partials in a fixed order (deterministic) and
// runs the epilogue.  Nothing waits on another CTA.
//
// Warp roles (192 threads): warp 0 issues TMA, warp 1 owns TMEM and issues
// tcgen05.mma (one thread), warps 2-5 drain the double-buffered accumulator
// (tcgen05.ld) and run the fused epilogue.  Every wait is bounded; a wait
// that gives up sets the context's error word and the CTA winds down.
#include <cuda.h>
#include <cuda_runtime.h>

#include <mutex>

#include "sm100_ptx.cuh"
#include "sph_common.cuh"
#include "sph_internal.h"

namespace sph {
namespace {

constexpr int kThreads = 192;
constexpr int kTileM = 128;          // vocabulary rows per tile (MMA M)
constexpr int kBlockK = 64;          // bf16 elements per 128-byte row slice
constexpr int kATileBytes = kTileM * kBlockK * 2;
constexpr int kMaxBN = 256;
constexpr size_t kSmemBudget = 220 * 1024;
constexpr long long kDrainLimit = 1ll << 31;   // cycles, for in-flight copies

struct TcParams {
  int R, n, K, KB, NT, RB, BN, Rp, stages;
  long long T;                 // total iterations RB * NT * KB
  const int32_t* ids;          // gather path: sorted ids
  int epilogue;
  const float* bias;
  float clip;
  float* partial_out;
  float* Y;
  unsigned* rowmax;
  const int8_t* codes;
  const float* row_scale;
  float* P;                    // split-tile partials [2 * grid][BN][128]
  int* counters;               // [tiles][4 quadrants], zero between calls
  unsigned* status;
  long long spin_limit;
};

__device__ __forceinline__ long long cta_of(long long i, long long T, int G) {
  return ((i + 1) * G + T - 1) / T - 1;    // owner of iteration i
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

template <int EPI>
__device__ __forceinline__ void finish_chunk(const TcParams& p, const float (&v)[16],
                                             int row0, int j, bool vj, int id,
                                             int lane) {
#pragma unroll
  for (int q = 0; q < 16; ++q) {
    const int r = row0 + q;
    const bool ok = vj && r < p.R;
    if constexpr (EPI == EPI_CLOUD) {
      float m = 0.f;
      if (ok) {
        float y = v[q];
        if (p.bias) y += p.bias[id];
        const int64_t o = (int64_t)r * p.n + j;
        if (p.partial_out) p.partial_out[o] = y;
        const float yc = fminf(fmaxf(y, -p.clip), p.clip);
        p.Y[o] = yc;
        m = fabsf(yc);
      }
      m = warp_max(m);
      if (lane == 0 && r < p.R && m > 0.f) atomicMax(&p.rowmax[r], __float_as_uint(m));
    } else {
      if (ok) {
        const int64_t o = (int64_t)r * p.n + j;
        p.Y[o] = v[q] + (float)p.codes[o] * p.row_scale[r];
      }
    }
  }
}

template <int HILO, bool GATHER, int EPI>
__global__ void __launch_bounds__(kThreads, 1)
tc_kernel(const __grid_constant__ CUtensorMap tmW,
          const __grid_constant__ CUtensorMap tmH, const TcParams p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_addr = ptx::smem_u32(smem_raw);
  uint8_t* base = smem_raw + (((raw_addr + 1023) & ~1023u) - raw_addr);
  const int BN = p.BN;
  const int stage_bytes = kATileBytes + HILO * BN * 128;
  const int S = p.stages;
  uint64_t* full = reinterpret_cast<uint64_t*>(base + (size_t)S * stage_bytes);
  uint64_t* empty = full + S;
  uint64_t* tfull = empty + S;         // [2]
  uint64_t* tempty = tfull + 2;        // [2]
  uint64_t* drain = tempty + 2;        // [1]
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* s_abort = reinterpret_cast<volatile int*>(tmem_holder + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  uint32_t ncols = 32;
  while (ncols < (uint32_t)(2 * BN)) ncols <<= 1;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      ptx::mbar_init(&full[s], 1);
      ptx::mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      ptx::mbar_init(&tfull[a], 1);
      ptx::mbar_init(&tempty[a], 4);
    }
    ptx::mbar_init(drain, 1);
    *s_abort = 0;
    ptx::fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    ptx::prefetch_tmap(&tmW);
    ptx::prefetch_tmap(&tmH);
  }
  if (warp == 1) ptx::tmem_alloc(tmem_holder, ncols);
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;

  const int G = gridDim.x;
  const long long it0 = (long long)blockIdx.x * p.T / G;
  const long long it1 = (long long)(blockIdx.x + 1) * p.T / G;
  const long long limit = p.spin_limit;

  auto give_up = [&]() {
    atomicOr(p.status, ERR_TIMEOUT);
    *s_abort = 1;
  };

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    Segments sg{it0, it1, p.KB};
    int stage = 0;
    uint32_t phase = 0;
    int tile, kb0, kb1;
    const uint32_t tx = (uint32_t)stage_bytes;
    bool stop = false;
    long long issued = 0;
    while (!stop && sg.next(tile, kb0, kb1)) {
      const int rb = tile / p.NT, t = tile - rb * p.NT;
      const int j0 = t * kTileM;
      int y[4] = {0, 0, 0, 0};
      if constexpr (GATHER) {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int j = min(j0 + 4 * lane + q, p.n - 1);
          y[q] = p.ids[j];
        }
      }
      for (int kb = kb0; kb < kb1; ++kb) {
        int ok = 1;
        if (lane == 0) ok = !*s_abort && ptx::mbar_wait(&empty[stage], phase ^ 1, limit);
        ok = __shfl_sync(0xFFFFFFFFu, ok, 0);
        if (!ok) {
          if (lane == 0 && !*s_abort) give_up();
          stop = true;
          break;
        }
        if (lane == 0) ptx::mbar_expect_tx(&full[stage], tx);
        __syncwarp();
        uint8_t* A = base + (size_t)stage * stage_bytes;
        uint8_t* B = A + kATileBytes;
        if constexpr (GATHER) {
          ptx::tma_gather4(A + 512 * lane, &tmW, kb * kBlockK, y[0], y[1], y[2], y[3],
                           &full[stage]);
        } else {
          if (lane == 0) ptx::tma_load_2d(A, &tmW, kb * kBlockK, j0, &full[stage]);
        }
        if (lane == 0) {
          ptx::tma_load_2d(B, &tmH, kb * kBlockK, rb * BN, &full[stage]);
          if (HILO == 2)
            ptx::tma_load_2d(B + BN * 128, &tmH, kb * kBlockK, p.Rp + rb * BN, &full[stage]);
        }
        ++issued;
        if (++stage == S) { stage = 0; phase ^= 1; }
      }
    }
    if (stop && lane == 0) {
      // let the copies already issued land before the CTA winds down
      for (long long k = issued > S ? issued - S : 0; k < issued; ++k)
        ptx::mbar_wait(&full[k % S], (uint32_t)((k / S) & 1), kDrainLimit);
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------- MMA issuer
    if (lane == 0) {
      Segments sg{it0, it1, p.KB};
      int stage = 0;
      uint32_t phase = 0;
      uint32_t tph[2] = {0, 0};
      int si = 0, tile, kb0, kb1;
      const uint32_t idesc = ptx::idesc_bf16_f32(kTileM, BN);
      bool stop = false;
      while (!stop && sg.next(tile, kb0, kb1)) {
        const int acc = si & 1;
        if (*s_abort || !ptx::mbar_wait(&tempty[acc], tph[acc] ^ 1, limit)) {
          if (!*s_abort) give_up();
          break;
        }
        tph[acc] ^= 1;
        ptx::tc_fence_after();
        const uint32_t d = tmem_base + (uint32_t)(acc * BN);
        for (int kb = kb0; kb < kb1; ++kb) {
          if (*s_abort || !ptx::mbar_wait(&full[stage], phase, limit)) {
            if (!*s_abort) give_up();
            stop = true;
            break;
          }
          ptx::tc_fence_after();
          const uint32_t a = ptx::smem_u32(base + (size_t)stage * stage_bytes);
          const uint32_t b = a + kATileBytes;
#pragma unroll
          for (int h = 0; h < HILO; ++h) {
#pragma unroll
            for (int kk = 0; kk < kBlockK / 16; ++kk) {
              ptx::umma_bf16(d, ptx::sdesc_k128(a + kk * 32),
                             ptx::sdesc_k128(b + h * BN * 128 + kk * 32), idesc,
                             (kb != kb0 || h != 0 || kk != 0) ? 1u : 0u);
            }
          }
          ptx::umma_commit(&empty[stage]);
          if (++stage == S) { stage = 0; phase ^= 1; }
        }
        if (stop) break;
        ptx::umma_commit(&tfull[acc]);
        ++si;
      }
      // all issued MMAs complete before TMEM is released
      ptx::umma_commit(drain);
      ptx::mbar_wait(drain, 0, limit);
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int quad = warp & 3;
    const int i = quad * 32 + lane;              // vocabulary row in the tile
    Segments sg{it0, it1, p.KB};
    uint32_t fph[2] = {0, 0};
    int si = 0, tile, kb0, kb1;
    while (sg.next(tile, kb0, kb1)) {
      const int acc = si & 1;
      int ok = 1;
      if (lane == 0) ok = !*s_abort && ptx::mbar_wait(&tfull[acc], fph[acc], limit);
      ok = __shfl_sync(0xFFFFFFFFu, ok, 0);
      if (!ok) {
        if (lane == 0 && !*s_abort) give_up();
        break;
      }
      fph[acc] ^= 1;
      ptx::tc_fence_after();
      const int rb = tile / p.NT, t = tile - rb * p.NT;
      const int j = t * kTileM + i;
      const bool vj = j < p.n;
      const int id = vj ? (GATHER ? p.ids[j] : j) : 0;
      const bool whole = kb0 == 0 && kb1 == p.KB;
      const uint32_t taddr = tmem_base + ((uint32_t)(quad * 32) << 16) + (uint32_t)(acc * BN);
      // a CTA's split tiles can only be its first and its last segment:
      // slot 2c holds the first, 2c+1 the last
      float* Pt = p.P + (size_t)(2 * blockIdx.x + (si == 0 ? 0 : 1)) * BN * kTileM;
      for (int ch = 0; ch < BN / 16; ++ch) {
        float v[16];
        ptx::tmem_ld16(taddr + ch * 16, v);
        if (whole) {
          finish_chunk<EPI>(p, v, rb * BN + ch * 16, j, vj, id, lane);
        } else {
#pragma unroll
          for (int q = 0; q < 16; ++q) Pt[(size_t)(ch * 16 + q) * kTileM + i] = v[q];
        }
      }
      ptx::tc_fence_before();
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(&tempty[acc]);
      if (!whole) {
        // split tile: this warp's 32 vocabulary rows are finished by the
        // last warp (over all contributing CTAs) of the same quadrant
        __threadfence();
        int old = 0;
        if (lane == 0) old = atomicAdd(&p.counters[tile * 4 + quad], 1);
        old = __shfl_sync(0xFFFFFFFFu, old, 0);
        const long long c0 = cta_of((long long)tile * p.KB, p.T, gridDim.x);
        const long long c1 = cta_of((long long)tile * p.KB + p.KB - 1, p.T, gridDim.x);
        if (old == (int)(c1 - c0)) {
          __threadfence();
          for (int ch = 0; ch < BN / 16; ++ch) {
            float v[16];
#pragma unroll
            for (int q = 0; q < 16; ++q) v[q] = 0.f;
            // contributors in CTA order: a fixed summation order
            for (long long c = c0; c <= c1; ++c) {
              const long long start = c * p.T / gridDim.x;
              const int slot = 2 * (int)c + ((start / p.KB) == tile ? 0 : 1);
              const float* Ps = p.P + (size_t)slot * BN * kTileM + (size_t)ch * 16 * kTileM + i;
#pragma unroll
              for (int q = 0; q < 16; ++q) v[q] += __ldcg(Ps + (size_t)q * kTileM);
            }
            finish_chunk<EPI>(p, v, rb * BN + ch * 16, j, vj, id, lane);
          }
          if (lane == 0) p.counters[tile * 4 + quad] = 0;
        }
      }
      ++si;
    }
  }

  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  if (warp == 1) ptx::tmem_dealloc(tmem_base, ncols);
}

// ---------------------------------------------------------------------------
// operand preparation: fp32 h -> bf16 hi (and lo) planes, zero padded
// ---------------------------------------------------------------------------
__global__ void split_h_kernel(const float* __restrict__ h, int64_t ld_h, int R,
                               int K, int Rp, int Kp, int hilo,
                               __nv_bfloat16* __restrict__ Hs,
                               int* __restrict__ counters, int ncounters) {
  const int64_t total = (int64_t)Rp * Kp;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total;
       e += (int64_t)gridDim.x * blockDim.x) {
    const int r = (int)(e / Kp), c = (int)(e - (int64_t)r * Kp);
    const float x = (r < R && c < K) ? h[(int64_t)r * ld_h + c] : 0.f;
    const __nv_bfloat16 hi = __float2bfloat16_rn(x);
    Hs[e] = hi;
    if (hilo == 2) Hs[total + e] = __float2bfloat16_rn(x - __bfloat162float(hi));
  }
  for (int t = blockIdx.x * blockDim.x + threadIdx.x; t < ncounters;
       t += gridDim.x * blockDim.x)
    counters[t] = 0;
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

size_t align256(size_t x) { return (x + 255) / 256 * 256; }

}  // namespace

TcPlan tc_plan(int rows, int n, int K, int act_bf16, int sm_count) {
  TcPlan pl{};
  pl.hilo = act_bf16 ? 1 : 2;
  if (rows <= kMaxBN) {
    pl.RB = 1;
    pl.BN = (rows + 15) / 16 * 16;
  } else {
    pl.RB = (rows + kMaxBN - 1) / kMaxBN;
    pl.BN = ((rows + pl.RB - 1) / pl.RB + 15) / 16 * 16;
  }
  pl.Rp = pl.RB * pl.BN;
  pl.KB = (K + kBlockK - 1) / kBlockK;
  pl.Kp = pl.KB * kBlockK;
  pl.NT = (n + kTileM - 1) / kTileM;
  pl.T = (long long)pl.RB * pl.NT * pl.KB;
  pl.G = (int)(pl.T < sm_count ? pl.T : sm_count);
  const int stage_bytes = kATileBytes + pl.hilo * pl.BN * 128;
  pl.stages = (int)((kSmemBudget - 2048) / stage_bytes);
  if (pl.stages > 8) pl.stages = 8;
  const int tiles = pl.RB * pl.NT;
  pl.hs_bytes = align256((size_t)pl.hilo * pl.Rp * pl.Kp * 2);
  // split tiles exist only when a CTA's range does not cover whole tiles
  const bool splits = pl.T % pl.G != 0 || (pl.T / pl.G) % pl.KB != 0;
  pl.p_bytes = splits ? align256((size_t)2 * pl.G * pl.BN * kTileM * 4) : 0;
  pl.cnt_bytes = align256((size_t)tiles * 4 * sizeof(int));
  pl.scratch_bytes = pl.hs_bytes + pl.p_bytes + pl.cnt_bytes;
  pl.smem_bytes = 1024 + (size_t)pl.stages * stage_bytes + 256;
  pl.ok = pl.stages >= 2;
  return pl;
}

template <int HILO, bool GATHER, int EPI>
static cudaError_t launch_inst(const CUtensorMap& mw, const CUtensorMap& mh,
                               const TcParams& prm, const TcPlan& pl,
                               cudaStream_t st) {
  auto kern = tc_kernel<HILO, GATHER, EPI>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)pl.smem_bytes);
  if (e != cudaSuccess) return e;
  kern<<<pl.G, kThreads, pl.smem_bytes, st>>>(mw, mh, prm);
  ++launch_count;
  return cudaGetLastError();
}

cudaError_t launch_tc(const GatherGemm& g, const TcPlan& pl, void* scratch,
                      long long spin_limit, cudaStream_t st) {
  if (!pl.ok || g.w_dtype != W_BF16) return cudaErrorNotSupported;
  char* sc = static_cast<char*>(scratch);
  auto* Hs = reinterpret_cast<__nv_bfloat16*>(sc);
  float* P = pl.p_bytes ? reinterpret_cast<float*>(sc + pl.hs_bytes) : nullptr;
  int* counters = reinterpret_cast<int*>(sc + pl.hs_bytes + pl.p_bytes);
  const int tiles = pl.RB * pl.NT;

  {
    const int64_t total = (int64_t)pl.Rp * pl.Kp;
    int blocks = (int)((total + 255) / 256);
    if (blocks > 4096) blocks = 4096;
    if (blocks < 1) blocks = 1;
    split_h_kernel<<<blocks, 256, 0, st>>>(g.h, g.ld_h, g.rows, g.K, pl.Rp, pl.Kp,
                                           pl.hilo, Hs, counters, tiles * 4);
    ++launch_count;
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }

  alignas(64) CUtensorMap mw, mh;
  const bool gather = g.ids != nullptr;
  // W: [V rows, K columns], row stride ld_w; box 64 columns x (1 | 128) rows
  if (!make_map(&mw, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, g.W, (uint64_t)g.K, (uint64_t)g.V,
                (uint64_t)g.ld_w * 2, kBlockK, gather ? 1u : (uint32_t)kTileM))
    return cudaErrorInvalidValue;
  if (!make_map(&mh, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, Hs, (uint64_t)pl.Kp,
                (uint64_t)pl.hilo * pl.Rp, (uint64_t)pl.Kp * 2, kBlockK,
                (uint32_t)pl.BN))
    return cudaErrorInvalidValue;

  TcParams prm{};
  prm.R = g.rows; prm.n = g.n; prm.K = g.K; prm.KB = pl.KB; prm.NT = pl.NT;
  prm.RB = pl.RB; prm.BN = pl.BN; prm.Rp = pl.Rp; prm.stages = pl.stages;
  prm.T = pl.T; prm.ids = g.ids; prm.epilogue = g.epilogue; prm.bias = g.bias;
  prm.clip = g.clip; prm.partial_out = g.partial_out; prm.Y = g.Y;
  prm.rowmax = g.rowmax; prm.codes = g.codes; prm.row_scale = g.row_scale;
  prm.P = P; prm.counters = counters;
  prm.status = g.status; prm.spin_limit = spin_limit;

  const bool hilo2 = pl.hilo == 2;
  if (g.epilogue == EPI_CLOUD) {
    if (gather) return hilo2 ? launch_inst<2, true, EPI_CLOUD>(mw, mh, prm, pl, st)
                             : launch_inst<1, true, EPI_CLOUD>(mw, mh, prm, pl, st);
    return hilo2 ? launch_inst<2, false, EPI_CLOUD>(mw, mh, prm, pl, st)
                 : launch_inst<1, false, EPI_CLOUD>(mw, mh, prm, pl, st);
  }
  if (gather) return hilo2 ? launch_inst<2, true, EPI_ENDPOINT>(mw, mh, prm, pl, st)
                           : launch_inst<1, true, EPI_ENDPOINT>(mw, mh, prm, pl, st);
  return hilo2 ? launch_inst<2, false, EPI_ENDPOINT>(mw, mh, prm, pl, st)
               : launch_inst<1, false, EPI_ENDPOINT>(mw, mh, prm, pl, st);
}

}  // namespace sph
