// CUDA-core gathered GEMV for the few-row regime (Eq. 11 / Eq. 12 over the
// kept vocabulary ids).
//
// One warp owns VPW gathered vocabulary rows at a time and streams each
// W row once with 16-byte non-allocating loads; the RT hidden-state rows of
// the current row tile sit in shared memory as fp32.  Accumulation is fp32
// FMA over exact bf16 / e4m3 weight values.  The epilogue is fused:
//   cloud    : + bias, optional unclipped store, clip, store, row |max|
//   endpoint : + code * row_scale  (dequantized cloud partial, Eq. 13)
// HBM traffic is the kept W rows once per row tile; rows > RT are handled by
// further row tiles (re-reading W), which is why the dispatcher routes more
// than a couple of rows to the tensor-core kernel.
#include <atomic>
#include <mutex>

#include "sm100_ptx.cuh"
#include "sph_common.cuh"
#include "sph_internal.h"

namespace sph {
namespace {

constexpr int kWarps = 8;
constexpr int kThreads = kWarps * 32;
constexpr size_t kSmemLimit = 200 * 1024;     // h tile budget (bytes)

__device__ __forceinline__ uint4 ld_stream_v4(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

// Expand one 16-byte weight vector into floats (8 bf16 or 16 e4m3).
template <int WDT>
__device__ __forceinline__ void expand(const uint4& v, float* w) {
  const uint32_t u[4] = {v.x, v.y, v.z, v.w};
  if constexpr (WDT == W_BF16) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      w[2 * i] = bf16_lo(u[i]);
      w[2 * i + 1] = bf16_hi(u[i]);
    }
  } else {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 a = e4m3x2_to_float2((uint16_t)(u[i] & 0xFFFFu));
      const float2 b = e4m3x2_to_float2((uint16_t)(u[i] >> 16));
      w[4 * i] = a.x;
      w[4 * i + 1] = a.y;
      w[4 * i + 2] = b.x;
      w[4 * i + 3] = b.y;
    }
  }
}

template <int WDT>
__device__ __forceinline__ float load_scalar_w(const void* W, int64_t off) {
  if constexpr (WDT == W_BF16) {
    const uint16_t b = reinterpret_cast<const uint16_t*>(W)[off];
    return __uint_as_float((uint32_t)b << 16);
  } else {
    const uint8_t b = reinterpret_cast<const uint8_t*>(W)[off];
    const uint16_t two = b;
    return e4m3x2_to_float2(two).x;
  }
}

// vocabulary rows a warp streams at once (more bytes in flight for few rows)
template <int RT>
constexpr int vpw() { return RT <= 2 ? 4 : 2; }

template <int RT, int WDT, int EPI>
__global__ void __launch_bounds__(kThreads)
gemv_kernel(const GatherGemm g, const int row0) {
  constexpr int kVPW = vpw<RT>();
  extern __shared__ float hs[];               // [RT][KP] fp32
  __shared__ unsigned smax[RT];
  const int K = g.K;
  const int KP = (K + 7) & ~7;                 // 32-byte aligned row stride
  const int rt = min(RT, g.rows - row0);
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  for (int i = threadIdx.x; i < RT * KP; i += kThreads) {
    const int r = i / KP, c = i - r * KP;
    float v = 0.f;
    if (r < rt && c < K) {
      v = g.h[(int64_t)(row0 + r) * g.ld_h + c];
      if (g.act_bf16) v = __bfloat162float(__float2bfloat16_rn(v));
    }
    hs[i] = v;
  }
  if (threadIdx.x < RT) smax[threadIdx.x] = 0u;
  __syncthreads();

  constexpr int EPV = WDT == W_BF16 ? 8 : 16;       // elements per 16 B
  constexpr int ESZ = WDT == W_BF16 ? 2 : 1;
  const int lane = threadIdx.x & 31;
  const int gwarp = blockIdx.x * kWarps + (threadIdx.x >> 5);
  const int nwarps = gridDim.x * kWarps;
  const int Kv = K / EPV * EPV;
  float lmax = 0.f;                                  // for row (lane % RT)

  for (int j0 = gwarp * kVPW; j0 < g.n; j0 += nwarps * kVPW) {
    float acc[kVPW][RT];
    const uint8_t* wrow[kVPW];
    bool ok[kVPW];
    int64_t vid[kVPW];
#pragma unroll
    for (int v = 0; v < kVPW; ++v) {
      const int j = j0 + v;
      ok[v] = j < g.n;
      vid[v] = ok[v] ? (g.ids ? (int64_t)g.ids[j] : (int64_t)j) : 0;
      wrow[v] = reinterpret_cast<const uint8_t*>(g.W) + vid[v] * g.ld_w * ESZ;
#pragma unroll
      for (int r = 0; r < RT; ++r) acc[v][r] = 0.f;
    }
    for (int k = lane * EPV; k < Kv; k += 32 * EPV) {
      uint4 raw[kVPW];
#pragma unroll
      for (int v = 0; v < kVPW; ++v)
        raw[v] = ok[v] ? ld_stream_v4(wrow[v] + (int64_t)k * ESZ)
                       : make_uint4(0, 0, 0, 0);
#pragma unroll
      for (int v = 0; v < kVPW; ++v) {
        float w[EPV];
        expand<WDT>(raw[v], w);
#pragma unroll
        for (int r = 0; r < RT; ++r) {
          const float* hp = hs + r * KP + k;
#pragma unroll
          for (int e = 0; e < EPV; e += 4) {
            const float4 hv = *reinterpret_cast<const float4*>(hp + e);
            acc[v][r] = fmaf(w[e], hv.x, acc[v][r]);
            acc[v][r] = fmaf(w[e + 1], hv.y, acc[v][r]);
            acc[v][r] = fmaf(w[e + 2], hv.z, acc[v][r]);
            acc[v][r] = fmaf(w[e + 3], hv.w, acc[v][r]);
          }
        }
      }
    }
    for (int k = Kv + lane; k < K; k += 32) {
#pragma unroll
      for (int v = 0; v < kVPW; ++v) {
        const float w = ok[v] ? load_scalar_w<WDT>(g.W, vid[v] * g.ld_w + k) : 0.f;
#pragma unroll
        for (int r = 0; r < RT; ++r) acc[v][r] = fmaf(w, hs[r * KP + k], acc[v][r]);
      }
    }
#pragma unroll
    for (int v = 0; v < kVPW; ++v)
#pragma unroll
      for (int r = 0; r < RT; ++r) acc[v][r] = warp_sum(acc[v][r]);

    // lane (v * RT + r) finishes element (row0 + r, j0 + v)
#pragma unroll
    for (int v = 0; v < kVPW; ++v) {
#pragma unroll
      for (int r = 0; r < RT; ++r) {
        if (lane != v * RT + r || !ok[v] || r >= rt) continue;
        const int j = j0 + v;
        const int64_t o = (int64_t)(row0 + r) * g.n + j;
        float y = acc[v][r];
        if constexpr (WDT == W_FP8) y *= g.w_scale[vid[v]];
        if constexpr (EPI == EPI_CLOUD) {
          if (g.bias) y += g.bias[vid[v]];
          if (g.partial_out) g.partial_out[o] = y;
          const float yc = fminf(fmaxf(y, -g.clip), g.clip);
          g.Y[o] = yc;
          lmax = fmaxf(lmax, fabsf(yc));
        } else if constexpr (EPI == EPI_FUSED) {
          // quantize the cloud's clipped partial (Eq. 18), emit the code
          // (and, at the first id, the row scale), dequantize it (Eq. 13)
          const RowQuant rq = row_quant(__ldcg(g.rowmax_in + row0 + r));
          const int code = quantize_one(__ldcg(g.yc + o), rq.k, rq.inv);
          g.codes_out[o] = (int8_t)code;
          if (j == 0) g.scale_out[row0 + r] = rq.s;
          g.Y[(int64_t)(row0 + r) * g.ldy + j] = y + (float)code * rq.s;
        } else {
          g.Y[(int64_t)(row0 + r) * g.ldy + j] =
              g.codes ? y + (float)g.codes[o] * g.row_scale[row0 + r] : y;
        }
      }
    }
  }
  if constexpr (EPI == EPI_CLOUD) {
    // lanes r, r+RT, ... hold maxima of row r
    if (lane < kVPW * RT) atomicMax(&smax[lane % RT], __float_as_uint(lmax));
    __syncthreads();
    if (threadIdx.x < rt) atomicMax(&g.rowmax[row0 + threadIdx.x], smax[threadIdx.x]);
    if (g.q_ticket) {
      // every block's partials and maxima are visible to the last block to
      // arrive, which quantizes them exactly as the quantize pass does
      // (row_quant, quantize_one) and leaves the maxima and its ticket at
      // zero for the next call
      __shared__ int s_last;
      __threadfence();
      __syncthreads();
      if (threadIdx.x == 0) s_last = atomicAdd(g.q_ticket, 1u) == gridDim.x - 1;
      __syncthreads();
      if (s_last) {
        __threadfence();
        __shared__ RowQuant s_rq[RT];
        if (threadIdx.x < rt) {
          const RowQuant rq = row_quant(__ldcg(g.rowmax + row0 + threadIdx.x));
          s_rq[threadIdx.x] = rq;
          g.q_scale[row0 + threadIdx.x] = rq.s;
        }
        __syncthreads();
        // eight independent loads a thread before their codes (one L2
        // round trip per batch, not per entry)
        const int total = rt * g.n;
        const int64_t o0 = (int64_t)row0 * g.n;
        for (int b = 0; b < total; b += 8 * kThreads) {
          float y[8];
#pragma unroll
          for (int u = 0; u < 8; ++u) {
            const int i = b + u * kThreads + threadIdx.x;
            y[u] = i < total ? __ldcg(g.Y + o0 + i) : 0.f;
          }
#pragma unroll
          for (int u = 0; u < 8; ++u) {
            const int i = b + u * kThreads + threadIdx.x;
            if (i < total) {
              const int r = i / g.n;
              g.q_codes[o0 + i] = (int8_t)quantize_one(y[u], s_rq[r].k, s_rq[r].inv);
            }
          }
        }
        if (threadIdx.x < rt) g.rowmax[row0 + threadIdx.x] = 0u;
        if (threadIdx.x == 0) *g.q_ticket = 0u;
      }
    }
  }
}

template <int RT, int WDT, int EPI>
cudaError_t launch_rt(const GatherGemm& g, int sm_count, cudaStream_t st) {
  const size_t smem = (size_t)RT * ((g.K + 7) & ~7) * sizeof(float);
  auto kern = gemv_kernel<RT, WDT, EPI>;
  // the shared-memory opt-in and the occupancy are host calls: made once per
  // device (and shared-memory size) and remembered
  constexpr int kMaxDev = 64, kOccSlots = 8;
  static std::atomic<bool> opted[kMaxDev];
  static std::mutex occ_mu;
  static struct { int dev; size_t smem; int occ; } occ_cache[kOccSlots];
  static int occ_next = 0;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const bool cacheable = dev >= 0 && dev < kMaxDev;
  if (!cacheable || !opted[dev].load()) {
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemLimit);
    if (e != cudaSuccess) return e;
    if (cacheable) opted[dev].store(true);
  }
  int occ = 0;
  {
    std::lock_guard<std::mutex> lock(occ_mu);
    for (const auto& c : occ_cache)
      if (c.occ > 0 && c.dev == dev && c.smem == smem) occ = c.occ;
  }
  if (occ == 0) {
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, kern, kThreads, smem);
    if (e != cudaSuccess) return e;
    if (occ < 1) occ = 1;
    std::lock_guard<std::mutex> lock(occ_mu);
    occ_cache[occ_next] = {dev, smem, occ};
    occ_next = (occ_next + 1) % kOccSlots;
  }
  const int work = (g.n + vpw<RT>() - 1) / vpw<RT>();       // warp tasks
  int blocks = (work + kWarps - 1) / kWarps;
  blocks = blocks < sm_count * occ ? blocks : sm_count * occ;
  if (blocks < 1) blocks = 1;
  for (int row0 = 0; row0 < g.rows; row0 += RT) {
    e = launch_pdl(kern, dim3(blocks), dim3(kThreads), smem, st, g, row0);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

// hidden-state rows one launch covers: as many of 8, 4, 2 as the rows and
// the shared-memory tile allow
int rows_per_launch(int rows, int K) {
  const size_t per_row = (size_t)((K + 7) & ~7) * sizeof(float);
  for (int rt = 8; rt > 1; rt >>= 1)
    if (rows >= rt && rt * per_row <= kSmemLimit) return rt;
  return 1;
}

template <int WDT, int EPI>
cudaError_t launch_wdt(const GatherGemm& g, int sm_count, cudaStream_t st) {
  switch (rows_per_launch(g.rows, g.K)) {
    case 8: return launch_rt<8, WDT, EPI>(g, sm_count, st);
    case 4: return launch_rt<4, WDT, EPI>(g, sm_count, st);
    case 2: return launch_rt<2, WDT, EPI>(g, sm_count, st);
  }
  return launch_rt<1, WDT, EPI>(g, sm_count, st);
}

}  // namespace

int gemv_max_k() { return (int)(kSmemLimit / sizeof(float)) & ~7; }
int gemv_rows_per_launch(int rows, int K) { return rows_per_launch(rows, K); }

cudaError_t launch_gemv(const GatherGemm& g_in, int sm_count, cudaStream_t st) {
  GatherGemm g = g_in;
  if (!g.ldy) g.ldy = g.n;
  // the last-block quantization needs every row in one launch
  if (g.q_ticket && (g.epilogue != EPI_CLOUD || !g.q_codes || !g.q_scale ||
                     rows_per_launch(g.rows, g.K) < g.rows ||
                     (int64_t)g.rows * g.n > kGemvQuantizeMax))
    return cudaErrorNotSupported;
  if (g.epilogue == EPI_FUSED) {
    if (g.w_dtype != W_BF16 || !g.yc || !g.rowmax_in || !g.codes_out || !g.scale_out)
      return cudaErrorNotSupported;
    return launch_wdt<W_BF16, EPI_FUSED>(g, sm_count, st);
  }
  if (g.w_dtype == W_BF16)
    return g.epilogue == EPI_CLOUD ? launch_wdt<W_BF16, EPI_CLOUD>(g, sm_count, st)
                                   : launch_wdt<W_BF16, EPI_ENDPOINT>(g, sm_count, st);
  return g.epilogue == EPI_CLOUD ? launch_wdt<W_FP8, EPI_CLOUD>(g, sm_count, st)
                                 : launch_wdt<W_FP8, EPI_ENDPOINT>(g, sm_count, st);
}

}  // namespace sph
