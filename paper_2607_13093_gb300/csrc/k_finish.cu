// Quantisation of the clipped cloud partials (Eq. 18 with b = 8): one
// symmetric fp32 scale per row, round to nearest even.  The quotient is the
// partial times the correctly rounded fp32 reciprocal of the scale, rounded
// once to an integer (quantize_one); the oracle divides in fp64, so a code
// can differ by one only where the quotient lies within one rounding of the
// reciprocal (about 8e-6 at 127) of a half-integer.
#include <climits>

#include "sm100_ptx.cuh"
#include "sph_common.cuh"
#include "sph_internal.h"

namespace sph {
namespace {

// ---------------------------------------------------------------------------
// quantize: s_r = fl32(max_r / 127); code = rint_even(yc * fl32(1 / s_r)), |code|<=127
// ---------------------------------------------------------------------------
// A work item is one row and a span of 2048 of its entries: the row's scale
// is found once per item.  Where rows start 16-byte aligned each thread takes
// eight consecutive entries (two 16-byte loads, one 8-byte store of the
// codes); otherwise it takes every 256th entry of the span, so that a warp's
// loads and stores stay contiguous.
constexpr int kQVec = 8;
constexpr int kQThreads = 256;
constexpr int kQSpan = kQThreads * kQVec;

__global__ void __launch_bounds__(kQThreads)
quantize_kernel(const float* __restrict__ Y, const unsigned* __restrict__ rowmax, int rows,
                int n, int8_t* __restrict__ codes, float* __restrict__ row_scale) {
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  const int spans = (n + kQSpan - 1) / kQSpan;
  const int64_t items = (int64_t)rows * spans;
  const bool narrow = items <= INT_MAX;
  // rows start 16-byte aligned in Y (and 8-byte aligned in codes) when n
  // allows; Y itself is 256-byte aligned
  const bool vec_load = (n & 3) == 0;
  const bool vec_store = (n & 7) == 0 && ((uintptr_t)codes & 7) == 0;
  for (int64_t it = blockIdx.x; it < items; it += gridDim.x) {
    int r, sp;
    if (narrow) {
      r = (int)((uint32_t)it / (uint32_t)spans);
      sp = (int)((uint32_t)it - (uint32_t)r * (uint32_t)spans);
    } else {
      r = (int)(it / spans);
      sp = (int)(it - (int64_t)r * spans);
    }
    const RowQuant rq = row_quant(rowmax[r]);
    const float k = rq.k, inv_s = rq.inv;
    if (sp == 0 && threadIdx.x == 0) row_scale[r] = rq.s;
    const int64_t row0 = (int64_t)r * n;
    if (!vec_load) {
      // rows not 16-byte aligned: entry i of the thread is column
      // span + i * 256 + thread, so each warp instruction reads 32 adjacent
      // partials and writes 32 adjacent codes
      const int cb = sp * kQSpan + threadIdx.x;
      float y[kQVec];
#pragma unroll
      for (int i = 0; i < kQVec; ++i) {
        const int c = cb + i * kQThreads;
        y[i] = c < n ? __ldcs(Y + row0 + c) : 0.f;
      }
#pragma unroll
      for (int i = 0; i < kQVec; ++i) {
        const int c = cb + i * kQThreads;
        if (c < n) codes[row0 + c] = (int8_t)quantize_one(y[i], k, inv_s);
      }
      continue;
    }
    const int c0 = sp * kQSpan + threadIdx.x * kQVec;
    if (c0 >= n) continue;
    const int64_t e0 = row0 + c0;
    const bool full = c0 + kQVec <= n;
    float y[kQVec];
    if (full) {
      const float4 u = __ldcs(reinterpret_cast<const float4*>(Y + e0));
      const float4 v = __ldcs(reinterpret_cast<const float4*>(Y + e0) + 1);
      y[0] = u.x; y[1] = u.y; y[2] = u.z; y[3] = u.w;
      y[4] = v.x; y[5] = v.y; y[6] = v.z; y[7] = v.w;
    } else {
#pragma unroll
      for (int i = 0; i < kQVec; ++i) y[i] = c0 + i < n ? Y[e0 + i] : 0.f;
    }
    uint32_t packed[2] = {0u, 0u};
#pragma unroll
    for (int i = 0; i < kQVec; ++i)
      packed[i >> 2] |= (uint32_t)(quantize_one(y[i], k, inv_s) & 0xFF) << (8 * (i & 3));
    if (full && vec_store) {
      *reinterpret_cast<uint2*>(codes + e0) = make_uint2(packed[0], packed[1]);
    } else {
#pragma unroll
      for (int i = 0; i < kQVec; ++i)
        if (c0 + i < n) codes[e0 + i] = (int8_t)((packed[i >> 2] >> (8 * (i & 3))) & 0xFF);
    }
  }
}

}  // namespace

cudaError_t launch_quantize(const float* Y, const unsigned* rowmax, int rows,
                            int n, int8_t* codes, float* row_scale,
                            cudaStream_t st) {
  const int64_t items = (int64_t)rows * ((n + kQSpan - 1) / kQSpan);
  int64_t blocks = items < 8192 ? items : 8192;
  if (blocks < 1) blocks = 1;
  return launch_pdl(quantize_kernel, dim3((unsigned)blocks), dim3(kQThreads), 0, st, Y, rowmax,
                    rows, n, codes, row_scale);
}

}  // namespace sph
