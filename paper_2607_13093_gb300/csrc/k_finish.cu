// Quantisation of the clipped cloud partials (Eq. 18 with b = 8): one
// symmetric fp32 scale per row, round to nearest even.  The quotient is the
// correctly rounded fp32 division; the oracle divides in fp64, so a code can
// differ by one only where the quotient lies within an fp32 rounding of a
// half-integer.
#include "sm100_ptx.cuh"
#include "sph_common.cuh"
#include "sph_internal.h"

namespace sph {
namespace {

// ---------------------------------------------------------------------------
// quantize: s_r = fl32(max_r / 127); code = rint_even(yc / s_r), |code|<=127
// ---------------------------------------------------------------------------
// The [rows, n] partials are walked as one flat array, eight entries per
// thread: two 16-byte loads, one 8-byte store of the codes (byte stores when
// the code buffer is not 8-byte aligned), and the row of each entry tracked
// across the (at most few) row boundaries inside the eight.
constexpr int kQVec = 8;

__device__ __forceinline__ float row_scale_of(const unsigned* rowmax, int r) {
  return __fdiv_rn(__uint_as_float(rowmax[r]), 127.0f);
}

__device__ __forceinline__ int quantize_one(float y, float s) {
  if (!(s > 0.f)) return 0;
  const int q = __float2int_rn(__fdiv_rn(y, s));
  return q > 127 ? 127 : (q < -127 ? -127 : q);
}

__global__ void quantize_kernel(const float* __restrict__ Y,
                                const unsigned* __restrict__ rowmax, int rows, int n,
                                int8_t* __restrict__ codes,
                                float* __restrict__ row_scale) {
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  for (int64_t r = tid; r < rows; r += stride) row_scale[r] = row_scale_of(rowmax, (int)r);
  const int64_t total = (int64_t)rows * n;
  const bool vec_store = ((uintptr_t)codes & 7) == 0;
  for (int64_t g = tid; g * kQVec < total; g += stride) {
    const int64_t e0 = g * kQVec;
    const bool full = e0 + kQVec <= total;
    float y[kQVec];
    if (full) {
      const float4 u = __ldcs(reinterpret_cast<const float4*>(Y + e0));
      const float4 v = __ldcs(reinterpret_cast<const float4*>(Y + e0) + 1);
      y[0] = u.x; y[1] = u.y; y[2] = u.z; y[3] = u.w;
      y[4] = v.x; y[5] = v.y; y[6] = v.z; y[7] = v.w;
    } else {
#pragma unroll
      for (int i = 0; i < kQVec; ++i) y[i] = e0 + i < total ? Y[e0 + i] : 0.f;
    }
    int r = (int)(e0 / n);
    int64_t next_row = (int64_t)(r + 1) * n;
    float s = row_scale_of(rowmax, r);
    uint32_t packed[2] = {0u, 0u};
#pragma unroll
    for (int i = 0; i < kQVec; ++i) {
      if (e0 + i >= total) break;
      while (e0 + i >= next_row) {
        ++r;
        next_row += n;
        s = row_scale_of(rowmax, r);
      }
      packed[i >> 2] |= (uint32_t)(quantize_one(y[i], s) & 0xFF) << (8 * (i & 3));
    }
    if (full && vec_store) {
      *reinterpret_cast<uint2*>(codes + e0) = make_uint2(packed[0], packed[1]);
    } else {
#pragma unroll
      for (int i = 0; i < kQVec; ++i)
        if (e0 + i < total) codes[e0 + i] = (int8_t)((packed[i >> 2] >> (8 * (i & 3))) & 0xFF);
    }
  }
}

}  // namespace

cudaError_t launch_quantize(const float* Y, const unsigned* rowmax, int rows,
                            int n, int8_t* codes, float* row_scale,
                            cudaStream_t st) {
  const int threads = 256;
  const int64_t groups = ((int64_t)rows * n + kQVec - 1) / kQVec;
  int64_t blocks = (groups + threads - 1) / threads;
  if (blocks < (rows + threads - 1) / threads) blocks = (rows + threads - 1) / threads;
  if (blocks > 4096) blocks = 4096;
  if (blocks < 1) blocks = 1;
  return launch_pdl(quantize_kernel, dim3((unsigned)blocks), dim3(threads), 0, st, Y, rowmax,
                    rows, n, codes, row_scale);
}

}  // namespace sph
