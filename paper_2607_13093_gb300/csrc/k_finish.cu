// Quantisation of the clipped cloud partials (Eq. 18 with b = 8): one
// symmetric scale per row, round to nearest even.
#include "sm100_ptx.cuh"
#include "sph_common.cuh"
#include "sph_internal.h"

namespace sph {
namespace {

// ---------------------------------------------------------------------------
// quantize: s_r = fl32(max_r / 127); code = rint_even(yc / s_r), |code|<=127
// ---------------------------------------------------------------------------
__global__ void quantize_kernel(const float* __restrict__ Y,
                                const unsigned* __restrict__ rowmax, int n,
                                int8_t* __restrict__ codes,
                                float* __restrict__ row_scale,
                                int rows) {
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  for (int r = blockIdx.y; r < rows; r += gridDim.y) {
    const float a = __uint_as_float(rowmax[r]);
    const float s = __fdiv_rn(a, 127.0f);
    if (blockIdx.x == 0 && threadIdx.x == 0) row_scale[r] = s;
    const float* y = Y + (int64_t)r * n;
    int8_t* c = codes + (int64_t)r * n;
    for (int j = blockIdx.x * blockDim.x + threadIdx.x; j < n;
         j += gridDim.x * blockDim.x) {
      int q = 0;
      if (s > 0.f) {
        q = __float2int_rn(__fdiv_rn(y[j], s));
        q = q > 127 ? 127 : (q < -127 ? -127 : q);
      }
      c[j] = (int8_t)q;
    }
  }
}

}  // namespace

cudaError_t launch_quantize(const float* Y, const unsigned* rowmax, int rows,
                            int n, int8_t* codes, float* row_scale,
                            cudaStream_t st) {
  const int threads = 256;
  int bx = (n + threads * 4 - 1) / (threads * 4);
  bx = bx < 1 ? 1 : (bx > 1024 ? 1024 : bx);
  dim3 grid(bx, rows < 65535 ? rows : 65535);
  return launch_pdl(quantize_kernel, grid, dim3(threads), 0, st, Y, rowmax, n, codes,
                    row_scale, rows);
}

}  // namespace sph
