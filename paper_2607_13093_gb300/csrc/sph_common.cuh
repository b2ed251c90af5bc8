// Device helpers shared by the split-head kernels: the counter-based
// generator, number-format conversions, block reductions and the layout of
// the context's scratch arena.
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <cuda_fp8.h>
#include <stdint.h>

namespace sph {

// ---------------------------------------------------------------------------
// Philox4x32 with 10 rounds (Salmon, Moraes, Dror, Shaw, SC'11).  A round
// multiplies counter words 0 and 2 by the two published multipliers, then
// mixes the high halves with the other two words and the key; the key is
// advanced by the two Weyl constants between rounds.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint4 philox4x32_10(uint4 ctr, uint2 key) {
#pragma unroll
  for (int round = 0; round < 10; ++round) {
    const uint32_t a = ctr.x, c = ctr.z;
    const uint32_t hi_a = __umulhi(0xD2511F53u, a), lo_a = 0xD2511F53u * a;
    const uint32_t hi_c = __umulhi(0xCD9E8D57u, c), lo_c = 0xCD9E8D57u * c;
    ctr = make_uint4(hi_c ^ ctr.y ^ key.x, lo_c, hi_a ^ ctr.w ^ key.y, lo_a);
    key.x += 0x9E3779B9u;
    key.y += 0xBB67AE85u;
  }
  return ctr;
}

// Uniform in [0, 1) on the 2^-24 grid from word 0 of the Philox output for
// counter (index, purpose, offset lo, offset hi) and key (seed lo, seed hi).
__device__ __forceinline__ float philox_uniform(uint64_t seed, uint32_t index,
                                                uint32_t purpose,
                                                uint64_t offset) {
  const uint4 r = philox4x32_10(
      make_uint4(index, purpose, (uint32_t)offset, (uint32_t)(offset >> 32)),
      make_uint2((uint32_t)seed, (uint32_t)(seed >> 32)));
  return (float)(r.x >> 8) * 5.9604644775390625e-08f;  // 2^-24
}

// ---------------------------------------------------------------------------
// number formats
// ---------------------------------------------------------------------------
__device__ __forceinline__ float bf16_lo(uint32_t pair) {   // element 0
  return __uint_as_float(pair << 16);
}
__device__ __forceinline__ float bf16_hi(uint32_t pair) {   // element 1
  return __uint_as_float(pair & 0xFFFF0000u);
}

// two e4m3 bytes (low byte = element 0) -> two floats, exact
__device__ __forceinline__ float2 e4m3x2_to_float2(uint16_t two) {
  const __half2_raw h = __nv_cvt_fp8x2_to_halfraw2((__nv_fp8x2_storage_t)two,
                                                   __NV_E4M3);
  return __half22float2(*reinterpret_cast<const __half2*>(&h));
}

// ---------------------------------------------------------------------------
// reductions
// ---------------------------------------------------------------------------
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xFFFFFFFFu, v, o));
  return v;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
  return v;
}

// Block-wide max / sum for blockDim.x a multiple of 32 (<= 1024).  `red`
// is a 32-float shared array; every thread receives the result.
__device__ __forceinline__ float block_max(float v, float* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  v = warp_max(v);
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  const int nw = blockDim.x >> 5;
  v = lane < nw ? red[lane] : -INFINITY;
  return warp_max(v);
}
__device__ __forceinline__ float block_sum(float v, float* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  v = warp_sum(v);
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  const int nw = blockDim.x >> 5;
  v = lane < nw ? red[lane] : 0.f;
  return warp_sum(v);
}

// Reduce 16 per-lane values over the 32 lanes of a warp, one result per
// value index: a butterfly that halves the array at every exchange (16
// shuffles in all).  Lane l ends with the reduction of index
// (l >> 1) & 15; lanes l and l ^ 1 hold the same result.
template <class Op>
__device__ __forceinline__ float warp_reduce_scatter16(const float (&v)[16], Op op, int lane) {
  float a8[8], a4[4], a2[2];
  const bool b16 = lane & 16, b8 = lane & 8, b4 = lane & 4, b2 = lane & 2;
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    const float keep = b16 ? v[k + 8] : v[k], give = b16 ? v[k] : v[k + 8];
    a8[k] = op(keep, __shfl_xor_sync(0xFFFFFFFFu, give, 16));
  }
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const float keep = b8 ? a8[k + 4] : a8[k], give = b8 ? a8[k] : a8[k + 4];
    a4[k] = op(keep, __shfl_xor_sync(0xFFFFFFFFu, give, 8));
  }
#pragma unroll
  for (int k = 0; k < 2; ++k) {
    const float keep = b4 ? a4[k + 2] : a4[k], give = b4 ? a4[k] : a4[k + 2];
    a2[k] = op(keep, __shfl_xor_sync(0xFFFFFFFFu, give, 4));
  }
  const float keep = b2 ? a2[1] : a2[0], give = b2 ? a2[0] : a2[1];
  float r = op(keep, __shfl_xor_sync(0xFFFFFFFFu, give, 2));
  return op(r, __shfl_xor_sync(0xFFFFFFFFu, r, 1));
}

struct MaxOp {
  __device__ float operator()(float a, float b) const { return fmaxf(a, b); }
};
struct SumOp {
  __device__ float operator()(float a, float b) const { return a + b; }
};

// ---------------------------------------------------------------------------
// the int8 quantizer (Eq. 18 with b = 8), shared by the quantize kernel and
// the fused endpoint epilogue so that both round identically
// ---------------------------------------------------------------------------
struct RowQuant {
  float s;     // row scale fl32(max / 127)
  float k;     // exact lift 2^64 for scales below 2^-64, else 1
  float inv;   // fl32(1 / (s * k)); 0 for an all-zero row (codes 0)
};
// From the bit pattern of the row's clipped |max|.  A scale below 2^-64
// (partials below about 1e-17) is lifted by the exact factor 2^64 on both
// sides so that its reciprocal stays finite.
__device__ __forceinline__ RowQuant row_quant(unsigned max_bits) {
  RowQuant q;
  q.s = __fdiv_rn(__uint_as_float(max_bits), 127.0f);
  q.k = q.s < 0x1p-64f ? 0x1p64f : 1.f;
  q.inv = q.s > 0.f ? __frcp_rn(q.s * q.k) : 0.f;
  return q;
}
// code = round-half-even(y / s) in [-127, 127], as the exact product
// (y k) * fl32(1 / (s k)) rounded once to an integer: one fused multiply-add
// of 1.5 * 2^23, whose sum lies in [2^23, 2^24) where the fp32 grid is the
// integers (|quotient| <= 127 here), so the FMA's round-to-nearest-even is
// the integer rounding and the low bits are the code.  (y k is exact: k is a
// power of two.)  This keeps the conversion on the FMA pipe.
__device__ __forceinline__ int quantize_one(float y, float k, float inv_s) {
  const float t = __fmaf_rn(y * k, inv_s, 12582912.0f);    // 1.5 * 2^23
  const int q = __float_as_int(t) - 0x4B400000;            // bits of 1.5 * 2^23
  return max(-127, min(127, q));
}

// 2^x by the special-function unit's approximation (`ex2.approx.ftz`: a
// relative error of a few ulp; results below 2^-126 flush to 0, which for
// softmax weights relative to the row maximum is below any weight that can
// move a draw).  One instruction, where exp2f adds a scaling path for
// subnormal results.
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// The int8 code in byte e (0..3) of a word whose bytes were first XORed with
// 0x80, as an exact float: the byte permute forms the fp32 2^23 + (code +
// 128), and one exact subtraction leaves the code.  (Integer and ALU pipes
// instead of an int-to-float conversion.)
__device__ __forceinline__ float code_f32(unsigned w_x80, int e) {
  return __uint_as_float(__byte_perm(w_x80, 0x4B000000u, 0x7440u | (unsigned)e)) - 8388736.0f;
}

// Non-negative floats order like their bit patterns, so a row maximum of
// |y| can be kept as an unsigned atomicMax.
__device__ __forceinline__ void atomic_max_nonneg(unsigned int* addr, float v) {
  atomicMax(addr, __float_as_uint(v));
}

}  // namespace sph
