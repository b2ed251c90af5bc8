// Row-wise kernels that finish the split-head step:
//   quantize : Eq. 18 with b = 8 on the clipped cloud partials
//   sample   : Eq. 14-15, inverse-CDF draw with a Philox uniform per row
//   verify   : speculative acceptance of k drafts per session (standard
//              speculative sampling, residual draw at the first rejection)
//
// Sampling is a two-level inverse CDF: each 128-id step of a row gets its
// weight sum (one warp per step, each lane summing 4 consecutive ids), a
// single warp scans the step sums in ascending id order to find the step
// holding u * total, then scans that step lane by lane.  Everything is in
// ascending vocabulary-id order, as the oracle's CDF.
#include "sm100_ptx.cuh"
#include "sph_common.cuh"
#include "sph_internal.h"

namespace sph {
namespace {

constexpr int kStep = 128;              // ids per step (32 lanes x 4)
constexpr int kSampleThreads = 512;
constexpr int kMaxSteps = 32768;        // n <= 4,194,304
constexpr int kMaxN = kMaxSteps * kStep;
constexpr int kAccept = -2;             // verify: draft accepted (-1 = id not kept)

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

// ---------------------------------------------------------------------------
// block-level inverse CDF over weights w(j) >= 0, j in [0, n)
// ---------------------------------------------------------------------------
// Step sums: warp w handles steps w, w + nwarps, ...; lane l sums ids
// 4l..4l+3 of the step in ascending order, then the warp adds the lanes.
template <class Wt>
__device__ float step_sums(int n, const Wt& wt, float* steps, float* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nw = blockDim.x >> 5;
  const int nsteps = (n + kStep - 1) / kStep;
  float tot = 0.f;
  for (int s = warp; s < nsteps; s += nw) {
    const int j0 = s * kStep + 4 * lane;
    float acc = 0.f;
#pragma unroll
    for (int e = 0; e < 4; ++e)
      if (j0 + e < n) acc += wt(j0 + e);
    acc = warp_sum(acc);
    if (lane == 0) steps[s] = acc;
    tot += acc;
  }
  __syncthreads();
  return block_sum(lane == 0 ? tot : 0.f, red);   // (not used for the search)
}

// Warp 0 only: find the first id whose CDF exceeds u * total, where the
// total and the prefix sums come from `steps` in ascending step order.
// Returns the id (lane 0's value is authoritative; all lanes agree).
template <class Wt>
__device__ int warp_search(int n, const Wt& wt, const float* steps, float u) {
  const int lane = threadIdx.x & 31;
  const int nsteps = (n + kStep - 1) / kStep;
  const int per = (nsteps + 31) / 32;
  const int s0 = min(nsteps, lane * per), s1 = min(nsteps, s0 + per);
  float local = 0.f;
  for (int s = s0; s < s1; ++s) local += steps[s];
  float incl = local;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const float t = __shfl_up_sync(0xFFFFFFFFu, incl, o);
    if (lane >= o) incl += t;
  }
  const float excl = incl - local;
  const float total = __shfl_sync(0xFFFFFFFFu, incl, 31);
  const float target = u * total;
  // the lane whose step range holds the target (last lane with weight
  // if rounding pushes the target past every range)
  const unsigned hit = __ballot_sync(0xFFFFFFFFu, local > 0.f && target >= excl && target < incl);
  const unsigned nzl = __ballot_sync(0xFFFFFFFFu, local > 0.f);
  int owner = hit ? __ffs(hit) - 1 : (nzl ? 31 - __clz(nzl) : 0);
  // owner walks its steps
  int sstar = -1;
  float before = 0.f;
  if (lane == owner) {
    float run = excl;
    int last_nz = -1;
    float before_last = excl;
    for (int s = s0; s < s1; ++s) {
      const float w = steps[s];
      if (w > 0.f) { last_nz = s; before_last = run; }
      if (w > 0.f && target < run + w) { sstar = s; before = run; break; }
      run += w;
    }
    if (sstar < 0) { sstar = last_nz; before = before_last; }
    if (sstar < 0) { sstar = s0; before = excl; }
  }
  sstar = __shfl_sync(0xFFFFFFFFu, sstar, owner);
  before = __shfl_sync(0xFFFFFFFFu, before, owner);
  const float t2 = target - before;
  // inside the step: lane l owns ids 4l..4l+3
  const int j0 = sstar * kStep + 4 * lane;
  float w[4];
  float lsum = 0.f;
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    w[e] = (j0 + e < n) ? wt(j0 + e) : 0.f;
    lsum += w[e];
  }
  float linc = lsum;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const float t = __shfl_up_sync(0xFFFFFFFFu, linc, o);
    if (lane >= o) linc += t;
  }
  const float lexc = linc - lsum;
  const unsigned h2 = __ballot_sync(0xFFFFFFFFu, lsum > 0.f && t2 >= lexc && t2 < linc);
  const unsigned nz2 = __ballot_sync(0xFFFFFFFFu, lsum > 0.f);
  const int l2 = h2 ? __ffs(h2) - 1 : (nz2 ? 31 - __clz(nz2) : 0);
  int jstar = -1;
  if (lane == l2) {
    float run = lexc;
    int last_nz = -1;
    for (int e = 0; e < 4; ++e) {
      if (w[e] > 0.f) last_nz = j0 + e;
      if (w[e] > 0.f && t2 < run + w[e]) { jstar = j0 + e; break; }
      run += w[e];
    }
    if (jstar < 0) jstar = last_nz >= 0 ? last_nz : min(j0, n - 1);
  }
  return __shfl_sync(0xFFFFFFFFu, jstar, l2);
}

__device__ float row_max(const float* z, int n, float* red) {
  float m = -INFINITY;
  for (int j = threadIdx.x; j < n; j += blockDim.x) m = fmaxf(m, z[j]);
  return block_max(m, red);
}

struct ExpWeight {                      // w_j = exp((z_j - m) / tau)
  const float* z;
  float m, inv_tau;
  __device__ float operator()(int j) const { return expf((z[j] - m) * inv_tau); }
};

struct ResidualWeight {                 // max(0, p_j - q_j)
  const float* z;
  const float* q;                       // nullptr: one-hot at xi
  float m, inv_tau, inv_sum;
  int xi;
  __device__ float operator()(int j) const {
    const float p = expf((z[j] - m) * inv_tau) * inv_sum;
    if (q) return fmaxf(0.f, p - q[j]);
    return j == xi ? 0.f : p;
  }
};

__global__ void __launch_bounds__(kSampleThreads)
sample_kernel(const float* __restrict__ Z, int n,
              const int32_t* __restrict__ ids, float inv_tau, uint64_t seed,
              uint64_t offset, int32_t* __restrict__ tokens) {
  extern __shared__ float steps[];
  __shared__ float red[32];
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  const int r = blockIdx.x;
  const float* z = Z + (int64_t)r * n;
  const float m = row_max(z, n, red);
  const ExpWeight wt{z, m, inv_tau};
  step_sums(n, wt, steps, red);
  __syncthreads();
  if (threadIdx.x < 32) {
    const float u = philox_uniform(seed, (uint32_t)r, 0u, offset);
    const int j = warp_search(n, wt, steps, u);
    if (threadIdx.x == 0) tokens[r] = ids ? ids[j] : j;
  }
}

// ---------------------------------------------------------------------------
// verification: one CTA per session
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

__global__ void __launch_bounds__(kSampleThreads)
verify_kernel(const float* __restrict__ Z, int k, int n,
              const int32_t* __restrict__ ids, int V, float inv_tau,
              const int32_t* __restrict__ draft, const float* __restrict__ q,
              uint64_t seed, uint64_t offset, int32_t* __restrict__ n_acc,
              int32_t* __restrict__ next_token) {
  extern __shared__ float steps[];
  __shared__ float red[32];
  __shared__ int s_decision;            // kAccept, or the rejected draft's index
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  const int s = blockIdx.x;
  const float u = philox_uniform(seed, (uint32_t)s, (uint32_t)(1 + k), offset);
  int i = 0;
  for (; i < k; ++i) {
    const float* z = Z + ((int64_t)s * (k + 1) + i) * n;
    const float m = row_max(z, n, red);
    const ExpWeight wt{z, m, inv_tau};
    const float S = step_sums(n, wt, steps, red);
    if (threadIdx.x == 0) {
      const int x = draft[(int64_t)s * k + i];
      const int xi = find_compact(ids, n, V, x);
      const float px = xi >= 0 ? expf((z[xi] - m) * inv_tau) / S : 0.f;
      const float* qrow = q ? q + ((int64_t)s * k + i) * n : nullptr;
      const float qx = xi >= 0 ? (qrow ? qrow[xi] : 1.f) : 0.f;
      const float r = philox_uniform(seed, (uint32_t)s, (uint32_t)(1 + i), offset);
      s_decision = (r * qx < px) ? kAccept : xi;
    }
    __syncthreads();
    const int dec = s_decision;
    __syncthreads();
    if (dec == kAccept) continue;
    // rejected at i: residual max(0, p_i - q_i)
    const float* qrow = q ? q + ((int64_t)s * k + i) * n : nullptr;
    const ResidualWeight rw{z, qrow, m, inv_tau, 1.f / S, dec};
    const float tot = step_sums(n, rw, steps, red);
    __syncthreads();
    int j;
    if (tot > 0.f) {
      if (threadIdx.x < 32) {
        j = warp_search(n, rw, steps, u);
        if (threadIdx.x == 0) { n_acc[s] = i; next_token[s] = ids ? ids[j] : j; }
      }
    } else {
      step_sums(n, wt, steps, red);
      __syncthreads();
      if (threadIdx.x < 32) {
        j = warp_search(n, wt, steps, u);
        if (threadIdx.x == 0) { n_acc[s] = i; next_token[s] = ids ? ids[j] : j; }
      }
    }
    return;
  }
  // all k accepted: bonus token from p_k
  const float* z = Z + ((int64_t)s * (k + 1) + k) * n;
  const float m = row_max(z, n, red);
  const ExpWeight wt{z, m, inv_tau};
  step_sums(n, wt, steps, red);
  __syncthreads();
  if (threadIdx.x < 32) {
    const int j = warp_search(n, wt, steps, u);
    if (threadIdx.x == 0) { n_acc[s] = k; next_token[s] = ids ? ids[j] : j; }
  }
}

}  // namespace

int sample_max_n() { return kMaxN; }

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

cudaError_t launch_sample(const float* Z, int rows, int n, const int32_t* ids,
                          float inv_tau, uint64_t seed, uint64_t offset,
                          int32_t* tokens, cudaStream_t st) {
  const size_t smem = (size_t)((n + kStep - 1) / kStep) * sizeof(float);
  cudaError_t e = cudaFuncSetAttribute(
      sample_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
      (int)(kMaxSteps * sizeof(float)));
  if (e != cudaSuccess) return e;
  return launch_pdl(sample_kernel, dim3(rows), dim3(kSampleThreads), smem, st, Z, n, ids,
                    inv_tau, seed, offset, tokens);
}

cudaError_t launch_verify(const float* Z, int sessions, int k, int n,
                          const int32_t* ids, int V, float inv_tau,
                          const int32_t* draft, const float* q, uint64_t seed,
                          uint64_t offset, int32_t* n_acc, int32_t* next_token,
                          cudaStream_t st) {
  const size_t smem = (size_t)((n + kStep - 1) / kStep) * sizeof(float);
  cudaError_t e = cudaFuncSetAttribute(
      verify_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
      (int)(kMaxSteps * sizeof(float)));
  if (e != cudaSuccess) return e;
  return launch_pdl(verify_kernel, dim3(sessions), dim3(kSampleThreads), smem, st, Z, k, n,
                    ids, V, inv_tau, draft, q, seed, offset, n_acc, next_token);
}

}  // namespace sph
