// Allocation-free variant of the cloud call.
//
// Some callers cannot allocate device memory at the time they run the
// cloud step: code running under an allocator that is locked or owned by
// another runtime, a custom memory pool that hands out only the buffers it
// was sized for, or a serving loop that must never touch cudaMalloc (which
// may synchronise the device) once it is running.  Such callers cannot create
// a context either, since a context owns scratch memory.  For them this
// file keeps the cloud call's scratch -- the clipped fp32 partials and the
// per-row maxima -- in one fixed, file-scope device array, and the entry
// point below uses it instead of context scratch.  The caller still passes
// every input and output buffer.
//
// The array costs kNoallocBytes of device memory on every GPU that loads
// the library's module, until the process exits.  With CUDA's lazy module
// loading (the default), a module -- this array included -- is loaded onto a
// device the first time one of its kernels or symbols is used there, so the
// FIRST call on each device does allocate device memory (and may
// synchronise): callers make one warm-up call before they enter the region
// where nothing may allocate.  Every later call allocates nothing.  All
// calls share the array: two calls whose kernels overlap on the GPU
// (different streams, or different host threads) corrupt each other's
// results, so such callers must serialise.
//
// The call always takes the CUDA-core GEMV path, which re-reads the kept W
// rows once per 8 hidden-state rows: it is meant for few rows.
#include <cmath>
#include <cstdio>
#include <mutex>

#include "sph.h"
#include "sph_internal.h"

namespace {

constexpr size_t kNoallocBytes = SPH_NOALLOC_SCRATCH_BYTES;
constexpr int kMaxDevices = 64;

// The shared scratch: [rows * n_keep] clipped partials, then [rows] maxima.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoallocBytes];

std::mutex g_setup_mu;
void* g_scratch_addr[kMaxDevices] = {};   // device address per device

size_t round256(size_t x) { return (x + 255) / 256 * 256; }

void put(char* msg, size_t len, const char* text) {
  if (msg && len) snprintf(msg, len, "%s", text);
}

}  // namespace

extern "C" sph_status sph_partial_logits_noalloc(
    int device, void* cuda_stream, const float* h_cloud, int64_t rows,
    int64_t ld_h, const void* W_h, sph_dtype w_dtype, int64_t V, int64_t d_h,
    int64_t ld_w, const float* w_row_scale, const float* bias,
    const int32_t* keep_ids, int64_t n_keep, float clip,
    sph_act_mode act_mode, int8_t* codes, float* row_scale,
    float* partial_out, size_t* payload_bytes, char* err_msg,
    size_t err_msg_len) {
  put(err_msg, err_msg_len, "");
  if (device < 0 || device >= kMaxDevices) {
    put(err_msg, err_msg_len, "device index out of range");
    return SPH_ERR_INVALID_ARG;
  }
  if (!h_cloud || !W_h || !codes || !row_scale) {
    put(err_msg, err_msg_len, "h_cloud, W_h, codes and row_scale must be non-NULL");
    return SPH_ERR_INVALID_ARG;
  }
  if (rows < 1 || rows > (1 << 20)) {
    put(err_msg, err_msg_len, "rows out of [1, 2^20]");
    return SPH_ERR_INVALID_ARG;
  }
  if (d_h < 1 || V < 1 || V > INT32_MAX || n_keep < 1 || n_keep > V ||
      ld_h < d_h || ld_w < d_h || (!keep_ids && n_keep != V)) {
    put(err_msg, err_msg_len, "inconsistent sizes (rows, d_h, V, n_keep, ld_h, ld_w)");
    return SPH_ERR_INVALID_ARG;
  }
  if (!(std::isfinite(clip) && clip > 0.f)) {
    put(err_msg, err_msg_len, "clip must be finite and > 0");
    return SPH_ERR_INVALID_ARG;
  }
  if ((w_dtype != SPH_DTYPE_BF16 && w_dtype != SPH_DTYPE_FP8_E4M3) ||
      (act_mode != SPH_ACT_FP32 && act_mode != SPH_ACT_BF16) ||
      (w_dtype == SPH_DTYPE_FP8_E4M3 && !w_row_scale)) {
    put(err_msg, err_msg_len, "bad w_dtype / act_mode, or fp8 weights without w_row_scale");
    return SPH_ERR_INVALID_ARG;
  }
  const int esz = w_dtype == SPH_DTYPE_BF16 ? 2 : 1;
  if (((uintptr_t)W_h & 15) || ((ld_w * esz) & 15)) {
    put(err_msg, err_msg_len, "W_h base and row stride must be 16-byte aligned");
    return SPH_ERR_INVALID_ARG;
  }
  if (d_h > sph::gemv_max_k()) {
    put(err_msg, err_msg_len, "d_h too large for the allocation-free path");
    return SPH_ERR_UNSUPPORTED;
  }
  // the fixed scratch must hold rows*n_keep floats plus rows maxima
  if (rows > (int64_t)(kNoallocBytes / 4) || n_keep > (int64_t)(kNoallocBytes / 4) ||
      round256((size_t)rows * (size_t)n_keep * 4) + round256((size_t)rows * 4) >
          kNoallocBytes) {
    char buf[160];
    snprintf(buf, sizeof buf,
             "rows*n_keep*4 + rows*4 bytes exceed the fixed scratch of %zu bytes",
             kNoallocBytes);
    put(err_msg, err_msg_len, buf);
    return SPH_ERR_UNSUPPORTED;
  }
  if (payload_bytes) *payload_bytes = sph_payload_bytes(rows, n_keep);

  int prev = -1;
  const cudaError_t ge = cudaGetDevice(&prev);
  if (ge != cudaSuccess) {
    put(err_msg, err_msg_len, cudaGetErrorString(ge));
    return SPH_ERR_CUDA;
  }
  if (prev != device && cudaSetDevice(device) != cudaSuccess) {
    put(err_msg, err_msg_len, "cudaSetDevice failed");
    return SPH_ERR_CUDA;
  }
  sph_status st = SPH_OK;
  void* base = nullptr;
  {
    // once per device, with that device current: the host-side name of the
    // array is not a device address, so look the address up
    std::lock_guard<std::mutex> lock(g_setup_mu);
    if (!g_scratch_addr[device]) {
      void* p = nullptr;
      const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
      if (e != cudaSuccess || !p) {
        put(err_msg, err_msg_len, "cudaGetSymbolAddress failed for the fixed scratch");
        st = SPH_ERR_CUDA;
      } else {
        g_scratch_addr[device] = p;
      }
    }
    base = g_scratch_addr[device];
  }
  if (st == SPH_OK) {
    cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
    float* Y = static_cast<float*>(base);
    unsigned* rowmax = reinterpret_cast<unsigned*>(
        static_cast<char*>(base) + round256((size_t)rows * (size_t)n_keep * 4));
    int sm_count = 0;
    cudaError_t e = cudaDeviceGetAttribute(&sm_count, cudaDevAttrMultiProcessorCount, device);
    // the maxima accumulate with atomicMax, so they must start at zero;
    // the partials are fully overwritten by every call
    if (e == cudaSuccess) e = cudaMemsetAsync(rowmax, 0, (size_t)rows * 4, stream);
    if (e == cudaSuccess) {
      sph::GatherGemm gg{};
      gg.h = h_cloud; gg.ld_h = ld_h; gg.rows = (int)rows;
      gg.W = W_h; gg.ld_w = ld_w; gg.V = V;
      gg.w_dtype = w_dtype == SPH_DTYPE_BF16 ? sph::W_BF16 : sph::W_FP8;
      gg.w_scale = w_row_scale; gg.K = (int)d_h;
      gg.ids = keep_ids; gg.n = (int)n_keep;
      gg.act_bf16 = act_mode == SPH_ACT_BF16;
      gg.epilogue = sph::EPI_CLOUD;
      gg.bias = bias; gg.clip = clip; gg.partial_out = partial_out;
      gg.Y = Y; gg.rowmax = rowmax; gg.status = nullptr;
      e = sph::launch_gemv(gg, sm_count, stream);
    }
    if (e == cudaSuccess)
      e = sph::launch_quantize(Y, rowmax, (int)rows, (int)n_keep, codes, row_scale, stream);
    if (e != cudaSuccess) {
      put(err_msg, err_msg_len, cudaGetErrorString(e));
      st = SPH_ERR_CUDA;
    }
  }
  if (prev >= 0 && prev != device) cudaSetDevice(prev);
  return st;
}
