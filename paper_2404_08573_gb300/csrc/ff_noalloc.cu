// An allocation-free variant of the bf16 forward pass, for callers that may
// not allocate device memory (for example code running where cudaMalloc is
// forbidden or already reserved by a host application's own memory pool, or
// code that must not change the device's memory footprint after start-up).
//
// The caller passes the layer input, weights, bias and every output.  The
// per-tile goodness partials that the forward GEMM hands to the goodness
// kernel live in the file-scope array below instead of a layer workspace.
// That array is a fixed part of every device that loads this library, held
// until the process exits.
#include "ff_internal.cuh"

namespace ff {
namespace {

// Scratch: [0, 64) words hold the kernels' error word when the caller passes
// no status pointer; partials start at word 64.
constexpr size_t kNoAllocScratchFloats = size_t(1) << 20;  // 4 MiB
constexpr size_t kNoAllocPartialOffset = 64;
static __device__ __align__(256) float g_noalloc_scratch[kNoAllocScratchFloats];

// Device address of the scratch array on the current device.  In host code
// the array's name is only a host-side stand-in, so the address is looked up
// with the caller's device current -- on every call rather than cached, so
// that a context recreated after cudaDeviceReset never sees a stale address
// (the lookup enqueues nothing; the first one on a device also loads the
// library's device code there).
cudaError_t scratch_address(float** out) {
  void* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
  if (e != cudaSuccess) return e;
  *out = static_cast<float*>(p);
  return cudaSuccess;
}

}  // namespace
}  // namespace ff

using namespace ff;

extern "C" FF_API ff_status ff_forward_noalloc(const void* x, const float* row_scale, const void* W_bf16,
                                               const float* bias, int rows, int in_features, int out_features,
                                               void* h_out, float* goodness, float* next_scale, int* device_status,
                                               void* stream) {
  if (rows < 0 || in_features < 1 || out_features < 1) return FF_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (rows == 0) {
    // nothing to compute; the status word still reads 0 afterwards
    if (device_status && cudaMemsetAsync(device_status, 0, sizeof(int), st) != cudaSuccess) return FF_ERR_CUDA;
    return FF_OK;
  }
  if (!x || !row_scale || !W_bf16 || !h_out) return FF_ERR_INVALID_ARG;
  const size_t partials = (size_t)tc_fwd_ntiles(rows, out_features, false) * (size_t)rows;
  if (partials > kNoAllocScratchFloats - kNoAllocPartialOffset) return FF_ERR_INVALID_ARG;
  if (!tc_supported()) return FF_ERR_UNSUPPORTED;
  float* scratch = nullptr;
  cudaError_t e = scratch_address(&scratch);
  if (e != cudaSuccess) return FF_ERR_CUDA;
  int* err = device_status ? device_status : reinterpret_cast<int*>(scratch);
  // the error word must start at zero; the partials are written before they are read
  e = cudaMemsetAsync(err, 0, sizeof(int), st);
  if (e != cudaSuccess) return FF_ERR_CUDA;
  const int ldK = row_stride(in_features), ldN = row_stride(out_features);
  float* gpart = scratch + kNoAllocPartialOffset;
  EpiArgs ep{row_scale, bias, h_out, ldN, gpart};
  e = tc_gemm_fwd(static_cast<const bf16*>(x), ldK, static_cast<const bf16*>(W_bf16), ldK, rows, out_features,
                  in_features, ep, err, st);
  if (e == cudaErrorInvalidValue) return FF_ERR_INVALID_ARG;  // operand alignment / tensor-map limits
  if (e != cudaSuccess) return FF_ERR_CUDA;
  FinalizeArgs fa{};
  fa.gpart = gpart;
  fa.ntiles = tc_fwd_ntiles(rows, out_features, false);
  fa.M = rows;
  fa.g_out = goodness;
  fa.s_next = next_scale;
  fa.err = err;
  e = launch_finalize(fa, st);
  return e == cudaSuccess ? FF_OK : FF_ERR_CUDA;
}
