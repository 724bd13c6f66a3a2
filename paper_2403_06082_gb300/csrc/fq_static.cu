// fq_linear_forward_static: the layer forward for callers that cannot allocate device memory.
//
// Some callers have no way to obtain a device buffer for the forward's scratch space: code
// running inside a host framework that owns every allocation and hands out only the tensors
// of the model, plugin interfaces whose signature carries inputs and outputs but no
// workspace, and C programs linked against this library without any allocator of their own.
// For them this entry point uses a scratch array that lives in the library itself: a
// file-scope __device__ array, reserved on every GPU that loads the library and held until
// the process exits.  It allocates nothing, ever.
//
// The array holds the same intermediate values a caller-provided workspace would hold (the
// device status word, z, u and the per-tile sums of z), so its size bounds the sizes this
// entry point accepts; larger requests are refused with FQ_ERR_UNSUPPORTED.  Every call uses
// the same array and leaves its contents behind for the next call, so calls whose kernels may
// run at the same time on the GPU (different streams, or different host threads) race on it.
// The device status word lives at the head of that array; fq_static_check reads it and, after
// a timeout, clears the array's header so that later calls start from a valid state.
//
// The array's device address is looked up on every call (cudaGetSymbolAddress, with the
// caller's device current), never cached: a cached address would outlive a device reset
// (cudaDeviceReset, or anything else that destroys and re-creates the primary context), after
// which the module is loaded again and the array may sit elsewhere.  The first call on a device
// (and the first after a reset) loads the library's device code there.
#include <cuda_runtime.h>

#include "fq_internal.h"

namespace fq {
namespace {

constexpr size_t kStaticScratchBytes = FQ_STATIC_SCRATCH_BYTES;

static __device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

// Device address of g_static_scratch on the current device.  The symbol's host-side name is a
// stand-in, not a device address, and must never be passed to a kernel.
cudaError_t scratch_for_current_device(void** out) {
  void* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_static_scratch);
  if (e != cudaSuccess) return e;
  *out = p;
  return cudaSuccess;
}

}  // namespace
}  // namespace fq

extern "C" fq_status fq_linear_forward_static(const void* x, int M, int d_in, const void* T_in,
                                              const fq_packed* C, const void* T_out_t,
                                              int d_out, const float* gamma, void* y, int mode,
                                              fq_stream_t stream) {
  if (!C) return FQ_ERR_INVALID_ARG;
  const size_t need = fq_workspace_bytes(M, d_in, C->n_in, C->n_out, d_out, mode);
  if (need == 0) return FQ_ERR_INVALID_ARG;
  if (need > fq::kStaticScratchBytes) return FQ_ERR_UNSUPPORTED;
  void* scratch = nullptr;
  if (fq::scratch_for_current_device(&scratch) != cudaSuccess) return FQ_ERR_CUDA;
  // Nothing left behind by the previous call needs clearing here: the status word at the head
  // of the scratch is zeroed by the forward itself before its kernels report into it, and z, u
  // and the sums of z are written before they are read within one call.
  return fq_linear_forward(x, M, d_in, T_in, C, T_out_t, d_out, gamma, y, scratch,
                           fq::kStaticScratchBytes, mode, stream);
}

extern "C" fq_status fq_static_check(fq_stream_t stream) {
  void* scratch = nullptr;
  if (fq::scratch_for_current_device(&scratch) != cudaSuccess) return FQ_ERR_CUDA;
  const fq_status st = fq_check(scratch, stream);
  if (st == FQ_ERR_TIMEOUT) {
    // the header's flags and counters may be mid-call: a zero-filled header is a valid start
    auto s = reinterpret_cast<cudaStream_t>(stream);
    if (cudaMemsetAsync(scratch, 0, fq::kWsHeader, s) != cudaSuccess ||
        cudaStreamSynchronize(s) != cudaSuccess)
      return FQ_ERR_CUDA;
  }
  return st;
}
