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
// The device status word lives in that array too, out of the caller's reach: device-side
// findings (a bounded wait that ran out) are not reported by this entry point.
#include <cuda_runtime.h>

#include <mutex>

#include "fq_internal.h"

namespace fq {
namespace {

constexpr size_t kStaticScratchBytes = FQ_STATIC_SCRATCH_BYTES;

static __device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

constexpr int kMaxDevices = 64;

// Device address of g_static_scratch on the current device, looked up once per device (the
// symbol's host-side name is not a device address and must never be passed to a kernel).
cudaError_t scratch_for_current_device(void** out) {
  static std::mutex mu;
  static void* addr[kMaxDevices] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> g(mu);
  if (!addr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_static_scratch);
    if (e != cudaSuccess) return e;
    addr[dev] = p;
  }
  *out = addr[dev];
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
