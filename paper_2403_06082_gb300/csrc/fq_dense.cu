// Weight reconstruction (include/framequant_dense.h): W_hat = T_out^T diag(gamma) C_hat T_in
// as the FQ_BF16 forward of the d_in unit vectors, then a transpose.  The forward of unit
// vector e_j is column j of W_hat, so the d_in x d_out output of the forward is W_hat^T.  The
// analysis of e_j is column j of T_in, exact in bf16, so the chain starts from that transpose
// and runs only the code product and the synthesis on the tensor cores.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>

#include "fq_internal.h"
#include "framequant_dense.h"

namespace fq {
namespace {

// out (cols x rows) = in (rows x cols)^T through 32 x 32 shared-memory tiles
__global__ void transpose_bf16_kernel(const __nv_bfloat16* __restrict__ in,
                                      __nv_bfloat16* __restrict__ out, int rows, int cols) {
  __shared__ __nv_bfloat16 tile[32][34];
  const int c0 = blockIdx.x * 32, r0 = blockIdx.y * 32;
  for (int dy = threadIdx.y; dy < 32; dy += 8) {
    const int r = r0 + dy, c = c0 + threadIdx.x;
    if (r < rows && c < cols) tile[dy][threadIdx.x] = in[static_cast<int64_t>(r) * cols + c];
  }
  __syncthreads();
  for (int dy = threadIdx.y; dy < 32; dy += 8) {
    const int c = c0 + dy, r = r0 + threadIdx.x;
    if (c < cols && r < rows) out[static_cast<int64_t>(c) * rows + r] = tile[threadIdx.x][dy];
  }
}

struct RecWs {
  size_t fwd_bytes, yt, total;
};

// the tensor-core chain's workspace for M = d_in tokens, then the d_in x d_out output
RecWs rec_ws(int d_in, int n_in, int n_out, int d_out) {
  RecWs L{};
  L.fwd_bytes = static_cast<size_t>(
      round_up(static_cast<int64_t>(tc_workspace_bytes(d_in, d_in, n_in, n_out, d_out, 0)), 256));
  size_t off = L.fwd_bytes;
  L.yt = off;
  off += static_cast<size_t>(round_up(static_cast<int64_t>(d_in) * d_out * 2, 256));
  L.total = off;
  return L;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace
}  // namespace fq

using namespace fq;

extern "C" {

size_t fq_reconstruct_workspace_bytes(int d_in, int n_in, int n_out, int d_out) {
  if (d_in <= 0 || n_in <= 0 || n_out <= 0 || d_out <= 0) return 0;
  return rec_ws(d_in, n_in, n_out, d_out).total;
}

fq_status fq_reconstruct_weight(const void* T_in, const fq_packed* C, const void* T_out_t,
                                int d_in, int d_out, const float* gamma, void* W_hat, void* ws,
                                size_t ws_bytes, fq_stream_t stream) {
  if (!T_in || !C || !T_out_t || !W_hat || d_in <= 0 || d_out <= 0) return FQ_ERR_INVALID_ARG;
  // the checks of the forward this call makes, before anything is launched
  if (const fq_status cs = check_packed(C)) return cs;
  if (d_in % 8 || d_out % 8 || !aligned16(W_hat) || !aligned16(T_in) || !aligned16(T_out_t) ||
      (gamma && !aligned16(gamma)))
    return FQ_ERR_ALIGNMENT;
  if (!ws) return FQ_ERR_WORKSPACE;
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return FQ_ERR_ALIGNMENT;
  if (ws_bytes < fq_reconstruct_workspace_bytes(d_in, C->n_in, C->n_out, d_out))
    return FQ_ERR_WORKSPACE;
  {
    int dev = 0, major = 0, minor = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess)
      return FQ_ERR_CUDA;
    if (major * 10 + minor != 103) return FQ_ERR_UNSUPPORTED;
  }
  const RecWs L = rec_ws(d_in, C->n_in, C->n_out, d_out);
  auto s = reinterpret_cast<cudaStream_t>(stream);
  char* w = static_cast<char*>(ws);
  auto* Yt = reinterpret_cast<__nv_bfloat16*>(w + L.yt);
  // every check of the chain passed above (sizes, alignment, workspace, device)
  const fq_status st =
      launch_tc_unit_forward(T_in, d_in, *C, T_out_t, d_out, gamma, Yt, w, L.fwd_bytes, s);
  if (st != FQ_OK) return st;
  transpose_bf16_kernel<<<dim3(static_cast<unsigned>(ceil_div(d_out, 32)),
                               static_cast<unsigned>(ceil_div(d_in, 32))),
                          dim3(32, 8), 0, s>>>(Yt, static_cast<__nv_bfloat16*>(W_hat), d_in,
                                               d_out);
  return cudaGetLastError() == cudaSuccess ? FQ_OK : FQ_ERR_CUDA;
}

}  // extern "C"
