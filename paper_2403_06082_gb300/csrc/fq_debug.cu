// FQ_FP32_DEBUG path: the three products of the layer in fp32 on CUDA cores, with z and u kept
// in fp32.  It exists to check the layer's semantics to ~1e-5 against the fp64 oracle; it is
// not tuned.  Each output element is one warp's dot product: lane l sums the terms k = l mod 32
// and a butterfly over the 32 lanes combines them, which keeps fp32 rounding near
// eps * sqrt(K / 32) instead of eps * sqrt(K).
#include "fq_device.cuh"
#include "fq_internal.h"

namespace fq {
namespace {

constexpr int kWarps = 8;   // rows per block (one warp per row)
constexpr int kTok = 8;     // tokens per warp

__device__ __forceinline__ float code_at(const uint32_t* __restrict__ words, int KB, int row,
                                         int col) {
  const int64_t widx = (static_cast<int64_t>(row / kRowTile) * KB + col / kColBlock) * 512 +
                       (row % kRowTile) * 4 + (col % kColBlock) / 16;
  const int c = col & 15;
  return static_cast<float>((__ldg(words + widx) >> (2 * (c >> 1) + 16 * (c & 1))) & 3u);
}

// out[m * R + i] = epilogue(sum_k A_i[k] * B[m * K + k]) for rows i < R, tokens m < M.
// CODES: A_i[k] is the 2-bit code q_ik and the epilogue is gamma_i (s_i acc + zero_i sum_k B).
template <bool CODES>
__global__ void __launch_bounds__(kWarps * 32) rowdot_kernel(
    const float* __restrict__ A, const uint32_t* __restrict__ words, int KB, int R, int K,
    const float* __restrict__ B, int M, float* __restrict__ out,
    const __half* __restrict__ scale, const __half* __restrict__ zero,
    const float* __restrict__ gamma) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int i = blockIdx.x * kWarps + warp;
  if (i >= R) return;
  const int m0 = blockIdx.y * kTok;
  const int nt = min(kTok, M - m0);
  float acc[kTok], zs[kTok];
#pragma unroll
  for (int t = 0; t < kTok; ++t) acc[t] = zs[t] = 0.f;
  const float* Ai = CODES ? nullptr : A + static_cast<int64_t>(i) * K;
  for (int k = lane; k < K; k += 32) {
    const float a = CODES ? code_at(words, KB, i, k) : __ldg(Ai + k);
#pragma unroll
    for (int t = 0; t < kTok; ++t) {
      if (t < nt) {
        const float b = __ldg(B + static_cast<int64_t>(m0 + t) * K + k);
        acc[t] = fmaf(a, b, acc[t]);
        if (CODES) zs[t] += b;
      }
    }
  }
#pragma unroll
  for (int t = 0; t < kTok; ++t) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      acc[t] += __shfl_xor_sync(0xffffffffu, acc[t], off);
      if (CODES) zs[t] += __shfl_xor_sync(0xffffffffu, zs[t], off);
    }
  }
  if (lane < nt) {
    float v = 0.f;
#pragma unroll
    for (int t = 0; t < kTok; ++t)
      if (t == lane) {
        v = acc[t];
        if (CODES) {
          v = __half2float(scale[i]) * v + __half2float(zero[i]) * zs[t];
          if (gamma) v *= gamma[i];
        }
      }
    out[static_cast<int64_t>(m0 + lane) * R + i] = v;
  }
}

}  // namespace

size_t debug_workspace_bytes(int M, int n_in, int n_out) {
  return kWsHeader + round_up(static_cast<int64_t>(M) * n_in * 4, 256) +
         round_up(static_cast<int64_t>(M) * n_out * 4, 256);
}

cudaError_t launch_debug_forward(const float* x, int M, int d_in, const float* T_in,
                                 const fq_packed& C, const float* T_out_t, int d_out,
                                 const float* gamma, float* y, char* ws, cudaStream_t s) {
  const int n_in = C.n_in, n_out = C.n_out;
  float* z = reinterpret_cast<float*>(ws + kWsHeader);
  float* u = reinterpret_cast<float*>(ws + kWsHeader +
                                      round_up(static_cast<int64_t>(M) * n_in * 4, 256));
  const int KB = static_cast<int>(ceil_div(n_in, kColBlock));
  const dim3 block(kWarps * 32);
  const unsigned gy = static_cast<unsigned>(ceil_div(M, kTok));
  // analysis: z = T_in x
  rowdot_kernel<false><<<dim3(static_cast<unsigned>(ceil_div(n_in, kWarps)), gy), block, 0, s>>>(
      T_in, nullptr, 0, n_in, d_in, x, M, z, nullptr, nullptr, nullptr);
  // frame-coefficient product with dequantization and optional gain
  rowdot_kernel<true><<<dim3(static_cast<unsigned>(ceil_div(n_out, kWarps)), gy), block, 0, s>>>(
      nullptr, C.words, KB, n_out, n_in, z, M, u, reinterpret_cast<const __half*>(C.scale_f16),
      reinterpret_cast<const __half*>(C.zero_f16), gamma);
  // synthesis: y = T_out^T u
  rowdot_kernel<false><<<dim3(static_cast<unsigned>(ceil_div(d_out, kWarps)), gy), block, 0, s>>>(
      T_out_t, nullptr, 0, d_out, n_out, u, M, y, nullptr, nullptr, nullptr);
  return cudaGetLastError();
}

}  // namespace fq
