// FQ_FP32_DEBUG path: the three products of the layer in fp32 on CUDA cores, with z and u kept
// in fp32.  It exists to check the layer's semantics to ~1e-5 against the fp64 oracle at every
// workload size (up to 12608 tokens on the ViT MLP), so it is a plain tiled SIMT product rather
// than a tuned one: a block computes a 64-row x 64-token tile of out = A B^T, staging 32-wide K
// slices of both operands in shared memory, each thread a 4 x 4 sub-tile.  Rounding: each
// thread sums every 32-wide K slice into a fresh partial before adding it to its running total,
// so the fp32 error grows like eps * (sqrt(32) + sqrt(K / 32)) rather than eps * sqrt(K).
#include "fq_device.cuh"
#include "fq_internal.h"

namespace fq {
namespace {

constexpr int kTileR = 64;   // output rows per block
constexpr int kTileM = 64;   // tokens per block
constexpr int kTileK = 32;   // K slice staged in shared memory
constexpr int kThreads = 256;

__device__ __forceinline__ float code_at(const uint32_t* __restrict__ words, int KB, int row,
                                         int col) {
  const int64_t widx = (static_cast<int64_t>(row / kRowTile) * KB + col / kColBlock) * 512 +
                       (row % kRowTile) * 4 + (col % kColBlock) / 16;
  const int c = col & 15;
  return static_cast<float>((__ldg(words + widx) >> (2 * (c >> 1) + 16 * (c & 1))) & 3u);
}

// out[m * R + i] = epilogue(sum_k A_i[k] * B[m * K + k]) for rows i < R, tokens m < M.
// CODES: A_i[k] is the 2-bit code q_ik and the epilogue is gamma_i (s_i acc + zero_i zsum[m]).
template <bool CODES>
__global__ void __launch_bounds__(kThreads) debug_gemm_kernel(
    const float* __restrict__ A, const uint32_t* __restrict__ words, int KB, int R, int K,
    const float* __restrict__ B, int M, float* __restrict__ out,
    const __half* __restrict__ scale, const __half* __restrict__ zero,
    const float* __restrict__ gamma, const float* __restrict__ zsum) {
  __shared__ float As[kTileK][kTileR + 1];
  __shared__ float Bs[kTileK][kTileM + 1];
  const int t = threadIdx.x;
  const int tx = t & 15, ty = t >> 4;             // token group, row group
  const int r0 = blockIdx.x * kTileR, m0 = blockIdx.y * kTileM;
  float total[4][4], part[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) total[i][j] = 0.f;
  for (int k0 = 0; k0 < K; k0 += kTileK) {
    // stage the slice: element e = t + 256 q is (row or token e / 32, k e % 32), so a warp reads
    // 32 consecutive k of one row (coalesced) and writes one column of the padded tile
#pragma unroll
    for (int q = 0; q < kTileR * kTileK / kThreads; ++q) {
      const int e = t + kThreads * q;
      const int r = e / kTileK, c = e % kTileK;
      const int row = r0 + r, k = k0 + c;
      float a = 0.f;
      if (row < R && k < K)
        a = CODES ? code_at(words, KB, row, k) : __ldg(A + static_cast<int64_t>(row) * K + k);
      As[c][r] = a;
      const int tok = m0 + r;
      Bs[c][r] = (tok < M && k < K) ? __ldg(B + static_cast<int64_t>(tok) * K + k) : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) part[i][j] = 0.f;
#pragma unroll 8
    for (int kk = 0; kk < kTileK; ++kk) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = As[kk][ty + 16 * i];
#pragma unroll
      for (int j = 0; j < 4; ++j) b[j] = Bs[kk][tx + 16 * j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) part[i][j] = fmaf(a[i], b[j], part[i][j]);
    }
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) total[i][j] += part[i][j];
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int row = r0 + ty + 16 * i;
    if (row >= R) continue;
    float s_i = 0.f, z_i = 0.f, g_i = 1.f;
    if (CODES) {
      s_i = __half2float(scale[row]);
      z_i = __half2float(zero[row]);
      if (gamma) g_i = gamma[row];
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int tok = m0 + tx + 16 * j;
      if (tok >= M) continue;
      float v = total[i][j];
      if (CODES) v = g_i * (s_i * v + z_i * zsum[tok]);
      out[static_cast<int64_t>(tok) * R + row] = v;
    }
  }
}

// zsum[m] = sum_k z[m * K + k]: one warp per token, lane l sums k = l mod 32, then a butterfly.
__global__ void __launch_bounds__(kThreads) row_sum_kernel(const float* __restrict__ z, int M,
                                                           int K, float* __restrict__ zsum) {
  const int m = blockIdx.x * (kThreads / 32) + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (m >= M) return;
  float s = 0.f;
  for (int k = lane; k < K; k += 32) s += __ldg(z + static_cast<int64_t>(m) * K + k);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
  if (lane == 0) zsum[m] = s;
}

struct DebugWs {
  size_t z, u, zsum, total;
};

DebugWs debug_ws(int M, int n_in, int n_out) {
  DebugWs L{};
  size_t off = kWsHeader;
  L.z = off;
  off += round_up(static_cast<int64_t>(M) * n_in * 4, 256);
  L.u = off;
  off += round_up(static_cast<int64_t>(M) * n_out * 4, 256);
  L.zsum = off;
  off += round_up(static_cast<int64_t>(M) * 4, 256);
  L.total = off;
  return L;
}

}  // namespace

size_t debug_workspace_bytes(int M, int n_in, int n_out) {
  return debug_ws(M, n_in, n_out).total;
}

cudaError_t launch_debug_forward(const float* x, int M, int d_in, const float* T_in,
                                 const fq_packed& C, const float* T_out_t, int d_out,
                                 const float* gamma, float* y, char* ws, cudaStream_t s) {
  const int n_in = C.n_in, n_out = C.n_out;
  const DebugWs L = debug_ws(M, n_in, n_out);
  float* z = reinterpret_cast<float*>(ws + L.z);
  float* u = reinterpret_cast<float*>(ws + L.u);
  float* zsum = reinterpret_cast<float*>(ws + L.zsum);
  const int KB = static_cast<int>(ceil_div(n_in, kColBlock));
  const dim3 block(kThreads);
  const unsigned gm = static_cast<unsigned>(ceil_div(M, kTileM));
  auto grid = [&](int R) { return dim3(static_cast<unsigned>(ceil_div(R, kTileR)), gm); };
  // analysis: z = T_in x
  debug_gemm_kernel<false><<<grid(n_in), block, 0, s>>>(T_in, nullptr, 0, n_in, d_in, x, M, z,
                                                         nullptr, nullptr, nullptr, nullptr);
  // sum of z per token, for the zero term of the dequantized product
  row_sum_kernel<<<static_cast<unsigned>(ceil_div(M, kThreads / 32)), block, 0, s>>>(z, M, n_in,
                                                                                     zsum);
  // frame-coefficient product with dequantization and optional gain
  debug_gemm_kernel<true><<<grid(n_out), block, 0, s>>>(
      nullptr, C.words, KB, n_out, n_in, z, M, u,
      reinterpret_cast<const __half*>(C.scale_f16), reinterpret_cast<const __half*>(C.zero_f16),
      gamma, zsum);
  // synthesis: y = T_out^T u
  debug_gemm_kernel<false><<<grid(d_out), block, 0, s>>>(T_out_t, nullptr, 0, d_out, n_out, u, M,
                                                         y, nullptr, nullptr, nullptr, nullptr);
  return cudaGetLastError();
}

}  // namespace fq
