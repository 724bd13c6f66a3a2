// Frame-domain GPTQ on the GPU (Algorithm 1, steps 2-4): the offline quantizer that turns the
// frame coefficients C = T_out W T_in^T into 2-bit codes while keeping the proxy loss
//     L(D_hat) = ||D C_prev - D_hat C_prev||_F^2 = tr((D - D_hat) H (D - D_hat)^T),
//     H = C_prev C_prev^T,   C_prev = T_in A_prev (calibration tokens in the frame domain)
// small (Sec. 3).  Everything runs in fp64: it is an offline step whose integer decisions
// (which level each coefficient rounds to, with the rounding errors of earlier columns fed into
// later ones) should not depend on the arithmetic's precision.
//
// Steps, in the order of the method:
//   1. optional clip of D to [mu - 2 sigma, mu + 2 sigma], mu and sigma over all of D;
//   2. each row's 2-bit grid, fixed before the iteration: zero = fp16(min), scale =
//      fp16((max - min) / 3) (1 when 0), and the diagonal de-noising gain P / (P + scale^2 / 12);
//   3. the damped Hessian H + damp mean(diag H) I and the upper factor U of its inverse,
//      H^-1 = U^T U.  With J the exchange matrix, J H J = L L^T (lower Cholesky) gives
//      H = (J L J)(J L J)^T, so U = (J L J)^-1 = J L^-1 J: one Cholesky and one triangular
//      inverse, no explicit inverse of H;
//   4. the columns in blocks of 128: column j of a block is rounded to each row's grid, its
//      rounding error e = (w_j - q_hat_j) / U_jj is spread over the block's later columns
//      (w_k -= e U_jk), and after the block over all later columns at once (a product with
//      U's block rows).
// W is held transposed (column j of every row contiguous) so that one thread per row reads and
// writes coalesced.  Inside a block the update is one rounded multiply and one rounded subtract,
// as the plain recursion writes it.
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <algorithm>

#include "fq_device.cuh"
#include "fq_internal.h"

namespace fq {
namespace {

constexpr int kBlockCols = 128;   // columns per block of the iteration
constexpr int kT = 256;           // threads per block of the simple kernels

// ---- fp64 tiled product: C[m][n] (+)= sum_k A(m, k) B(k, n), A and B given by element strides.
constexpr int kGM = 64, kGN = 64, kGK = 16;

__global__ void __launch_bounds__(256) gemm_f64_kernel(
    const double* __restrict__ A, int64_t a_m, int64_t a_k, const double* __restrict__ B,
    int64_t b_k, int64_t b_n, double* __restrict__ C, int64_t ldc, int M, int N, int K,
    int subtract) {
  __shared__ double As[kGK][kGM + 1];
  __shared__ double Bs[kGK][kGN + 1];
  const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
  const int m0 = blockIdx.y * kGM, n0 = blockIdx.x * kGN;
  double acc[4][4] = {};
  for (int k0 = 0; k0 < K; k0 += kGK) {
    for (int t = threadIdx.x; t < kGM * kGK; t += 256) {
      // A: m fastest within a k row of the tile; B: n fastest
      const int r = t % kGM, kk = t / kGM;
      const int gm = m0 + r, gk = k0 + kk, gn = n0 + r;
      As[kk][r] = (gm < M && gk < K) ? A[gm * a_m + gk * a_k] : 0.0;
      Bs[kk][r] = (gn < N && gk < K) ? B[gk * b_k + gn * b_n] : 0.0;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < kGK; ++kk) {
      double a[4], b[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) a[q] = As[kk][ty + 16 * q], b[q] = Bs[kk][tx + 16 * q];
#pragma unroll
      for (int p = 0; p < 4; ++p)
#pragma unroll
        for (int q = 0; q < 4; ++q) acc[p][q] = fma(a[p], b[q], acc[p][q]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int p = 0; p < 4; ++p)
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int gm = m0 + ty + 16 * p, gn = n0 + tx + 16 * q;
      if (gm < M && gn < N) {
        double* c = C + gm * ldc + gn;
        *c = subtract ? *c - acc[p][q] : acc[p][q];
      }
    }
}

cudaError_t gemm_f64(const double* A, int64_t a_m, int64_t a_k, const double* B, int64_t b_k,
                     int64_t b_n, double* C, int64_t ldc, int M, int N, int K, bool subtract,
                     cudaStream_t s) {
  if (M <= 0 || N <= 0) return cudaSuccess;
  const dim3 grid(static_cast<unsigned>(ceil_div(N, kGN)), static_cast<unsigned>(ceil_div(M, kGM)));
  gemm_f64_kernel<<<grid, 256, 0, s>>>(A, a_m, a_k, B, b_k, b_n, C, ldc, M, N, K,
                                       subtract ? 1 : 0);
  return cudaGetLastError();
}

// ---- mean and standard deviation over all of D, two passes, fixed order: kParts blocks sum
// grid-strided shares, then one block adds the partial sums in order.
constexpr int kParts = 512;

__global__ void __launch_bounds__(kT) partial_sum_kernel(const double* __restrict__ D, int64_t n,
                                                         const double* __restrict__ mom,
                                                         int deviations,
                                                         double* __restrict__ part) {
  __shared__ double red[kT];
  const double mu = deviations ? mom[0] : 0.0;
  double s = 0.0;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(kT) + threadIdx.x; i < n;
       i += static_cast<int64_t>(kParts) * kT) {
    const double d = D[i] - mu;
    s += deviations ? d * d : D[i];
  }
  red[threadIdx.x] = s;
  __syncthreads();
  for (int w = kT / 2; w > 0; w >>= 1) {
    if (threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) part[blockIdx.x] = red[0];
}

// mom[0] = sum / n (first pass), mom[1] = sqrt(sum / n) (second pass)
__global__ void __launch_bounds__(kT) final_sum_kernel(const double* __restrict__ part, int64_t n,
                                                       int second, double* __restrict__ mom) {
  __shared__ double red[kT];
  double s = 0.0;
  for (int i = threadIdx.x; i < kParts; i += kT) s += part[i];
  red[threadIdx.x] = s;
  __syncthreads();
  for (int w = kT / 2; w > 0; w >>= 1) {
    if (threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    const double m = red[0] / static_cast<double>(n);
    mom[second] = second ? sqrt(m) : m;
  }
}

// WT[j][i] = clip(D[i][j]) (or D[i][j]): the working copy, transposed
__global__ void clip_transpose_kernel(const double* __restrict__ D, int n_out, int n_in,
                                      const double* __restrict__ mom, int clip,
                                      double* __restrict__ WT) {
  __shared__ double tile[32][33];
  const int c0 = blockIdx.x * 32, r0 = blockIdx.y * 32;
  double lo = -INFINITY, hi = INFINITY;
  if (clip) {
    lo = mom[0] - 2.0 * mom[1];
    hi = mom[0] + 2.0 * mom[1];
  }
  for (int dy = threadIdx.y; dy < 32; dy += 8) {
    const int r = r0 + dy, c = c0 + threadIdx.x;
    if (r < n_out && c < n_in) tile[dy][threadIdx.x] = fmin(fmax(D[static_cast<int64_t>(r) * n_in + c], lo), hi);
  }
  __syncthreads();
  for (int dy = threadIdx.y; dy < 32; dy += 8) {
    const int c = c0 + dy, r = r0 + threadIdx.x;
    if (c < n_in && r < n_out) WT[static_cast<int64_t>(c) * n_out + r] = tile[threadIdx.x][dy];
  }
}

// One block per row i (reading column i of WT): min, max, mean square -> fp16 zero and scale,
// the de-noising gain.
__global__ void __launch_bounds__(kT) row_grid_kernel(const double* __restrict__ WT, int n_out,
                                                      int n_in, __half* __restrict__ scale,
                                                      __half* __restrict__ zero,
                                                      double* __restrict__ s64,
                                                      double* __restrict__ z64,
                                                      float* __restrict__ gamma) {
  const int i = blockIdx.x;
  __shared__ double smn[kT], smx[kT], ssq[kT];
  double mn = INFINITY, mx = -INFINITY, sq = 0.0;
  for (int j = threadIdx.x; j < n_in; j += kT) {
    const double v = WT[static_cast<int64_t>(j) * n_out + i];
    mn = fmin(mn, v);
    mx = fmax(mx, v);
    sq += v * v;
  }
  smn[threadIdx.x] = mn;
  smx[threadIdx.x] = mx;
  ssq[threadIdx.x] = sq;
  __syncthreads();
  for (int w = kT / 2; w > 0; w >>= 1) {
    if (threadIdx.x < w) {
      smn[threadIdx.x] = fmin(smn[threadIdx.x], smn[threadIdx.x + w]);
      smx[threadIdx.x] = fmax(smx[threadIdx.x], smx[threadIdx.x + w]);
      ssq[threadIdx.x] += ssq[threadIdx.x + w];
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    const __half hz = __double2half(smn[0]);
    __half hs = __double2half((smx[0] - smn[0]) / 3.0);
    if (__half2float(hs) == 0.f) hs = __float2half(1.f);
    zero[i] = hz;
    scale[i] = hs;
    const double sc = static_cast<double>(__half2float(hs));
    s64[i] = sc;
    z64[i] = static_cast<double>(__half2float(hz));
    if (gamma) {
      const double P = ssq[0] / n_in;
      gamma[i] = static_cast<float>(P / (P + sc * sc / 12.0));
    }
  }
}

// K = J (H + damp mean(diag H) I) J, lower triangle used
__global__ void damp_reverse_kernel(const double* __restrict__ H, int n, double damp,
                                    double* __restrict__ K) {
  __shared__ double red[kT];
  double s = 0.0;
  for (int i = threadIdx.x; i < n; i += kT) s += H[static_cast<int64_t>(i) * n + i];
  red[threadIdx.x] = s;
  __syncthreads();
  for (int w = kT / 2; w > 0; w >>= 1) {
    if (threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
    __syncthreads();
  }
  const double add = damp * (red[0] / n);
  const int64_t total = static_cast<int64_t>(n) * n;
  for (int64_t e = blockIdx.x * static_cast<int64_t>(kT) + threadIdx.x; e < total;
       e += static_cast<int64_t>(gridDim.x) * kT) {
    const int i = static_cast<int>(e / n), j = static_cast<int>(e % n);
    double v = H[static_cast<int64_t>(n - 1 - i) * n + (n - 1 - j)];
    if (i == j) v += add;
    K[e] = v;
  }
}

// Right-looking Cholesky, step j: K[i][k] -= K[i][j] K[k][j] / K[j][j] for j < k <= i.  The
// columns are scaled at the end (L[i][j] = K[i][j] / sqrt(K[j][j])).
__global__ void chol_step_kernel(double* __restrict__ K, int n, int j) {
  const int k = j + 1 + blockIdx.x * 16 + threadIdx.x;
  const int i = j + 1 + blockIdx.y * 16 + threadIdx.y;
  if (k >= n || i >= n || k > i) return;
  const double piv = K[static_cast<int64_t>(j) * n + j];
  K[static_cast<int64_t>(i) * n + k] -=
      K[static_cast<int64_t>(i) * n + j] * K[static_cast<int64_t>(k) * n + j] / piv;
}

// L[i][j] = K[i][j] / sqrt(K[j][j]) below the diagonal (the diagonal itself is replaced by the
// next kernel, so every pivot is read here unchanged); a pivot that is not positive means the
// damped H was not positive definite
__global__ void chol_scale_kernel(double* __restrict__ K, int n, int32_t* __restrict__ status) {
  const int64_t total = static_cast<int64_t>(n) * n;
  for (int64_t e = blockIdx.x * static_cast<int64_t>(kT) + threadIdx.x; e < total;
       e += static_cast<int64_t>(gridDim.x) * kT) {
    const int i = static_cast<int>(e / n), j = static_cast<int>(e % n);
    const double piv = K[static_cast<int64_t>(j) * n + j];
    if (i == j && !(piv > 0.0)) report(status, FQ_ERR_DEVICE_CHECK);
    if (j < i) K[e] = K[e] / sqrt(piv);
  }
}

__global__ void chol_diag_kernel(double* __restrict__ K, int n) {
  for (int j = blockIdx.x * kT + threadIdx.x; j < n; j += gridDim.x * kT)
    K[static_cast<int64_t>(j) * n + j] = sqrt(K[static_cast<int64_t>(j) * n + j]);
}

// X = L^-1 (lower), one block per column c: x_c = 1 / L_cc, x_i = -(sum_{c<=k<i} L_ik x_k) / L_ii.
// Written straight into U = J X J: U[n-1-i][n-1-c] = X[i][c].
__global__ void __launch_bounds__(kT) tri_inverse_kernel(const double* __restrict__ L, int n,
                                                         double* __restrict__ U) {
  extern __shared__ double xs[];                 // x_c .. x_{n-1}
  __shared__ double red[kT];
  const int c = blockIdx.x;
  if (threadIdx.x == 0) xs[0] = 1.0 / L[static_cast<int64_t>(c) * n + c];
  __syncthreads();
  for (int i = c + 1; i < n; ++i) {
    const double* Li = L + static_cast<int64_t>(i) * n;
    double s = 0.0;
    for (int k = c + threadIdx.x; k < i; k += kT) s += Li[k] * xs[k - c];
    red[threadIdx.x] = s;
    __syncthreads();
    for (int w = kT / 2; w > 0; w >>= 1) {
      if (threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
      __syncthreads();
    }
    if (threadIdx.x == 0) xs[i - c] = -red[0] / Li[i];
    __syncthreads();
  }
  for (int i = threadIdx.x; i < n; i += kT) {
    const double x = i < c ? 0.0 : xs[i - c];
    U[static_cast<int64_t>(n - 1 - i) * n + (n - 1 - c)] = x;
  }
}

// Block b0 .. b1-1 of the iteration, one thread per row i of W (WT column i).
__global__ void __launch_bounds__(kT) gptq_block_kernel(double* __restrict__ WT, int n_out,
                                                        int n_in, const double* __restrict__ U,
                                                        const double* __restrict__ s64,
                                                        const double* __restrict__ z64, int b0,
                                                        int b1, uint8_t* __restrict__ codesT,
                                                        double* __restrict__ ET) {
  const int i = blockIdx.x * kT + threadIdx.x;
  if (i >= n_out) return;
  const double s = s64[i], z = z64[i];
  for (int j = b0; j < b1; ++j) {
    const double w = WT[static_cast<int64_t>(j) * n_out + i];
    const double q = fmin(fmax(rint((w - z) / s), 0.0), 3.0);
    codesT[static_cast<int64_t>(j) * n_out + i] = static_cast<uint8_t>(q);
    const double* Uj = U + static_cast<int64_t>(j) * n_in;
    const double e = (w - __dadd_rn(__dmul_rn(s, q), z)) / Uj[j];
    ET[static_cast<int64_t>(j - b0) * n_out + i] = e;
    for (int k = j + 1; k < b1; ++k) {
      double* wk = WT + static_cast<int64_t>(k) * n_out + i;
      *wk = __dsub_rn(*wk, __dmul_rn(e, Uj[k]));
    }
  }
}

// codes[i][j] = codesT[j][i]
__global__ void transpose_u8_kernel(const uint8_t* __restrict__ in, int rows, int cols,
                                    uint8_t* __restrict__ out) {
  __shared__ uint8_t tile[32][33];
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

struct GptqWs {
  size_t status, mom, part, s64, z64, WT, K, U, ET, codesT, total;
};

GptqWs gptq_ws(int n_out, int n_in) {
  GptqWs L{};
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t at = off;
    off += round_up(static_cast<int64_t>(bytes), 256);
    return at;
  };
  L.status = take(4);
  L.mom = take(2 * 8);
  L.part = take(kParts * 8);
  L.s64 = take(static_cast<size_t>(n_out) * 8);
  L.z64 = take(static_cast<size_t>(n_out) * 8);
  L.WT = take(static_cast<size_t>(n_out) * n_in * 8);
  L.K = take(static_cast<size_t>(n_in) * n_in * 8);
  L.U = take(static_cast<size_t>(n_in) * n_in * 8);
  L.ET = take(static_cast<size_t>(n_out) * kBlockCols * 8);
  L.codesT = take(static_cast<size_t>(n_out) * n_in);
  L.total = off;
  return L;
}

unsigned grid_cap(int64_t total) {
  return static_cast<unsigned>(std::max<int64_t>(1, std::min<int64_t>(ceil_div(total, kT), 4096)));
}

bool a8(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 7u) == 0; }

}  // namespace
}  // namespace fq

using namespace fq;

extern "C" {

fq_status fq_gptq_hessian(const double* Z, int N, int n_in, double* H, fq_stream_t stream) {
  if (!Z || !H || N <= 0 || n_in <= 0) return FQ_ERR_INVALID_ARG;
  if (!a8(Z) || !a8(H)) return FQ_ERR_ALIGNMENT;
  // H[i][j] = sum_t Z[t][i] Z[t][j]: A(i, t) = Z[t n_in + i], B(t, j) = Z[t n_in + j]
  return gemm_f64(Z, 1, n_in, Z, n_in, 1, H, n_in, n_in, n_in, N, false,
                  reinterpret_cast<cudaStream_t>(stream)) == cudaSuccess
             ? FQ_OK
             : FQ_ERR_CUDA;
}

size_t fq_gptq_workspace_bytes(int n_out, int n_in) {
  if (n_out <= 0 || n_in <= 0) return 0;
  return gptq_ws(n_out, n_in).total;
}

fq_status fq_quantize_gptq(const double* C, int n_out, int n_in, const double* H, double damp,
                           int clip, uint8_t* codes, uint16_t* scale, uint16_t* zero,
                           float* gamma, void* ws, size_t ws_bytes, fq_stream_t stream) {
  if (!C || !H || !codes || !scale || !zero || n_out <= 0 || n_in <= 0 || !(damp >= 0.0))
    return FQ_ERR_INVALID_ARG;
  if (!a8(C) || !a8(H) || (reinterpret_cast<uintptr_t>(scale) & 1u) ||
      (reinterpret_cast<uintptr_t>(zero) & 1u) || (gamma && (reinterpret_cast<uintptr_t>(gamma) & 3u)))
    return FQ_ERR_ALIGNMENT;
  if (!ws) return FQ_ERR_WORKSPACE;
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return FQ_ERR_ALIGNMENT;
  const GptqWs L = gptq_ws(n_out, n_in);
  if (ws_bytes < L.total) return FQ_ERR_WORKSPACE;
  auto s = reinterpret_cast<cudaStream_t>(stream);
  char* w = static_cast<char*>(ws);
  auto* status = reinterpret_cast<int32_t*>(w + L.status);
  auto* mom = reinterpret_cast<double*>(w + L.mom);
  auto* s64 = reinterpret_cast<double*>(w + L.s64);
  auto* z64 = reinterpret_cast<double*>(w + L.z64);
  auto* WT = reinterpret_cast<double*>(w + L.WT);
  auto* K = reinterpret_cast<double*>(w + L.K);
  auto* U = reinterpret_cast<double*>(w + L.U);
  auto* ET = reinterpret_cast<double*>(w + L.ET);
  auto* codesT = reinterpret_cast<uint8_t*>(w + L.codesT);
  const int64_t nD = static_cast<int64_t>(n_out) * n_in;
  const int64_t nH = static_cast<int64_t>(n_in) * n_in;
  if (cudaMemsetAsync(status, 0, 4, s) != cudaSuccess) return FQ_ERR_CUDA;
  // 1. clip (Algorithm 1, steps 2-3) into the transposed working copy
  auto* part = reinterpret_cast<double*>(w + L.part);
  if (clip) {
    partial_sum_kernel<<<kParts, kT, 0, s>>>(C, nD, mom, 0, part);
    final_sum_kernel<<<1, kT, 0, s>>>(part, nD, 0, mom);
    partial_sum_kernel<<<kParts, kT, 0, s>>>(C, nD, mom, 1, part);
    final_sum_kernel<<<1, kT, 0, s>>>(part, nD, 1, mom);
  }
  clip_transpose_kernel<<<dim3(static_cast<unsigned>(ceil_div(n_in, 32)),
                               static_cast<unsigned>(ceil_div(n_out, 32))),
                          dim3(32, 8), 0, s>>>(C, n_out, n_in, mom, clip, WT);
  // 2. each row's grid and gain
  row_grid_kernel<<<static_cast<unsigned>(n_out), kT, 0, s>>>(
      WT, n_out, n_in, reinterpret_cast<__half*>(scale), reinterpret_cast<__half*>(zero), s64,
      z64, gamma);
  // 3. U with H^-1 = U^T U
  damp_reverse_kernel<<<grid_cap(nH), kT, 0, s>>>(H, n_in, damp, K);
  for (int j = 0; j + 1 < n_in; ++j) {
    const int t = n_in - j - 1;
    const dim3 g(static_cast<unsigned>(ceil_div(t, 16)), static_cast<unsigned>(ceil_div(t, 16)));
    chol_step_kernel<<<g, dim3(16, 16), 0, s>>>(K, n_in, j);
  }
  chol_scale_kernel<<<grid_cap(nH), kT, 0, s>>>(K, n_in, status);
  chol_diag_kernel<<<grid_cap(n_in), kT, 0, s>>>(K, n_in);
  const size_t xs_bytes = static_cast<size_t>(n_in) * 8;
  if (xs_bytes > 200 * 1024) return FQ_ERR_UNSUPPORTED;
  if (xs_bytes > 48 * 1024 &&
      cudaFuncSetAttribute(tri_inverse_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(xs_bytes)) != cudaSuccess)
    return FQ_ERR_CUDA;
  tri_inverse_kernel<<<static_cast<unsigned>(n_in), kT, xs_bytes, s>>>(K, n_in, U);
  // 4. the columns, block by block
  for (int b0 = 0; b0 < n_in; b0 += kBlockCols) {
    const int b1 = std::min(n_in, b0 + kBlockCols);
    gptq_block_kernel<<<static_cast<unsigned>(ceil_div(n_out, kT)), kT, 0, s>>>(
        WT, n_out, n_in, U, s64, z64, b0, b1, codesT, ET);
    // WT[k][i] -= sum_jj U[b0 + jj][k] ET[jj][i] for k >= b1
    if (b1 < n_in &&
        gemm_f64(U + static_cast<int64_t>(b0) * n_in + b1, 1, n_in, ET, n_out, 1,
                 WT + static_cast<int64_t>(b1) * n_out, n_out, n_in - b1, n_out, b1 - b0, true,
                 s) != cudaSuccess)
      return FQ_ERR_CUDA;
  }
  transpose_u8_kernel<<<dim3(static_cast<unsigned>(ceil_div(n_out, 32)),
                             static_cast<unsigned>(ceil_div(n_in, 32))),
                        dim3(32, 8), 0, s>>>(codesT, n_in, n_out, codes);
  if (cudaGetLastError() != cudaSuccess) return FQ_ERR_CUDA;
  // the status word reports a Hessian that was not positive definite after damping
  int32_t st = 0;
  if (cudaMemcpyAsync(&st, status, 4, cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return FQ_ERR_CUDA;
  return st ? FQ_ERR_DEVICE_CHECK : FQ_OK;
}

}  // extern "C"
