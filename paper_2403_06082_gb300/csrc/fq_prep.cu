// Offline preparation of a frame-quantized layer on the GPU (not on the inference path):
//   fq_frame_build    the real (k, rho, d) tight fusion frame's analysis operator, optionally
//                     rotated (Sec. 2.2; Appendix J; Appendix K: P = R T)
//   fq_coefficients   C = T_out W T_in^T (Sec. 3, D_l = P_l^T Theta_l P_prev), fp32
//   fq_quantize_rtn   per-row 2-bit round-to-nearest with fp16 scale/zero and the diagonal
//                     de-noising gain (Algorithm 1 with RTN in place of GPTQ; Appendix I)
// Spectral tetris and the QR factorisations of the rotation's Gaussian draws are small and run
// on the host; everything of size n x d runs in the kernels below.
#include <cuda_fp16.h>

#include <cmath>
#include <cstring>
#include <vector>

#include "fq_device.cuh"
#include "fq_internal.h"

namespace fq {
namespace {

// ------------------------------------------------------------------ host: spectral tetris
// F (rho_c x d_c, row-major, double) with unit columns and orthogonal rows of squared norm
// d_c / rho_c, filled left to right: ones while a row lacks at least 1, then the remainder
// x in (0, 1) with the 2x2 block (1/sqrt2)[[sqrt x, sqrt x], [sqrt(2-x), -sqrt(2-x)]], which
// also gives the next row 2 - x.  Exact bookkeeping in units of 1/rho_c.
bool spectral_tetris(int rho_c, int d_c, std::vector<double>& F) {
  if (rho_c <= 0 || d_c < 2 * rho_c) return false;
  F.assign(static_cast<size_t>(rho_c) * d_c, 0.0);
  const int64_t target = d_c;            // squared row norm, in units of 1/rho_c
  const int64_t unit = rho_c;
  int64_t carried = 0;
  int col = 0;
  for (int j = 0; j < rho_c; ++j) {
    int64_t rem = target - carried;
    while (rem >= unit) {
      if (col >= d_c) return false;
      F[static_cast<size_t>(j) * d_c + col++] = 1.0;
      rem -= unit;
    }
    if (rem > 0) {
      if (j + 1 >= rho_c || col + 1 >= d_c) return false;
      const double x = static_cast<double>(rem) / unit;
      const double top = std::sqrt(x / 2.0), bot = std::sqrt((2.0 - x) / 2.0);
      F[static_cast<size_t>(j) * d_c + col] = top;
      F[static_cast<size_t>(j) * d_c + col + 1] = top;
      F[static_cast<size_t>(j + 1) * d_c + col] = bot;
      F[static_cast<size_t>(j + 1) * d_c + col + 1] = -bot;
      col += 2;
      carried = 2 * unit - rem;
    } else {
      carried = 0;
    }
  }
  return col == d_c;
}

// Modulation by k-th roots of unity gives a tight family exactly when distinct columns n, m of
// F with n = m (mod k) are orthogonal.
bool modulation_tight(const std::vector<double>& F, int rho_c, int d_c, int k) {
  for (int shift = k; shift < d_c; shift += k)
    for (int n = 0; n + shift < d_c; ++n) {
      double dot = 0.0;
      for (int j = 0; j < rho_c; ++j)
        dot += F[static_cast<size_t>(j) * d_c + n] * F[static_cast<size_t>(j) * d_c + n + shift];
      if (std::fabs(dot) > 1e-12) return false;
    }
  return true;
}

}  // namespace

// ------------------------------------------------------------------ host: Haar factor
// Q of the Householder QR of a square matrix G (row-major, a x a), with the columns signed so
// that R has a positive diagonal; Q is written row-major.
void haar_q(const double* G, int a, std::vector<double>& Q) {
  std::vector<double> A(G, G + static_cast<size_t>(a) * a);   // becomes R
  std::vector<double> V(static_cast<size_t>(a) * a, 0.0);     // Householder vectors (columns)
  std::vector<double> beta(a, 0.0);
  for (int j = 0; j < a; ++j) {
    double norm = 0.0;
    for (int i = j; i < a; ++i) norm += A[i * a + j] * A[i * a + j];
    norm = std::sqrt(norm);
    const double x0 = A[j * a + j];
    const double alpha = x0 >= 0 ? -norm : norm;
    double vnorm2 = 0.0;
    for (int i = j; i < a; ++i) {
      const double v = (i == j) ? x0 - alpha : A[i * a + j];
      V[i * a + j] = v;
      vnorm2 += v * v;
    }
    beta[j] = vnorm2 > 0 ? 2.0 / vnorm2 : 0.0;
    for (int c = j; c < a; ++c) {
      double s = 0.0;
      for (int i = j; i < a; ++i) s += V[i * a + j] * A[i * a + c];
      s *= beta[j];
      for (int i = j; i < a; ++i) A[i * a + c] -= s * V[i * a + j];
    }
  }
  // Q = H_0 H_1 ... H_{a-1}: apply to the identity from the last reflection back
  Q.assign(static_cast<size_t>(a) * a, 0.0);
  for (int i = 0; i < a; ++i) Q[i * a + i] = 1.0;
  for (int j = a - 1; j >= 0; --j)
    for (int c = 0; c < a; ++c) {
      double s = 0.0;
      for (int i = j; i < a; ++i) s += V[i * a + j] * Q[i * a + c];
      s *= beta[j];
      for (int i = j; i < a; ++i) Q[i * a + c] -= s * V[i * a + j];
    }
  for (int c = 0; c < a; ++c)
    if (A[c * a + c] < 0)
      for (int i = 0; i < a; ++i) Q[i * a + c] = -Q[i * a + c];
}

namespace {

// ------------------------------------------------------------------ device kernels
// Real analysis operator of the modulated, Parseval-normalised, realified frame.  Row
// 2 (j k + k_i) + e, column 2 c + f: with v = F[j][c] exp(2 pi i k_i c / k) / sqrt(k),
// (e, f) = (0,0): Re v, (0,1): Im v, (1,0): -Im v, (1,1): Re v.
__global__ void tff_fill_kernel(const double* __restrict__ F, int rho_c, int d_c, int k,
                                float* __restrict__ T, int64_t total) {
  const int64_t d = 2 * static_cast<int64_t>(d_c);
  for (int64_t idx = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; idx < total;
       idx += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t row = idx / d;
    const int col = static_cast<int>(idx % d);
    const int64_t b = row >> 1;
    const int e = static_cast<int>(row & 1), f = col & 1, c = col >> 1;
    const int j = static_cast<int>(b / k), ki = static_cast<int>(b % k);
    const double fv = F[static_cast<int64_t>(j) * d_c + c];
    float out = 0.f;
    if (fv != 0.0) {
      const int64_t m = (static_cast<int64_t>(ki) * c) % k;
      double s, co;
      sincospi(2.0 * static_cast<double>(m) / k, &s, &co);
      const double scale = fv / sqrt(static_cast<double>(k));
      const double re = co * scale, im = s * scale;
      const double v = (e == 0) ? (f == 0 ? re : im) : (f == 0 ? -im : re);
      out = static_cast<float>(v);
    }
    T[idx] = out;
  }
}

__global__ void eye_kernel(float* __restrict__ T, int d) {
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < d; i += gridDim.x * blockDim.x)
    T[static_cast<int64_t>(i) * d + i] = 1.f;
}

// C[i][j] = sum_k A[i][k] * B[j][k] (+ C if accumulate), fp32, both operands K-contiguous,
// batched over blockIdx.z with element strides. 64 x 64 tiles, 4 x 4 outputs per thread.
constexpr int kGT = 64, kGK = 16;
__global__ void __launch_bounds__(256) gemm_nt_f32(const float* __restrict__ A,
                                                   const float* __restrict__ B,
                                                   float* __restrict__ C, int64_t M, int N, int K,
                                                   int64_t sA, int64_t sB, int64_t sC) {
  __shared__ float As[kGK][kGT + 4];
  __shared__ float Bs[kGK][kGT + 4];
  A += blockIdx.z * sA;
  B += blockIdx.z * sB;
  C += blockIdx.z * sC;
  const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
  const int64_t i0 = static_cast<int64_t>(blockIdx.x) * kGT;
  const int j0 = blockIdx.y * kGT;
  float acc[4][4] = {};
  for (int k0 = 0; k0 < K; k0 += kGK) {
    for (int t = threadIdx.x; t < kGT * kGK; t += 256) {
      const int r = t / kGK, kk = t % kGK;
      const int64_t gi = i0 + r;
      const int gj = j0 + r, gk = k0 + kk;
      As[kk][r] = (gi < M && gk < K) ? A[static_cast<int64_t>(gi) * K + gk] : 0.f;
      Bs[kk][r] = (gj < N && gk < K) ? B[static_cast<int64_t>(gj) * K + gk] : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < kGK; ++kk) {
      float a[4], b[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) a[q] = As[kk][ty * 4 + q], b[q] = Bs[kk][tx * 4 + q];
#pragma unroll
      for (int p = 0; p < 4; ++p)
#pragma unroll
        for (int q = 0; q < 4; ++q) acc[p][q] = fmaf(a[p], b[q], acc[p][q]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int p = 0; p < 4; ++p)
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int64_t gi = i0 + ty * 4 + p;
      const int gj = j0 + tx * 4 + q;
      if (gi < M && gj < N) C[gi * N + gj] = acc[p][q];
    }
}

cudaError_t gemm_nt(const float* A, const float* B, float* C, int64_t M, int N, int K, int batch,
                    int64_t sA, int64_t sB, int64_t sC, cudaStream_t s) {
  dim3 grid(static_cast<unsigned>(ceil_div(M, kGT)), static_cast<unsigned>(ceil_div(N, kGT)),
            static_cast<unsigned>(batch));
  gemm_nt_f32<<<grid, 256, 0, s>>>(A, B, C, M, N, K, sA, sB, sC);
  return cudaGetLastError();
}

// X[row][p][q] = T[row][p b + q] * signs[p b + q]
__global__ void sign_kernel(const float* __restrict__ T, const float* __restrict__ signs,
                            float* __restrict__ X, int64_t total, int d) {
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < total;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x)
    X[i] = T[i] * signs[i % d];
}

// per row: Zt[row][q][p] = Z[row][p][q]  (Z is a x b)
__global__ void transpose_rows_kernel(const float* __restrict__ Z, float* __restrict__ Zt,
                                      int64_t total, int a, int b) {
  const int64_t d = static_cast<int64_t>(a) * b;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < total;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t row = i / d;
    const int r = static_cast<int>(i % d);
    const int q = r / a, p = r % a;
    Zt[i] = Z[row * d + static_cast<int64_t>(p) * b + q];
  }
}

// out[row][i] = Y[row].flat[perm[i]] with Y[row][p][q] stored transposed as Yt[row][q][p]
__global__ void permute_kernel(const float* __restrict__ Yt, const int* __restrict__ perm,
                               float* __restrict__ out, int64_t total, int a, int b) {
  const int64_t d = static_cast<int64_t>(a) * b;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < total;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t row = i / d;
    const int f = perm[i % d];
    const int p = f / b, q = f % b;
    out[i] = Yt[row * d + static_cast<int64_t>(q) * a + p];
  }
}

// One block per row: min/max, fp16 zero and scale, 2-bit codes, gain.
__global__ void __launch_bounds__(256) rtn_kernel(const float* __restrict__ C, int n_in,
                                                  uint8_t* __restrict__ codes,
                                                  __half* __restrict__ scale,
                                                  __half* __restrict__ zero,
                                                  float* __restrict__ gamma) {
  const int64_t row = blockIdx.x;
  const float* c = C + row * n_in;
  float mn = INFINITY, mx = -INFINITY;
  double sq = 0.0;
  for (int j = threadIdx.x; j < n_in; j += blockDim.x) {
    const float v = c[j];
    mn = fminf(mn, v);
    mx = fmaxf(mx, v);
    sq += static_cast<double>(v) * v;
  }
  __shared__ float smn[8], smx[8];
  __shared__ double ssq[8];
  __shared__ float s_scale, s_zero;
  for (int off = 16; off; off >>= 1) {
    mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, off));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
    sq += __shfl_xor_sync(0xffffffffu, sq, off);
  }
  const int w = threadIdx.x >> 5;
  if ((threadIdx.x & 31) == 0) smn[w] = mn, smx[w] = mx, ssq[w] = sq;
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int i = 1; i < static_cast<int>(blockDim.x >> 5); ++i) {
      mn = fminf(mn, smn[i]);
      mx = fmaxf(mx, smx[i]);
      sq += ssq[i];
    }
    const __half hz = __double2half(static_cast<double>(mn));
    __half hs = __double2half((static_cast<double>(mx) - mn) / 3.0);
    if (__half2float(hs) == 0.f) hs = __float2half(1.f);
    zero[row] = hz;
    scale[row] = hs;
    s_zero = __half2float(hz);
    s_scale = __half2float(hs);
    if (gamma) {
      const double P = sq / n_in;
      const double N = static_cast<double>(s_scale) * s_scale / 12.0;
      gamma[row] = static_cast<float>(P / (P + N));
    }
  }
  __syncthreads();
  const float zr = s_zero, sc = s_scale;
  for (int j = threadIdx.x; j < n_in; j += blockDim.x) {
    const float q = rintf((c[j] - zr) / sc);
    codes[row * n_in + j] = static_cast<uint8_t>(fminf(fmaxf(q, 0.f), 3.f));
  }
}

unsigned grid_for(int64_t total) {
  return static_cast<unsigned>(std::min<int64_t>(ceil_div(total, 256), 152 * 32));
}

}  // namespace
}  // namespace fq

using namespace fq;

extern "C" {

namespace {
struct FrameWs {
  size_t buf, F, Qa, Qb, signs, perm, total;
};
FrameWs frame_ws(int k, int rho, int d, int a, int b) {
  FrameWs L{};
  const int64_t n = static_cast<int64_t>(k) * rho;
  size_t off = 0;
  L.buf = off;
  off += round_up(2 * n * d * 4, 256);                                  // two n x d scratch
  L.F = off;
  off += round_up(static_cast<int64_t>(rho / 2) * (d / 2) * 8 + 8, 256);  // F (double)
  L.Qa = off;
  off += round_up(static_cast<int64_t>(a) * a * 4 + 4, 256);
  L.Qb = off;
  off += round_up(static_cast<int64_t>(b) * b * 4 + 4, 256);
  L.signs = off;
  off += round_up(static_cast<int64_t>(d) * 4, 256);
  L.perm = off;
  off += round_up(static_cast<int64_t>(d) * 4, 256);
  L.total = off;
  return L;
}
}  // namespace

size_t fq_frame_workspace_bytes(int k, int rho, int d, int a, int b) {
  if (k <= 0 || rho <= 0 || d <= 0 || a < 0 || b < 0) return 0;
  return frame_ws(k, rho, d, a, b).total;
}

fq_status fq_frame_build(int k, int rho, int d, const fq_rotation* rot, float* T, void* ws,
                         size_t ws_bytes, fq_stream_t stream) {
  if (!T || k <= 0 || rho <= 0 || d <= 0) return FQ_ERR_INVALID_ARG;
  auto s = reinterpret_cast<cudaStream_t>(stream);
  const int64_t n = static_cast<int64_t>(k) * rho;
  const int64_t total = n * d;
  std::vector<double> F;
  int rho_c = rho / 2, d_c = d / 2;
  if (k == 1 && rho == d) {          // the trivial (1, d, d) frame: the identity
    rho_c = d_c = 0;
  } else {
    if (rho % 2 || d % 2) return FQ_ERR_INVALID_ARG;
    if (!spectral_tetris(rho_c, d_c, F) || !modulation_tight(F, rho_c, d_c, k))
      return FQ_ERR_INVALID_ARG;
  }
  if (rot) {
    if (!rot->gauss_a || !rot->gauss_b || !rot->perm || !rot->signs || rot->a <= 0 ||
        rot->b <= 0 || static_cast<int64_t>(rot->a) * rot->b != d)
      return FQ_ERR_INVALID_ARG;
    std::vector<char> seen(d, 0);
    for (int i = 0; i < d; ++i) {
      const int64_t p = rot->perm[i];
      if (p < 0 || p >= d || seen[p] || (rot->signs[i] != 1.0 && rot->signs[i] != -1.0))
        return FQ_ERR_INVALID_ARG;
      seen[p] = 1;
    }
  }
  const FrameWs L = frame_ws(k, rho, d, rot ? rot->a : 0, rot ? rot->b : 0);
  if (!ws || ws_bytes < L.total) return FQ_ERR_WORKSPACE;
  char* w = static_cast<char*>(ws);
  float* buf0 = reinterpret_cast<float*>(w + L.buf);
  float* buf1 = buf0 + total;
  double* dF = reinterpret_cast<double*>(w + L.F);

  if (rho_c == 0) {
    float* dst = rot ? buf0 : T;
    if (cudaMemsetAsync(dst, 0, total * 4, s) != cudaSuccess) return FQ_ERR_CUDA;
    eye_kernel<<<static_cast<unsigned>(ceil_div(d, 256)), 256, 0, s>>>(dst, d);
    if (cudaGetLastError() != cudaSuccess) return FQ_ERR_CUDA;
  } else {
    if (cudaMemcpyAsync(dF, F.data(), F.size() * 8, cudaMemcpyHostToDevice, s) != cudaSuccess)
      return FQ_ERR_CUDA;
    tff_fill_kernel<<<grid_for(total), 256, 0, s>>>(dF, rho_c, d_c, k, rot ? buf0 : T, total);
    if (cudaGetLastError() != cudaSuccess) return FQ_ERR_CUDA;
    if (!rot && cudaStreamSynchronize(s) != cudaSuccess) return FQ_ERR_CUDA;
  }
  if (!rot) return FQ_OK;

  const int a = rot->a, b = rot->b;
  std::vector<double> Qa, Qb;
  haar_q(rot->gauss_a, a, Qa);
  haar_q(rot->gauss_b, b, Qb);
  std::vector<float> qa(Qa.begin(), Qa.end()), qb(Qb.begin(), Qb.end()), sg(d);
  std::vector<int> pm(d);
  for (int i = 0; i < d; ++i) sg[i] = static_cast<float>(rot->signs[i]), pm[i] = static_cast<int>(rot->perm[i]);
  float* dQa = reinterpret_cast<float*>(w + L.Qa);
  float* dQb = reinterpret_cast<float*>(w + L.Qb);
  float* dSg = reinterpret_cast<float*>(w + L.signs);
  int* dPm = reinterpret_cast<int*>(w + L.perm);
  if (cudaMemcpyAsync(dQa, qa.data(), qa.size() * 4, cudaMemcpyHostToDevice, s) != cudaSuccess ||
      cudaMemcpyAsync(dQb, qb.data(), qb.size() * 4, cudaMemcpyHostToDevice, s) != cudaSuccess ||
      cudaMemcpyAsync(dSg, sg.data(), sg.size() * 4, cudaMemcpyHostToDevice, s) != cudaSuccess ||
      cudaMemcpyAsync(dPm, pm.data(), pm.size() * 4, cudaMemcpyHostToDevice, s) != cudaSuccess)
    return FQ_ERR_CUDA;
  // X = T D (buf0 -> T as scratch), Z = X Qb^T, Zt per row, Yt = Zt Qa^T, out = permuted Y
  sign_kernel<<<grid_for(total), 256, 0, s>>>(buf0, dSg, T, total, d);
  cudaError_t e = gemm_nt(T, dQb, buf1, n * a, b, b, 1, 0, 0, 0, s);
  if (e != cudaSuccess) return FQ_ERR_CUDA;
  transpose_rows_kernel<<<grid_for(total), 256, 0, s>>>(buf1, buf0, total, a, b);
  e = gemm_nt(buf0, dQa, buf1, n * b, a, a, 1, 0, 0, 0, s);
  if (e != cudaSuccess) return FQ_ERR_CUDA;
  permute_kernel<<<grid_for(total), 256, 0, s>>>(buf1, dPm, T, total, a, b);
  if (cudaGetLastError() != cudaSuccess) return FQ_ERR_CUDA;
  // host vectors above are freed on return; the copies from them must be complete
  return cudaStreamSynchronize(s) == cudaSuccess ? FQ_OK : FQ_ERR_CUDA;
}

size_t fq_coefficients_workspace_bytes(int d_out, int n_in) {
  if (d_out <= 0 || n_in <= 0) return 0;
  return static_cast<size_t>(round_up(static_cast<int64_t>(n_in) * d_out * 4, 256));
}

fq_status fq_coefficients(const float* W, int d_out, int d_in, const float* T_in, int n_in,
                          const float* T_out, int n_out, float* C, void* ws, size_t ws_bytes,
                          fq_stream_t stream) {
  if (!W || !T_in || !T_out || !C || d_out <= 0 || d_in <= 0 || n_in <= 0 || n_out <= 0)
    return FQ_ERR_INVALID_ARG;
  if (!ws || ws_bytes < fq_coefficients_workspace_bytes(d_out, n_in)) return FQ_ERR_WORKSPACE;
  auto s = reinterpret_cast<cudaStream_t>(stream);
  float* Pt = static_cast<float*>(ws);                    // Pt = T_in W^T  (n_in x d_out)
  if (gemm_nt(T_in, W, Pt, n_in, d_out, d_in, 1, 0, 0, 0, s) != cudaSuccess) return FQ_ERR_CUDA;
  if (gemm_nt(T_out, Pt, C, n_out, n_in, d_out, 1, 0, 0, 0, s) != cudaSuccess)   // C = T_out Pt^T
    return FQ_ERR_CUDA;
  return FQ_OK;
}

fq_status fq_quantize_rtn(const float* C, int n_out, int n_in, uint8_t* codes, uint16_t* scale,
                          uint16_t* zero, float* gamma, fq_stream_t stream) {
  if (!C || !codes || !scale || !zero || n_out <= 0 || n_in <= 0) return FQ_ERR_INVALID_ARG;
  auto s = reinterpret_cast<cudaStream_t>(stream);
  rtn_kernel<<<static_cast<unsigned>(n_out), 256, 0, s>>>(
      C, n_in, codes, reinterpret_cast<__half*>(scale), reinterpret_cast<__half*>(zero), gamma);
  return cudaGetLastError() == cudaSuccess ? FQ_OK : FQ_ERR_CUDA;
}

}  // extern "C"
