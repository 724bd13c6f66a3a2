// Forward pass with frames in structured form (the decode path, M <= 64 tokens).
//
// With d a multiple of rho, the un-rotated analysis operator T_u of the (k, rho, d) frame is
// block-diagonal (Appendix J): run j = 0 .. rho/2 - 1 covers the complex coordinates
// c = j w .. (j+1) w - 1 (w = d / rho; complex coordinate c is real coordinates 2c, 2c + 1), and
// its k frame vectors are the realified rows of exp(2 pi i k_i c / k) / sqrt(k).  The rotated
// frame is T = T_u R^T, R = Pi (Q_a kron Q_b) D (Appendix K), so
//     analysis   z = T_u (R^T x):   z_(j,k_i) = k^-1/2 sum_c exp(-2 pi i k_i c / k) v_c
//     synthesis  y = R (T_u^T u):   y_c = k^-1/2 sum_(k_i) exp(+2 pi i k_i c / k) u_(j,k_i)
// with complex pairs (real part at the even row or coordinate, imaginary at the odd one).
//
// One forward is five kernels chained with programmatic dependent launch:
//   rotate<analysis>   v = R_in^T x        (fp32, workspace)
//   run_analysis       z = T_u,in v        (bf16, the fused decode kernel's z slot)
//   decode core        u = gamma (C_hat z) (the fused decode kernel with its code product only)
//   run_synthesis      s = T_u,out^T u     (fp32, workspace)
//   rotate<synthesis>  y = R_out s         (bf16)
// The rotations and run transforms are fp32 on CUDA cores: at decode batch sizes they are a few
// MFLOP per token, while the dense operators they replace are 2 n d bytes of HBM traffic.
// Each kernel triggers its dependents at entry, stages its constant inputs (roots of unity,
// rotation rows), and waits for its predecessor before touching the workspace or its input.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <mutex>
#include <set>
#include <vector>

#include "fq_device.cuh"
#include "fq_internal.h"

namespace fq {
namespace {

constexpr int kRunWarps = 8;       // warps of a run-transform CTA: segments of the reduction
constexpr int kRunTokens = 8;      // tokens per run-transform CTA
constexpr int kMaxRotRows = 8;     // rows of the a x b rotated block per rotation CTA
constexpr int kMaxRunW = 2560;     // complex coordinates per run
constexpr int kMaxK = 4096;        // frame vectors per run

// ------------------------------------------------------------------------------ rotations
// CTA (token t, rows r0 .. r0 + G - 1 of the a x b block); thread c < b owns column c
// (b <= 1024; the CTA has at least 256 threads for the loads).
//   analysis:  V = Pi^T x (V[perm[i]] = x_i), Y = Q_a^T V Q_b, out = D vec(Y)      A = Q_a^T, B = Q_b
//   synthesis: V = D s, Y = Q_a V Q_b^T, out = Pi vec(Y) (out[iperm[e]] = vec(Y)_e) A = Q_a, B = Q_b^T
// B is staged through shared memory kRotChunk rows at a time (coalesced loads, all in flight
// together), so no thread waits on a chain of dependent L2 loads.
constexpr int kRotChunk = 32;

template <bool kSynth>
__global__ void __launch_bounds__(1024) rotate_kernel(const void* __restrict__ in,
                                                      void* __restrict__ out, int d, int a,
                                                      int b, int G, const float* __restrict__ A,
                                                      const float* __restrict__ B,
                                                      const int32_t* __restrict__ perm,
                                                      const int32_t* __restrict__ iperm,
                                                      const float* __restrict__ signs) {
  extern __shared__ float sm[];
  float* V = sm;                    // [d]
  float* Ar = V + d;                // [G][a]
  float* T1 = Ar + G * a;           // [G][b]
  float* Bs = T1 + G * b;           // [kRotChunk][b]
  const int t = blockIdx.y, r0 = blockIdx.x * G, nt = blockDim.x;
  const int rows = min(G, a - r0);
  const int c = threadIdx.x;
  const bool col = c < b;
  pdl_launch_dependents();
  for (int i = threadIdx.x; i < rows * a; i += nt) Ar[i] = A[static_cast<int64_t>(r0) * a + i];
  pdl_wait();
  if (kSynth) {
    const float* s = static_cast<const float*>(in) + static_cast<int64_t>(t) * d;
#pragma unroll 8
    for (int i = threadIdx.x; i < d; i += nt) V[i] = signs[i] * s[i];
  } else {
    const __nv_bfloat16* x = static_cast<const __nv_bfloat16*>(in) + static_cast<int64_t>(t) * d;
#pragma unroll 8
    for (int i = threadIdx.x; i < d; i += nt) V[perm[i]] = __bfloat162float(x[i]);
  }
  __syncthreads();
  float acc[kMaxRotRows];
#pragma unroll
  for (int g = 0; g < kMaxRotRows; ++g) acc[g] = 0.f;
  if (col) {
    for (int r = 0; r < a; ++r) {
      const float v = V[r * b + c];
#pragma unroll
      for (int g = 0; g < kMaxRotRows; ++g)
        if (g < rows) acc[g] = fmaf(Ar[g * a + r], v, acc[g]);
    }
#pragma unroll
    for (int g = 0; g < kMaxRotRows; ++g)
      if (g < rows) T1[g * b + c] = acc[g];
  }
#pragma unroll
  for (int g = 0; g < kMaxRotRows; ++g) acc[g] = 0.f;
  for (int k0 = 0; k0 < b; k0 += kRotChunk) {
    const int kn = min(kRotChunk, b - k0);
    __syncthreads();            // T1 written (first chunk), the previous chunk consumed
#pragma unroll 8
    for (int i = threadIdx.x; i < kn * b; i += nt) Bs[i] = B[static_cast<int64_t>(k0) * b + i];
    __syncthreads();
    if (col) {
      for (int kk = 0; kk < kn; ++kk) {
        const float w = Bs[kk * b + c];
#pragma unroll
        for (int g = 0; g < kMaxRotRows; ++g)
          if (g < rows) acc[g] = fmaf(T1[g * b + k0 + kk], w, acc[g]);
      }
    }
  }
  if (!col) return;
#pragma unroll
  for (int g = 0; g < kMaxRotRows; ++g) {
    if (g >= rows) continue;
    const int e = (r0 + g) * b + c;
    if (kSynth) {
      static_cast<__nv_bfloat16*>(out)[static_cast<int64_t>(t) * d + iperm[e]] =
          __float2bfloat16_rn(acc[g]);
    } else {
      static_cast<float*>(out)[static_cast<int64_t>(t) * d + e] = signs[e] * acc[g];
    }
  }
}

// Without a rotation: a copy that converts (bf16 -> fp32 for the analysis, fp32 -> bf16 for the
// synthesis).
template <bool kSynth>
__global__ void __launch_bounds__(256) copy_kernel(const void* __restrict__ in,
                                                   void* __restrict__ out, int64_t n) {
  pdl_launch_dependents();
  pdl_wait();
  for (int64_t i = blockIdx.x * 256ll + threadIdx.x; i < n; i += gridDim.x * 256ll) {
    if (kSynth)
      static_cast<__nv_bfloat16*>(out)[i] = __float2bfloat16_rn(static_cast<const float*>(in)[i]);
    else
      static_cast<float*>(out)[i] = __bfloat162float(static_cast<const __nv_bfloat16*>(in)[i]);
  }
}

// -------------------------------------------------------------------------- run transforms
// Analysis of run j for frame vectors k_i = kc .. kc + 31 (lane) and tokens t0 .. t0 + 7: warp q
// sums over its segment of the run's w complex coordinates, the segments are added in warp
// order.  The root index (k_i c) mod k advances by k_i per coordinate.
__global__ void __launch_bounds__(kRunWarps * 32) run_analysis_kernel(
    const float* __restrict__ v, __nv_bfloat16* __restrict__ z, int M, int d, int n, int k,
    int w, int kchunks, float rk, const float2* __restrict__ roots) {
  extern __shared__ float sm[];
  float2* rt = reinterpret_cast<float2*>(sm);                     // [k]
  float2* xs = rt + k;                                            // [kRunTokens][w]
  float2* red = xs + kRunTokens * w;                              // [warps][tokens][32]
  const int j = blockIdx.x / kchunks, kc = (blockIdx.x % kchunks) * 32;
  const int t0 = blockIdx.y * kRunTokens, nt = min(kRunTokens, M - t0);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  pdl_launch_dependents();
#pragma unroll 4
  for (int i = threadIdx.x; i < k; i += blockDim.x) rt[i] = roots[i];
  pdl_wait();
#pragma unroll 8
  for (int i = threadIdx.x; i < kRunTokens * w; i += blockDim.x) {
    const int tt = i / w, c = i % w;
    xs[i] = tt < nt ? *reinterpret_cast<const float2*>(
                          v + static_cast<int64_t>(t0 + tt) * d + 2 * (static_cast<int64_t>(j) * w + c))
                    : make_float2(0.f, 0.f);
  }
  __syncthreads();
  const int ki = kc + lane;
  const int seg = (w + kRunWarps - 1) / kRunWarps;
  const int c0 = warp * seg, c1 = min(w, c0 + seg);
  float re[kRunTokens], im[kRunTokens];
#pragma unroll
  for (int tt = 0; tt < kRunTokens; ++tt) re[tt] = im[tt] = 0.f;
  if (ki < k && c0 < c1) {
    int idx = static_cast<int>((static_cast<int64_t>(ki) * (static_cast<int64_t>(j) * w + c0)) % k);
    for (int c = c0; c < c1; ++c) {
      const float2 r = rt[idx];
#pragma unroll
      for (int tt = 0; tt < kRunTokens; ++tt) {
        const float2 x = xs[tt * w + c];
        re[tt] = fmaf(x.x, r.x, fmaf(x.y, r.y, re[tt]));
        im[tt] = fmaf(x.y, r.x, fmaf(-x.x, r.y, im[tt]));
      }
      idx += ki;
      if (idx >= k) idx -= k;
    }
  }
#pragma unroll
  for (int tt = 0; tt < kRunTokens; ++tt)
    red[(warp * kRunTokens + tt) * 32 + lane] = make_float2(re[tt], im[tt]);
  __syncthreads();
  for (int i = threadIdx.x; i < kRunTokens * 32; i += blockDim.x) {
    const int tt = i / 32, l = i % 32, kk = kc + l;
    if (tt >= nt || kk >= k) continue;
    float sr = 0.f, si = 0.f;
    for (int q = 0; q < kRunWarps; ++q) {
      const float2 p = red[(q * kRunTokens + tt) * 32 + l];
      sr += p.x;
      si += p.y;
    }
    *reinterpret_cast<__nv_bfloat162*>(z + static_cast<int64_t>(t0 + tt) * n +
                                        2 * (static_cast<int64_t>(j) * k + kk)) =
        __floats2bfloat162_rn(sr * rk, si * rk);
  }
}

// Synthesis of run j for complex coordinates c = j w + cc .. + 31 (lane) and tokens t0 .. t0 + 7:
// warp q sums over its segment of the k frame vectors; the root index (k_i c) mod k advances by
// c mod k per frame vector.
__global__ void __launch_bounds__(kRunWarps * 32) run_synthesis_kernel(
    const __nv_bfloat16* __restrict__ u, float* __restrict__ s, int M, int d, int n, int k,
    int w, int cchunks, float rk, const float2* __restrict__ roots) {
  extern __shared__ float sm[];
  float2* rt = reinterpret_cast<float2*>(sm);                             // [k]
  float2* red = rt + k;                                                   // [warps][tokens][32]
  __nv_bfloat162* us = reinterpret_cast<__nv_bfloat162*>(red + kRunWarps * kRunTokens * 32);  // [tokens][k]
  const int j = blockIdx.x / cchunks, cc = (blockIdx.x % cchunks) * 32;
  const int t0 = blockIdx.y * kRunTokens, nt = min(kRunTokens, M - t0);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  pdl_launch_dependents();
#pragma unroll 4
  for (int i = threadIdx.x; i < k; i += blockDim.x) rt[i] = roots[i];
  pdl_wait();
#pragma unroll 8
  for (int i = threadIdx.x; i < kRunTokens * k; i += blockDim.x) {
    const int tt = i / k, q = i % k;
    us[i] = tt < nt ? *reinterpret_cast<const __nv_bfloat162*>(
                          u + static_cast<int64_t>(t0 + tt) * n + 2 * (static_cast<int64_t>(j) * k + q))
                    : __floats2bfloat162_rn(0.f, 0.f);
  }
  __syncthreads();
  const int c = cc + lane;                       // complex coordinate within the run
  const int seg = (k + kRunWarps - 1) / kRunWarps;
  const int q0 = warp * seg, q1 = min(k, q0 + seg);
  float yr[kRunTokens], yi[kRunTokens];
#pragma unroll
  for (int tt = 0; tt < kRunTokens; ++tt) yr[tt] = yi[tt] = 0.f;
  if (c < w && q0 < q1) {
    const int64_t cabs = static_cast<int64_t>(j) * w + c;
    const int step = static_cast<int>(cabs % k);
    int idx = static_cast<int>((static_cast<int64_t>(q0) * cabs) % k);
    for (int q = q0; q < q1; ++q) {
      const float2 r = rt[idx];
#pragma unroll
      for (int tt = 0; tt < kRunTokens; ++tt) {
        const float2 p = __bfloat1622float2(us[tt * k + q]);
        yr[tt] = fmaf(p.x, r.x, fmaf(-p.y, r.y, yr[tt]));
        yi[tt] = fmaf(p.y, r.x, fmaf(p.x, r.y, yi[tt]));
      }
      idx += step;
      if (idx >= k) idx -= k;
    }
  }
#pragma unroll
  for (int tt = 0; tt < kRunTokens; ++tt)
    red[(warp * kRunTokens + tt) * 32 + lane] = make_float2(yr[tt], yi[tt]);
  __syncthreads();
  for (int i = threadIdx.x; i < kRunTokens * 32; i += blockDim.x) {
    const int tt = i / 32, l = i % 32, cl = cc + l;
    if (tt >= nt || cl >= w) continue;
    float sr = 0.f, si = 0.f;
    for (int q = 0; q < kRunWarps; ++q) {
      const float2 p = red[(q * kRunTokens + tt) * 32 + l];
      sr += p.x;
      si += p.y;
    }
    *reinterpret_cast<float2*>(s + static_cast<int64_t>(t0 + tt) * d +
                               2 * (static_cast<int64_t>(j) * w + cl)) =
        make_float2(sr * rk, si * rk);
  }
}

// ------------------------------------------------------------------------------ host side
struct FrameBuf {
  size_t Qa, QaT, Qb, QbT, perm, iperm, signs, roots, total;
};

FrameBuf frame_buf(int k, int d, int a, int b) {
  FrameBuf L{};
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off += static_cast<size_t>(round_up(static_cast<int64_t>(bytes), 256));
    return o;
  };
  const size_t qa = static_cast<size_t>(a) * a * 4, qb = static_cast<size_t>(b) * b * 4;
  L.Qa = take(qa);
  L.QaT = take(qa);
  L.Qb = take(qb);
  L.QbT = take(qb);
  L.perm = take(static_cast<size_t>(d) * 4);
  L.iperm = take(static_cast<size_t>(d) * 4);
  L.signs = take(static_cast<size_t>(d) * 4);
  L.roots = take(static_cast<size_t>(k) * 8);
  L.total = off;
  return L;
}

bool valid_triple(int k, int rho, int d) {
  return k > 0 && rho >= 2 && rho % 2 == 0 && d > 0 && d % rho == 0 && k >= d / rho;
}

bool valid_frame(const fq_frame* f) {
  if (!f || !valid_triple(f->k, f->rho, f->d) || !f->roots) return false;
  if (f->a == 0 && f->b == 0) return true;
  return f->a > 0 && f->b > 0 && static_cast<int64_t>(f->a) * f->b == f->d && f->Qa && f->QaT &&
         f->Qb && f->QbT && f->perm && f->iperm && f->signs;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

struct ImplWs {
  size_t z, u, v, s, total;
};

ImplWs impl_ws(int M, int d_in, int n_in, int n_out, int d_out) {
  ImplWs L{};
  L.z = decode_core_z_offset();
  L.u = decode_core_u_offset(M, n_in);
  size_t off = decode_workspace_bytes(M, d_in, n_in, n_out, d_out);
  L.v = off;
  off += static_cast<size_t>(round_up(static_cast<int64_t>(M) * d_in * 4, 256));
  L.s = off;
  off += static_cast<size_t>(round_up(static_cast<int64_t>(M) * d_out * 4, 256));
  L.total = off;
  return L;
}

size_t rot_smem(const fq_frame& f, int G) {
  return (static_cast<size_t>(f.d) + static_cast<size_t>(G) * (f.a + f.b) +
          static_cast<size_t>(kRotChunk) * f.b) * 4;
}
size_t ana_smem(const fq_frame& f) {
  const int w = f.d / f.rho;
  return (static_cast<size_t>(f.k) + kRunTokens * w + kRunWarps * kRunTokens * 32) * 8;
}
size_t syn_smem(const fq_frame& f) {
  return (static_cast<size_t>(f.k) + kRunWarps * kRunTokens * 32) * 8 +
         static_cast<size_t>(kRunTokens) * f.k * 4;
}

constexpr size_t kMaxSmem = 227 * 1024;

bool frame_fits(const fq_frame& f) {
  const int w = f.d / f.rho;
  if (w > kMaxRunW || f.k > kMaxK) return false;
  if (f.a > 0 && (f.b > 1024 || rot_smem(f, kMaxRotRows) > kMaxSmem)) return false;
  return ana_smem(f) <= kMaxSmem && syn_smem(f) <= kMaxSmem;
}

cudaError_t set_smem_attributes() {
  static std::mutex mu;
  static std::set<int> done;
  int dev = 0;
  cudaGetDevice(&dev);
  std::lock_guard<std::mutex> g(mu);
  if (done.count(dev)) return cudaSuccess;
  const int bytes = static_cast<int>(kMaxSmem);
  cudaError_t e = cudaFuncSetAttribute(rotate_kernel<false>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(rotate_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             bytes);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(run_analysis_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             bytes);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(run_synthesis_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             bytes);
  if (e == cudaSuccess) done.insert(dev);
  return e;
}

// Launch with programmatic stream serialization (the kernel may start while its predecessor
// in the stream finishes; it waits with griddepcontrol.wait before reading its inputs).
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t s, Args... args) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

int rot_rows_per_cta(int a, int M) {
  return std::max(1, std::min(kMaxRotRows, static_cast<int>(ceil_div(static_cast<int64_t>(a) * M, 296))));
}

// R^T x (analysis, bf16 in, fp32 out) or R s (synthesis, fp32 in, bf16 out) for M tokens
template <bool kSynth>
cudaError_t rotate(const fq_frame& f, int M, const void* in, void* out, cudaStream_t s) {
  if (f.a == 0) {
    const int64_t n = static_cast<int64_t>(M) * f.d;
    const unsigned grid = static_cast<unsigned>(std::min<int64_t>(ceil_div(n, 256), 1184));
    return launch_pdl(copy_kernel<kSynth>, dim3(grid), dim3(256), 0, s, in, out, n);
  }
  const int G = rot_rows_per_cta(f.a, M);
  // one thread per column of the a x b block, at least 256 for the loads
  const int threads = static_cast<int>(std::min<int64_t>(1024, std::max<int64_t>(256, round_up(f.b, 32))));
  return launch_pdl(rotate_kernel<kSynth>, dim3(static_cast<unsigned>(ceil_div(f.a, G)), M),
                    dim3(threads), rot_smem(f, G), s, in, out, f.d, f.a, f.b, G,
                    kSynth ? f.Qa : f.QaT, kSynth ? f.QbT : f.Qb, f.perm, f.iperm, f.signs);
}

}  // namespace
}  // namespace fq

using namespace fq;

extern "C" {

size_t fq_frame_implicit_bytes(int k, int rho, int d, int a, int b) {
  if (!valid_triple(k, rho, d) || a < 0 || b < 0) return 0;
  if ((a == 0) != (b == 0) || (a > 0 && static_cast<int64_t>(a) * b != d)) return 0;
  return frame_buf(k, d, a, b).total;
}

fq_status fq_frame_implicit(int k, int rho, int d, const fq_rotation* rot, void* buf,
                            size_t bytes, fq_frame* out, fq_stream_t stream) {
  if (!out || !valid_triple(k, rho, d)) return FQ_ERR_INVALID_ARG;
  const int a = rot ? rot->a : 0, b = rot ? rot->b : 0;
  if (rot) {
    if (!rot->gauss_a || !rot->gauss_b || !rot->perm || !rot->signs || a <= 0 || b <= 0 ||
        static_cast<int64_t>(a) * b != d)
      return FQ_ERR_INVALID_ARG;
    std::vector<char> seen(d, 0);
    for (int i = 0; i < d; ++i) {
      const int64_t p = rot->perm[i];
      if (p < 0 || p >= d || seen[p] || (rot->signs[i] != 1.0 && rot->signs[i] != -1.0))
        return FQ_ERR_INVALID_ARG;
      seen[p] = 1;
    }
  }
  const FrameBuf L = frame_buf(k, d, a, b);
  if (!buf || bytes < L.total) return FQ_ERR_WORKSPACE;
  if ((reinterpret_cast<uintptr_t>(buf) & 255u) != 0) return FQ_ERR_ALIGNMENT;
  auto s = reinterpret_cast<cudaStream_t>(stream);
  char* base = static_cast<char*>(buf);
  // roots of unity exp(2 pi i m / k), m = 0 .. k-1 (host, double precision)
  std::vector<float> roots(2 * static_cast<size_t>(k));
  const double two_pi = 6.283185307179586476925286766559;
  for (int m = 0; m < k; ++m) {
    const double th = two_pi * m / k;
    roots[2 * m] = static_cast<float>(std::cos(th));
    roots[2 * m + 1] = static_cast<float>(std::sin(th));
  }
  std::vector<float> qa, qat, qb, qbt, sg;
  std::vector<int32_t> pm, ipm;
  if (rot) {
    std::vector<double> Qa, Qb;
    haar_q(rot->gauss_a, a, Qa);
    haar_q(rot->gauss_b, b, Qb);
    qa.resize(static_cast<size_t>(a) * a);
    qat.resize(qa.size());
    for (int i = 0; i < a; ++i)
      for (int j = 0; j < a; ++j) {
        qa[static_cast<size_t>(i) * a + j] = static_cast<float>(Qa[static_cast<size_t>(i) * a + j]);
        qat[static_cast<size_t>(j) * a + i] = static_cast<float>(Qa[static_cast<size_t>(i) * a + j]);
      }
    qb.resize(static_cast<size_t>(b) * b);
    qbt.resize(qb.size());
    for (int i = 0; i < b; ++i)
      for (int j = 0; j < b; ++j) {
        qb[static_cast<size_t>(i) * b + j] = static_cast<float>(Qb[static_cast<size_t>(i) * b + j]);
        qbt[static_cast<size_t>(j) * b + i] = static_cast<float>(Qb[static_cast<size_t>(i) * b + j]);
      }
    sg.resize(d);
    pm.resize(d);
    ipm.resize(d);
    for (int i = 0; i < d; ++i) {
      sg[i] = static_cast<float>(rot->signs[i]);
      pm[i] = static_cast<int32_t>(rot->perm[i]);
      ipm[pm[i]] = i;
    }
  }
  auto up = [&](size_t off, const void* src, size_t n) {
    return n == 0 || cudaMemcpyAsync(base + off, src, n, cudaMemcpyHostToDevice, s) == cudaSuccess;
  };
  if (!up(L.roots, roots.data(), roots.size() * 4) || !up(L.Qa, qa.data(), qa.size() * 4) ||
      !up(L.QaT, qat.data(), qat.size() * 4) || !up(L.Qb, qb.data(), qb.size() * 4) ||
      !up(L.QbT, qbt.data(), qbt.size() * 4) || !up(L.signs, sg.data(), sg.size() * 4) ||
      !up(L.perm, pm.data(), pm.size() * 4) || !up(L.iperm, ipm.data(), ipm.size() * 4))
    return FQ_ERR_CUDA;
  // the host vectors are released on return: the copies from them must be complete
  if (cudaStreamSynchronize(s) != cudaSuccess) return FQ_ERR_CUDA;
  fq_frame f{};
  f.k = k;
  f.rho = rho;
  f.d = d;
  f.a = a;
  f.b = b;
  f.roots = reinterpret_cast<const float*>(base + L.roots);
  if (rot) {
    f.Qa = reinterpret_cast<const float*>(base + L.Qa);
    f.QaT = reinterpret_cast<const float*>(base + L.QaT);
    f.Qb = reinterpret_cast<const float*>(base + L.Qb);
    f.QbT = reinterpret_cast<const float*>(base + L.QbT);
    f.perm = reinterpret_cast<const int32_t*>(base + L.perm);
    f.iperm = reinterpret_cast<const int32_t*>(base + L.iperm);
    f.signs = reinterpret_cast<const float*>(base + L.signs);
  }
  *out = f;
  return FQ_OK;
}

size_t fq_implicit_workspace_bytes(int M, int d_in, int n_in, int n_out, int d_out) {
  if (M <= 0 || M > kDecodeMaxM || d_in <= 0 || n_in <= 0 || n_out <= 0 || d_out <= 0) return 0;
  return impl_ws(M, d_in, n_in, n_out, d_out).total;
}

fq_status fq_linear_forward_implicit(const void* x, int M, const fq_frame* F_in,
                                     const fq_packed* C, const fq_frame* F_out,
                                     const float* gamma, void* y, void* ws, size_t ws_bytes,
                                     int max_sms, fq_stream_t stream) {
  if (!x || !y || !C || max_sms < 0 || M <= 0) return FQ_ERR_INVALID_ARG;
  if (const fq_status cs = check_packed(C)) return cs;
  if (!valid_frame(F_in) || !valid_frame(F_out)) return FQ_ERR_INVALID_ARG;
  const fq_frame fi = *F_in, fo = *F_out;
  const int n_in = fi.k * fi.rho, n_out = fo.k * fo.rho;
  if (C->n_in != n_in || C->n_out != n_out) return FQ_ERR_INVALID_ARG;
  if (n_in % 16 || n_out % 16 || fi.d % 8 || fo.d % 8) return FQ_ERR_ALIGNMENT;
  if (!aligned16(x) || !aligned16(y) || (gamma && !aligned16(gamma)) || !aligned16(fi.roots) ||
      !aligned16(fo.roots))
    return FQ_ERR_ALIGNMENT;
  if (!ws) return FQ_ERR_WORKSPACE;
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return FQ_ERR_ALIGNMENT;
  if (M > kDecodeMaxM || !frame_fits(fi) || !frame_fits(fo)) return FQ_ERR_UNSUPPORTED;
  const ImplWs L = impl_ws(M, fi.d, n_in, n_out, fo.d);
  if (ws_bytes < L.total) return FQ_ERR_WORKSPACE;
  {
    int dev = 0, major = 0, minor = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess)
      return FQ_ERR_CUDA;
    if (major * 10 + minor != 103) return FQ_ERR_UNSUPPORTED;
  }
  if (set_smem_attributes() != cudaSuccess) return FQ_ERR_CUDA;
  auto s = reinterpret_cast<cudaStream_t>(stream);
  char* w = static_cast<char*>(ws);
  float* v = reinterpret_cast<float*>(w + L.v);
  float* sy = reinterpret_cast<float*>(w + L.s);
  auto* z = reinterpret_cast<__nv_bfloat16*>(w + L.z);
  auto* u = reinterpret_cast<__nv_bfloat16*>(w + L.u);
  const unsigned tchunks = static_cast<unsigned>(ceil_div(M, kRunTokens));

  if (rotate<false>(fi, M, x, v, s) != cudaSuccess) return FQ_ERR_CUDA;
  {
    const int wi = fi.d / fi.rho, kch = static_cast<int>(ceil_div(fi.k, 32));
    const float rk = static_cast<float>(1.0 / std::sqrt(static_cast<double>(fi.k)));
    if (launch_pdl(run_analysis_kernel, dim3(static_cast<unsigned>(fi.rho / 2 * kch), tchunks),
                   dim3(kRunWarps * 32), ana_smem(fi), s, v, z, M, fi.d, n_in, fi.k, wi, kch, rk,
                   reinterpret_cast<const float2*>(fi.roots)) != cudaSuccess)
      return FQ_ERR_CUDA;
  }
  const fq_status st = launch_decode_core(M, *C, gamma, w, ws_bytes, max_sms, s);
  if (st != FQ_OK) return st;
  {
    const int wo = fo.d / fo.rho, cch = static_cast<int>(ceil_div(wo, 32));
    const float rk = static_cast<float>(1.0 / std::sqrt(static_cast<double>(fo.k)));
    if (launch_pdl(run_synthesis_kernel, dim3(static_cast<unsigned>(fo.rho / 2 * cch), tchunks),
                   dim3(kRunWarps * 32), syn_smem(fo), s, u, sy, M, fo.d, n_out, fo.k, wo, cch, rk,
                   reinterpret_cast<const float2*>(fo.roots)) != cudaSuccess)
      return FQ_ERR_CUDA;
  }
  if (rotate<true>(fo, M, sy, y, s) != cudaSuccess) return FQ_ERR_CUDA;
  return FQ_OK;
}

}  // extern "C"
