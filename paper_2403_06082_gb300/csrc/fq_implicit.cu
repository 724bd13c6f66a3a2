// Forward pass with frames in structured form (the decode path, M <= 64 tokens).
//
// With d a multiple of rho, the un-rotated analysis operator T_u of the (k, rho, d) frame is
// block-diagonal (Appendix J): run j = 0 .. rho/2 - 1 covers the complex coordinates
// c = j w .. (j+1) w - 1 (w = d / rho; complex coordinate c is real coordinates 2c, 2c + 1), and
// its k frame vectors are the realified rows of exp(2 pi i k_i c / k) / sqrt(k).  The rotated
// frame is T = T_u R^T, R = Pi (Q_a kron Q_b) D (Appendix K), so
//     z = T_u (R^T x),        y = R (T_u^T u).
//
// One forward is three kernels chained with programmatic dependent launch:
//   rotate<analysis>   v = R_in^T x   (bf16)
//   the fused decode kernel with block-sparse frame operands: z = T_u,in v, the 2-bit code
//                      product, s = T_u,out^T u, all on the tensor cores (its analysis and
//                      synthesis read only the K blocks of each row tile's runs, stored as
//                      contiguous pre-swizzled 16 KiB tiles: about 1/8 of the dense operator
//                      for rho = 16)
//   rotate<synthesis>  y = R_out s   (bf16)
// Without a rotation the fused kernel reads x and writes y itself.  The rotations are two small
// products per token on CUDA cores (a x a and b x b with a b = d).
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstring>
#include <mutex>
#include <set>
#include <vector>

#include "fq_device.cuh"
#include "fq_internal.h"

namespace fq {
namespace {


// ------------------------------------------------------------------------------ rotations
// CTA (token t, rows r0 .. r0 + 7 of the a x b block); bf16 in and out.
//   analysis:  V = Pi^T x (V[perm[i]] = x_i), Y = Q_a^T V Q_b, out = D vec(Y)      A = Q_a^T, B = Q_b
//   synthesis: V = D s, Y = Q_a V Q_b^T, out = Pi vec(Y) (out[iperm[e]] = vec(Y)_e) A = Q_a, B = Q_b^T
// The CTA is KG groups of r threads (r = b rounded up to a warp): thread (c, g) owns column c and
// the reduction indices g, g + KG, ... of both products, for all eight rows at once (eight
// accumulators; the eight row values of a reduction index are one 32-byte broadcast read of a
// row-interleaved copy).  The KG partial sums of an entry are added in group order through
// shared memory.  The factors do not depend on the previous kernel: A's rows, and all of B
// when b <= kRotStageB and the CTA's shared memory stays within kRotSmemStaged (so that two
// CTAs fit an SM), are requested in shared memory before the wait for the input, with
// asynchronous copies all in flight at once; otherwise B streams through kRotBufs buffers of
// kRotChunk rows, so that its loads overlap the products (the first chunks are requested
// before the wait).
constexpr int kRotRows = 8;        // rows of the a x b block per rotation CTA
constexpr int kRotStageB = 128;
constexpr size_t kRotSmemStaged = 110 * 1024;
constexpr int kRotChunk = 16;
constexpr int kRotBufs = 4;
constexpr int kRotMaxGroups = 4;

// One launch rotates the tokens of up to FQ_MAX_GROUP layers (blockIdx.z = layer).
struct RotLayer {
  const __nv_bfloat16* in;
  __nv_bfloat16* out;
  int d, a, b;
  int bp, KG;             // column slots (b rounded up to 32) and reduction groups
  int staged;             // all of B in shared memory (else streamed in chunks)
  const float* A;
  const float* B;
  const int32_t* perm;
  const int32_t* iperm;
  const float* signs;
};
struct RotBatch {
  RotLayer L[FQ_MAX_GROUP];
};

__device__ __forceinline__ void cp_async16(float* smem_dst, const float* gsrc) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(smem_dst)), "l"(gsrc)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}
__device__ __forceinline__ void cp_async_wait_pending() {
  asm volatile("cp.async.wait_group %0;" ::"n"(kRotBufs - 1) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.wait_group 0;" ::: "memory");
}

__device__ __forceinline__ void fma8(float (&acc)[kRotRows], const float* r8, float v) {
  const float4 u0 = *reinterpret_cast<const float4*>(r8);
  const float4 u1 = *reinterpret_cast<const float4*>(r8 + 4);
  acc[0] = fmaf(u0.x, v, acc[0]);
  acc[1] = fmaf(u0.y, v, acc[1]);
  acc[2] = fmaf(u0.z, v, acc[2]);
  acc[3] = fmaf(u0.w, v, acc[3]);
  acc[4] = fmaf(u1.x, v, acc[4]);
  acc[5] = fmaf(u1.y, v, acc[5]);
  acc[6] = fmaf(u1.z, v, acc[6]);
  acc[7] = fmaf(u1.w, v, acc[7]);
}

template <bool kSynth>
__global__ void __launch_bounds__(1024) rotate_kernel(const __grid_constant__ RotBatch rb) {
  const RotLayer& ly = rb.L[blockIdx.z];
  const __nv_bfloat16* __restrict__ in = ly.in;
  __nv_bfloat16* __restrict__ out = ly.out;
  const int d = ly.d, a = ly.a, b = ly.b, bp = ly.bp, KG = ly.KG;
  const float* __restrict__ A = ly.A;
  const float* __restrict__ B = ly.B;
  const int32_t* __restrict__ perm = ly.perm;
  const int32_t* __restrict__ iperm = ly.iperm;
  const float* __restrict__ signs = ly.signs;
  pdl_launch_dependents();
  const int r0 = static_cast<int>(blockIdx.x) * kRotRows;
  if (r0 >= a) {
    pdl_wait();
    return;
  }
  extern __shared__ float4 rot_smem4[];
  float* V = reinterpret_cast<float*>(rot_smem4);   // [d], d rounded up to 4
  float* At = V + ((d + 3) & ~3);                   // [a][8]: At[i][g] = A[r0 + g][i]
  float* T1t = At + a * kRotRows;                   // [b][8]: T1t[k][g] = (A V)[r0 + g][k]
  float* P = T1t + b * kRotRows;                    // [KG][8][bp] partial sums
  float* Bs = P + KG * kRotRows * bp;               // all of B, or kRotBufs chunks of it
  const int t = blockIdx.y, nt = blockDim.x, tid = threadIdx.x;
  const int rows = min(kRotRows, a - r0);
  const int c = tid % bp, kg = tid / bp;
  const bool active = c < b && kg < KG;
  const bool staged = ly.staged != 0;
  const bool async = (b & 3) == 0;
  const int nch = (b + kRotChunk - 1) / kRotChunk;
  // chunk ch of B (rows ch * kRotChunk ..) into buffer ch mod kRotBufs; every thread commits a
  // group per call, so that the group count stays uniform
  auto stage_chunk = [&](int ch) {
    if (ch < nch) {
      const int k0 = ch * kRotChunk, kn = min(kRotChunk, b - k0);
      const float* src = B + static_cast<int64_t>(k0) * b;
      float* dst = Bs + (ch % kRotBufs) * kRotChunk * b;
      for (int i = tid; i < kn * b / 4; i += nt) cp_async16(dst + 4 * i, src + 4 * i);
    }
    cp_async_commit();
  };
  for (int i = tid; i < a * kRotRows; i += nt) {
    const int ii = i / kRotRows, g = i % kRotRows;
    At[i] = g < rows ? A[static_cast<int64_t>(r0 + g) * a + ii] : 0.f;
  }
  if (staged) {
    if (async) {
      for (int i = tid; i < b * b / 4; i += nt) cp_async16(Bs + 4 * i, B + 4 * i);
      cp_async_commit();
    } else {
#pragma unroll 8
      for (int i = tid; i < b * b; i += nt) Bs[i] = B[i];
    }
  } else if (async) {
    for (int ch = 0; ch < kRotBufs - 1; ++ch) stage_chunk(ch);
  }
  pdl_wait();
  const __nv_bfloat16* src = in + static_cast<int64_t>(t) * d;
  if (kSynth) {
#pragma unroll 8
    for (int i = tid; i < d; i += nt) V[i] = signs[i] * __bfloat162float(src[i]);
  } else {
#pragma unroll 8
    for (int i = tid; i < d; i += nt) V[perm[i]] = __bfloat162float(src[i]);
  }
  if (staged && async) cp_async_wait_all();
  __syncthreads();
  float acc[kRotRows];
  // T1 = A[rows] V: this thread's partial over i = kg, kg + KG, ...
#pragma unroll
  for (int g = 0; g < kRotRows; ++g) acc[g] = 0.f;
  if (active) {
#pragma unroll 4
    for (int i = kg; i < a; i += KG) fma8(acc, At + i * kRotRows, V[i * b + c]);
#pragma unroll
    for (int g = 0; g < kRotRows; ++g) P[(kg * kRotRows + g) * bp + c] = acc[g];
  }
  __syncthreads();
  for (int e = tid; e < b * kRotRows; e += nt) {
    const int k = e / kRotRows, g = e % kRotRows;
    float s = 0.f;
    for (int q = 0; q < KG; ++q) s += P[(q * kRotRows + g) * bp + k];
    T1t[e] = s;
  }
  __syncthreads();
  // Y = T1 B: this thread's partial over k = kg, kg + KG, ...
#pragma unroll
  for (int g = 0; g < kRotRows; ++g) acc[g] = 0.f;
  if (staged) {
    if (active) {
#pragma unroll 4
      for (int k = kg; k < b; k += KG) fma8(acc, T1t + k * kRotRows, Bs[k * b + c]);
    }
  } else {
    for (int ch = 0; ch < nch; ++ch) {
      const int k0 = ch * kRotChunk, k1 = min(b, k0 + kRotChunk);
      const float* Bc = Bs;
      if (async) {
        stage_chunk(ch + kRotBufs - 1);
        cp_async_wait_pending();     // chunk ch has landed (for this thread's copies)
        __syncthreads();             // ... and for every thread's
        Bc = Bs + (ch % kRotBufs) * kRotChunk * b;
      } else {
        for (int i = tid; i < (k1 - k0) * b; i += nt) Bs[i] = B[static_cast<int64_t>(k0) * b + i];
        __syncthreads();
      }
      if (active) {
        const int first = k0 + ((kg - k0 % KG) % KG + KG) % KG;
        for (int k = first; k < k1; k += KG) fma8(acc, T1t + k * kRotRows, Bc[(k - k0) * b + c]);
      }
      __syncthreads();               // the buffer is read before it is refilled
    }
  }
  if (active) {
#pragma unroll
    for (int g = 0; g < kRotRows; ++g) P[(kg * kRotRows + g) * bp + c] = acc[g];
  }
  __syncthreads();
  __nv_bfloat16* dst = out + static_cast<int64_t>(t) * d;
  for (int e = tid; e < rows * b; e += nt) {
    const int g = e / b, cc = e - g * b;
    float y = 0.f;
    for (int q = 0; q < KG; ++q) y += P[(q * kRotRows + g) * bp + cc];
    const int o = (r0 + g) * b + cc;
    if (kSynth)
      dst[iperm[o]] = __float2bfloat16_rn(y);
    else
      dst[o] = __float2bfloat16_rn(signs[o] * y);
  }
}

// ------------------------------------------------------------------------------ host side
constexpr int kTR = 128, kTK = 64;            // operand tile: 128 rows x 64 bf16 (16 KiB)
constexpr int kTileBytes = kTR * kTK * 2;

// The row tiles of a block-sparse frame operand and the K blocks each one touches.
//   analysis  (T_u, n x d):   row tile t covers frame rows [128 t, +128); run j owns frame rows
//             [2 k j, 2 k (j+1)) and real coordinates [2 w j, 2 w (j+1)) (the K range)
//   synthesis (T_u^T, d x n): row tile t covers coordinates [128 t, +128); run j owns them in
//             [2 w j, 2 w (j+1)) and frame rows [2 k j, 2 k (j+1)) (the K range)
struct SparseShape {
  int rows, cols, RT, KB;
  int run_rows, run_cols;        // rows and columns of one run in this orientation
  std::vector<int32_t> idx;      // [RT][3]: kb_lo, kb_hi, first stored tile
  int count = 0;
};

SparseShape sparse_shape(int k, int rho, int d, bool synthesis) {
  const int n = k * rho, w = d / rho;
  SparseShape S;
  S.rows = synthesis ? d : n;
  S.cols = synthesis ? n : d;
  S.run_rows = synthesis ? 2 * w : 2 * k;
  S.run_cols = synthesis ? 2 * k : 2 * w;
  S.RT = static_cast<int>(ceil_div(S.rows, kTR));
  S.KB = static_cast<int>(ceil_div(S.cols, kTK));
  S.idx.resize(3 * static_cast<size_t>(S.RT));
  for (int t = 0; t < S.RT; ++t) {
    const int r0 = t * kTR, r1 = std::min(S.rows, r0 + kTR);
    const int j0 = r0 / S.run_rows, j1 = (r1 - 1) / S.run_rows;
    const int lo = static_cast<int>((static_cast<int64_t>(j0) * S.run_cols) / kTK);
    const int hi = static_cast<int>(std::min<int64_t>(
        S.KB, ceil_div(static_cast<int64_t>(j1 + 1) * S.run_cols, kTK)));
    S.idx[3 * t] = lo;
    S.idx[3 * t + 1] = hi;
    S.idx[3 * t + 2] = S.count;
    S.count += hi - lo;
  }
  return S;
}

// bf16 bit pattern of a float, rounding to nearest even (the operands are finite)
uint16_t bf16_bits(float f) {
  uint32_t u;
  std::memcpy(&u, &f, 4);
  u += 0x7FFFu + ((u >> 16) & 1u);
  return static_cast<uint16_t>(u >> 16);
}

// The stored tiles of one orientation: entry (r, c) of the un-rotated analysis operator is,
// for frame row r = 2 (j k + k_i) + e and real coordinate c = 2 q + f with q in run j,
// v = exp(2 pi i k_i q / k) / sqrt(k) realified as (e, f) = (0,0) Re v, (0,1) Im v,
// (1,0) -Im v, (1,1) Re v (Appendix J; 0 outside the run), computed in double, rounded to fp32
// and then to bf16 like the dense operator.  Each tile is written in the 128-byte-swizzled
// shared-memory image of a K-major 128 x 64 tile: row r's 16-byte chunk h at chunk h ^ (r mod 8).
void fill_tiles(int k, int rho, int d, const SparseShape& S, bool synthesis,
                const std::vector<double>& cs, const std::vector<double>& sn,
                std::vector<uint16_t>& out) {
  const int w = d / rho;
  const double rk = 1.0 / std::sqrt(static_cast<double>(k));
  out.assign(static_cast<size_t>(S.count) * kTR * kTK, 0);
  for (int t = 0; t < S.RT; ++t) {
    const int lo = S.idx[3 * t], hi = S.idx[3 * t + 1], first = S.idx[3 * t + 2];
    for (int kb = lo; kb < hi; ++kb) {
      uint16_t* tile = out.data() + static_cast<size_t>(first + kb - lo) * kTR * kTK;
      for (int r = 0; r < kTR; ++r) {
        const int gr = t * kTR + r;
        if (gr >= S.rows) continue;
        for (int cc = 0; cc < kTK; ++cc) {
          const int gc = kb * kTK + cc;
          if (gc >= S.cols) continue;
          const int frow = synthesis ? gc : gr, coord = synthesis ? gr : gc;
          const int b2 = frow >> 1, e = frow & 1, f = coord & 1, q = coord >> 1;
          const int j = b2 / k, ki = b2 % k;
          if (q < j * w || q >= (j + 1) * w) continue;
          const int m = static_cast<int>((static_cast<int64_t>(ki) * q) % k);
          const double re = cs[m] * rk, im = sn[m] * rk;
          const double v = e == 0 ? (f == 0 ? re : im) : (f == 0 ? -im : re);
          const int pos = r * kTK + ((((cc >> 3) ^ (r & 7)) << 3) | (cc & 7));
          tile[pos] = bf16_bits(static_cast<float>(v));
        }
      }
    }
  }
}

struct FrameBuf {
  size_t Qa, QaT, Qb, QbT, perm, iperm, signs, ana_tiles, ana_idx, syn_tiles, syn_idx, total;
};

FrameBuf frame_buf(int k, int rho, int d, int a, int b) {
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
  const SparseShape A = sparse_shape(k, rho, d, false), S = sparse_shape(k, rho, d, true);
  L.ana_tiles = take(static_cast<size_t>(A.count) * kTileBytes);
  L.ana_idx = take(A.idx.size() * 4);
  L.syn_tiles = take(static_cast<size_t>(S.count) * kTileBytes);
  L.syn_idx = take(S.idx.size() * 4);
  L.total = off;
  return L;
}

bool valid_triple(int k, int rho, int d) {
  return k > 0 && rho >= 2 && rho % 2 == 0 && d > 0 && d % rho == 0 && k >= d / rho;
}

bool valid_frame(const fq_frame* f) {
  if (!f || !valid_triple(f->k, f->rho, f->d)) return false;
  if (!f->ana_tiles || !f->ana_idx || !f->syn_tiles || !f->syn_idx || f->ana_count <= 0 ||
      f->syn_count <= 0)
    return false;
  if (f->a == 0 && f->b == 0) return true;
  return f->a > 0 && f->b > 0 && static_cast<int64_t>(f->a) * f->b == f->d && f->Qa && f->QaT &&
         f->Qb && f->QbT && f->perm && f->iperm && f->signs;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

struct ImplWs {
  size_t v, s, total, group;
};

// the fused kernel's workspace (header, z, u), then the rotated tokens and the un-rotated output
ImplWs impl_ws(int M, int d_in, int n_in, int n_out, int d_out) {
  ImplWs L{};
  size_t off = decode_workspace_bytes(M, d_in, n_in, n_out, d_out);
  L.group = off;
  L.v = off;
  off += static_cast<size_t>(round_up(static_cast<int64_t>(M) * d_in * 2, 256));
  L.s = off;
  off += static_cast<size_t>(round_up(static_cast<int64_t>(M) * d_out * 2, 256));
  L.total = off;
  return L;
}

// a rotation CTA's column slots (b rounded up to a warp), reduction groups and threads
int rot_slots(int b) { return static_cast<int>(round_up(b, 32)); }
int rot_groups(int b, int nt) {
  return std::max(1, std::min(kRotMaxGroups, nt / rot_slots(b)));
}
int rot_threads(int b) {
  return rot_slots(b) * std::max(1, std::min(kRotMaxGroups, 1024 / rot_slots(b)));
}

size_t rot_smem_with(const fq_frame& f, int KG, bool staged) {
  const size_t bb = staged ? static_cast<size_t>(f.b) * f.b
                           : static_cast<size_t>(kRotBufs) * kRotChunk * f.b;
  return (static_cast<size_t>(round_up(f.d, 4)) + static_cast<size_t>(kRotRows) * (f.a + f.b) +
          static_cast<size_t>(KG) * kRotRows * rot_slots(f.b) + bb) *
         4;
}
// all of B in shared memory when it is small and leaves room for two CTAs per SM
bool rot_staged(const fq_frame& f, int KG) {
  return f.b <= kRotStageB && rot_smem_with(f, KG, true) <= kRotSmemStaged;
}
size_t rot_smem(const fq_frame& f, int KG) { return rot_smem_with(f, KG, rot_staged(f, KG)); }

constexpr size_t kMaxSmem = 227 * 1024;

bool frame_fits(const fq_frame& f) {
  if (ceil_div(static_cast<int64_t>(f.k) * f.rho, kTR) > kWsMaxTiles ||
      ceil_div(f.d, kTR) > kWsMaxTiles)
    return false;
  return f.a == 0 ||
         (f.b <= 1024 && rot_smem(f, rot_groups(f.b, rot_threads(f.b))) <= kMaxSmem);
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

// R^T x (analysis) or R s (synthesis) for M tokens of n layers in one launch, bf16 in and out;
// layers without a rotation are skipped
template <bool kSynth>
cudaError_t rotate_batch(int n, const fq_frame* const* f, const void* const* in,
                         void* const* out, int M, cudaStream_t s) {
  RotBatch rb{};
  int nb = 0, gx = 1, threads = 32;
  size_t smem = 0;
  for (int l = 0; l < n; ++l)
    if (f[l]->a != 0) threads = std::max(threads, rot_threads(f[l]->b));
  for (int l = 0; l < n; ++l) {
    if (f[l]->a == 0) continue;
    const fq_frame& F = *f[l];
    const int KG = rot_groups(F.b, threads);
    rb.L[nb] = RotLayer{static_cast<const __nv_bfloat16*>(in[l]), static_cast<__nv_bfloat16*>(out[l]),
                        F.d, F.a, F.b, rot_slots(F.b), KG, rot_staged(F, KG) ? 1 : 0,
                        kSynth ? F.Qa : F.QaT,
                        kSynth ? F.QbT : F.Qb, F.perm, F.iperm, F.signs};
    gx = std::max(gx, static_cast<int>(ceil_div(F.a, kRotRows)));
    smem = std::max(smem, rot_smem(F, KG));
    ++nb;
  }
  if (nb == 0) return cudaSuccess;
  return launch_pdl(rotate_kernel<kSynth>, dim3(static_cast<unsigned>(gx), M, nb), dim3(threads),
                    smem, s, rb);
}

template <bool kSynth>
cudaError_t rotate(const fq_frame& f, int M, const void* in, void* out, cudaStream_t s) {
  const fq_frame* fp = &f;
  return rotate_batch<kSynth>(1, &fp, &in, &out, M, s);
}

}  // namespace
}  // namespace fq

using namespace fq;

extern "C" {

size_t fq_frame_implicit_bytes(int k, int rho, int d, int a, int b) {
  if (!valid_triple(k, rho, d) || a < 0 || b < 0) return 0;
  if ((a == 0) != (b == 0) || (a > 0 && static_cast<int64_t>(a) * b != d)) return 0;
  return frame_buf(k, rho, d, a, b).total;
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
  const FrameBuf L = frame_buf(k, rho, d, a, b);
  if (!buf || bytes < L.total) return FQ_ERR_WORKSPACE;
  if ((reinterpret_cast<uintptr_t>(buf) & 255u) != 0) return FQ_ERR_ALIGNMENT;
  auto s = reinterpret_cast<cudaStream_t>(stream);
  char* base = static_cast<char*>(buf);
  // the two orientations of the un-rotated operator, tile by tile (host, double precision)
  std::vector<double> cs(k), sn(k);
  const double two_pi = 6.283185307179586476925286766559;
  for (int m = 0; m < k; ++m) {
    cs[m] = std::cos(two_pi * m / k);
    sn[m] = std::sin(two_pi * m / k);
  }
  const SparseShape SA = sparse_shape(k, rho, d, false), SS = sparse_shape(k, rho, d, true);
  std::vector<uint16_t> ta, ts;
  fill_tiles(k, rho, d, SA, false, cs, sn, ta);
  fill_tiles(k, rho, d, SS, true, cs, sn, ts);
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
  if (!up(L.ana_tiles, ta.data(), ta.size() * 2) || !up(L.ana_idx, SA.idx.data(), SA.idx.size() * 4) ||
      !up(L.syn_tiles, ts.data(), ts.size() * 2) || !up(L.syn_idx, SS.idx.data(), SS.idx.size() * 4) ||
      !up(L.Qa, qa.data(), qa.size() * 4) || !up(L.QaT, qat.data(), qat.size() * 4) ||
      !up(L.Qb, qb.data(), qb.size() * 4) || !up(L.QbT, qbt.data(), qbt.size() * 4) ||
      !up(L.signs, sg.data(), sg.size() * 4) || !up(L.perm, pm.data(), pm.size() * 4) ||
      !up(L.iperm, ipm.data(), ipm.size() * 4))
    return FQ_ERR_CUDA;
  // the host vectors are released on return: the copies from them must be complete
  if (cudaStreamSynchronize(s) != cudaSuccess) return FQ_ERR_CUDA;
  fq_frame f{};
  f.k = k;
  f.rho = rho;
  f.d = d;
  f.a = a;
  f.b = b;
  f.ana_tiles = reinterpret_cast<const uint8_t*>(base + L.ana_tiles);
  f.ana_idx = reinterpret_cast<const int32_t*>(base + L.ana_idx);
  f.ana_count = SA.count;
  f.syn_tiles = reinterpret_cast<const uint8_t*>(base + L.syn_tiles);
  f.syn_idx = reinterpret_cast<const int32_t*>(base + L.syn_idx);
  f.syn_count = SS.count;
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
  if (!aligned16(x) || !aligned16(y) || (gamma && !aligned16(gamma)) ||
      !aligned16(fi.ana_tiles) || !aligned16(fo.syn_tiles))
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
  void* v = fi.a > 0 ? static_cast<void*>(w + L.v) : const_cast<void*>(x);
  void* sy = fo.a > 0 ? static_cast<void*>(w + L.s) : y;
  if (fi.a > 0 && rotate<false>(fi, M, x, v, s) != cudaSuccess) return FQ_ERR_CUDA;
  DecGroupLayer g{v, fi.d, nullptr, *C, nullptr, fo.d, gamma, sy};
  g.tin = SparseOperand{fi.ana_tiles, fi.ana_idx, fi.ana_count};
  g.tout = SparseOperand{fo.syn_tiles, fo.syn_idx, fo.syn_count};
  const fq_status st = launch_decode_group(M, 1, &g, w, L.group, max_sms, false, nullptr, 0, 0, s);
  if (st != FQ_OK) return st;
  if (fo.a > 0 && rotate<true>(fo, M, sy, y, s) != cudaSuccess) return FQ_ERR_CUDA;
  return FQ_OK;
}


size_t fq_implicit_group_workspace_bytes(int M, int n_layers, const fq_implicit_layer* layers) {
  if (M <= 0 || M > kDecodeMaxM || n_layers < 1 || n_layers > FQ_MAX_GROUP || !layers) return 0;
  DecGroupLayer g[FQ_MAX_GROUP];
  size_t extra = 0;
  for (int l = 0; l < n_layers; ++l) {
    const fq_implicit_layer& L = layers[l];
    if (!L.C || !L.F_in || !L.F_out) return 0;
    g[l] = DecGroupLayer{nullptr, L.F_in->d, nullptr, *L.C, nullptr, L.F_out->d, nullptr, nullptr};
    extra += static_cast<size_t>(round_up(static_cast<int64_t>(M) * L.F_in->d * 2, 256)) +
             static_cast<size_t>(round_up(static_cast<int64_t>(M) * L.F_out->d * 2, 256));
  }
  const size_t base = decode_group_workspace_bytes(M, n_layers, g);
  return base == 0 ? 0 : base + extra;
}

fq_status fq_linear_forward_implicit_group(int M, int n_layers, const fq_implicit_layer* layers,
                                           void* ws, size_t ws_bytes, int max_sms,
                                           fq_stream_t stream) {
  if (!layers || n_layers < 1 || n_layers > FQ_MAX_GROUP || max_sms < 0 || M <= 0)
    return FQ_ERR_INVALID_ARG;
  for (int l = 0; l < n_layers; ++l) {
    const fq_implicit_layer& L = layers[l];
    if (!L.x || !L.y || !L.C) return FQ_ERR_INVALID_ARG;
    if (const fq_status cs = check_packed(L.C)) return cs;
    if (!valid_frame(L.F_in) || !valid_frame(L.F_out)) return FQ_ERR_INVALID_ARG;
    const fq_frame &fi = *L.F_in, &fo = *L.F_out;
    if (L.C->n_in != fi.k * fi.rho || L.C->n_out != fo.k * fo.rho) return FQ_ERR_INVALID_ARG;
    if (fi.d % 8 || fo.d % 8) return FQ_ERR_ALIGNMENT;
    if (!aligned16(L.x) || !aligned16(L.y) || (L.gamma && !aligned16(L.gamma)) ||
        !aligned16(fi.ana_tiles) || !aligned16(fo.syn_tiles))
      return FQ_ERR_ALIGNMENT;
    if (!frame_fits(fi) || !frame_fits(fo)) return FQ_ERR_UNSUPPORTED;
    for (int j = 0; j < n_layers; ++j)
      if (j != l && (layers[j].y == L.y || layers[j].x == L.y)) return FQ_ERR_INVALID_ARG;
    if (L.x == L.y) return FQ_ERR_INVALID_ARG;
  }
  if (M > kDecodeMaxM) return FQ_ERR_UNSUPPORTED;
  if (!ws) return FQ_ERR_WORKSPACE;
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return FQ_ERR_ALIGNMENT;
  const size_t need = fq_implicit_group_workspace_bytes(M, n_layers, layers);
  if (need == 0) return FQ_ERR_INVALID_ARG;
  if (ws_bytes < need) return FQ_ERR_WORKSPACE;
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
  // the fused kernel's workspace first, then every layer's rotated tokens and output
  DecGroupLayer g[FQ_MAX_GROUP];
  for (int l = 0; l < n_layers; ++l) {
    const fq_implicit_layer& L = layers[l];
    g[l] = DecGroupLayer{nullptr, L.F_in->d, nullptr, *L.C, nullptr, L.F_out->d, L.gamma, nullptr};
  }
  size_t off = decode_group_workspace_bytes(M, n_layers, g);
  const size_t group_bytes = off;
  for (int l = 0; l < n_layers; ++l) {
    const fq_implicit_layer& L = layers[l];
    const fq_frame &fi = *L.F_in, &fo = *L.F_out;
    void* v = fi.a > 0 ? static_cast<void*>(w + off) : const_cast<void*>(L.x);
    off += static_cast<size_t>(round_up(static_cast<int64_t>(M) * fi.d * 2, 256));
    void* sy = fo.a > 0 ? static_cast<void*>(w + off) : L.y;
    off += static_cast<size_t>(round_up(static_cast<int64_t>(M) * fo.d * 2, 256));
    g[l].x = v;
    g[l].y = sy;
    g[l].tin = SparseOperand{fi.ana_tiles, fi.ana_idx, fi.ana_count};
    g[l].tout = SparseOperand{fo.syn_tiles, fo.syn_idx, fo.syn_count};
  }
  const fq_frame* fin[FQ_MAX_GROUP];
  const fq_frame* fout[FQ_MAX_GROUP];
  const void* xin[FQ_MAX_GROUP];
  void* vout[FQ_MAX_GROUP];
  const void* sin_[FQ_MAX_GROUP];
  void* yout[FQ_MAX_GROUP];
  for (int l = 0; l < n_layers; ++l) {
    fin[l] = layers[l].F_in;
    fout[l] = layers[l].F_out;
    xin[l] = layers[l].x;
    vout[l] = const_cast<void*>(g[l].x);
    sin_[l] = g[l].y;
    yout[l] = layers[l].y;
  }
  if (rotate_batch<false>(n_layers, fin, xin, vout, M, s) != cudaSuccess) return FQ_ERR_CUDA;
  const fq_status st =
      launch_decode_group(M, n_layers, g, w, group_bytes, max_sms, false, nullptr, 0, 0, s);
  if (st != FQ_OK) return st;
  if (rotate_batch<true>(n_layers, fout, sin_, yout, M, s) != cudaSuccess) return FQ_ERR_CUDA;
  return FQ_OK;
}

}  // extern "C"
