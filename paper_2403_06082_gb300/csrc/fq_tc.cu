// FQ_BF16 path: the three products of the frame-quantized layer on the sm_103a tensor cores.
//
// Every phase is one persistent, warp-specialised kernel computing
//     out[t][i] = epilogue( sum_k A[i][k] * B[t][k] )      (i < R rows, t < M tokens)
// with the weight-side operand A as the 128-row MMA operand and the tokens as the N operand
// (N = BN in {16, ..., 256}), so one kernel serves decode (M <= 16) and prefill (M in the
// thousands).  Phases (Sec. 3.2):
//   analysis   A = T_in (n_in x d_in),  B = x,  out = z (bf16) and per-tile sums of z
//   core       A = 2-bit codes of C_hat (n_out x n_in) decoded to bf16 in shared memory,
//              B = z, out = u = gamma * (s * acc + zero * sum(z))   (bf16)
//   synthesis  A = T_out^T (d_out x n_out), B = u, out = y (bf16)
//
// Warp roles:  warp 0 TMA producer (one lane), warp 1 TMEM owner + MMA issuer (one lane),
//              warps 2-5 epilogue (thread = accumulator row), warps 6-9 code decoders (core).
// Operand tiles are 64 bf16 wide in K (one 128-byte swizzle atom) and staged through a ring
// of shared-memory stages guarded by mbarriers; accumulators are double-buffered in TMEM so
// the epilogue of one work unit overlaps the MMAs of the next.  Work units are (row tile,
// token tile, K split); when a tile's K range is split, fp32 partials go to the workspace and
// the last CTA to finish the tile (an atomic ticket, no spinning) reduces them in a fixed
// order and applies the epilogue.  Consecutive phases are chained with programmatic
// dependent launch: a dependent kernel starts on SMs as they free up, prefetches its weight
// operand into L2, and waits (griddepcontrol.wait) before it touches the previous phase's
// output.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <mutex>

#include "fq_device.cuh"
#include "fq_internal.h"

namespace fq {
namespace {

enum Phase : int { kAnalysis = 0, kCore = 1, kSynthesis = 2 };

constexpr int kBM = 128;                    // MMA M (rows of A per tile)
constexpr int kBK = 64;                     // K per stage (one 128-byte swizzle atom of bf16)
constexpr int kATileBytes = kBM * kBK * 2;  // 16 KiB
constexpr int kCodeBytes = kBM * kBK / 4;   // 2 KiB of packed codes per stage
constexpr int kMaxSplits = 16;
constexpr int kMaxSMs = 160;                // upper bound on SMs, for the workspace bound
constexpr int kMaxCounterTiles = 1024;
constexpr int kSmemBudget = 200 * 1024;

struct PhaseArgs {
  int R, K, M;
  int RT, TT, S, KB, kb_per_split, units;
  const uint32_t* words;     // core: packed codes
  __nv_bfloat16* out;        // [M][R]
  float* partial;            // [S][M][R] when S > 1
  unsigned* counters;        // [RT * TT] tickets when S > 1
  float* zsum_part;          // analysis writes [RT][M]; core reads [zsum_tiles][M]
  int zsum_tiles;
  const __half* scale;
  const __half* zero;
  const float* gamma;
  int32_t* status;
};

template <int BN>
struct Cfg {
  static constexpr int kBTileBytes = BN * kBK * 2;
  static constexpr int kStageBytes = kATileBytes + kBTileBytes + kCodeBytes;
  static constexpr int kStages = std::min(12, kSmemBudget / kStageBytes);
  static constexpr int kChunk = 16;                      // accumulator columns per TMEM load
  static constexpr uint32_t kTmemCols = 2 * BN < 32 ? 32 : 2 * BN;
};

template <int PHASE>
constexpr int threads_for() { return PHASE == kCore ? 320 : 192; }

template <int BN>
constexpr int smem_bytes_for() {
  // stages + barriers/bookkeeping + 1 KiB alignment slack
  return Cfg<BN>::kStages * Cfg<BN>::kStageBytes + 2048 + BN * 4 + 1024;
}

__device__ __forceinline__ void unit_coords(const PhaseArgs& p, int u, int& rt, int& tt,
                                            int& ks) {
  rt = u % p.RT;
  const int rest = u / p.RT;
  tt = rest % p.TT;
  ks = rest / p.TT;
}

// Decode 64 2-bit codes (4 words, layout of framequant.h) into 64 exact bf16 values and store
// them as one 128-byte row of a K-major tile with the 128-byte swizzle (16-byte chunk c of row
// r lands at chunk c ^ (r mod 8)).  q in {0..3} becomes bf16(128 + q) by placing q in the low
// mantissa bits of 128.0 (0x4300) and then 128 is subtracted exactly.
__device__ __forceinline__ void decode_row(const uint4 w4, uint8_t* tile, int r) {
  const uint32_t wv[4] = {w4.x, w4.y, w4.z, w4.w};
  const __nv_bfloat162 bias = __floats2bfloat162_rn(128.f, 128.f);
  uint8_t* row = tile + r * 128;
#pragma unroll
  for (int wi = 0; wi < 4; ++wi) {
    uint32_t h[8];
#pragma unroll
    for (int p = 0; p < 8; ++p) {
      const uint32_t bits = ((wv[wi] >> (2 * p)) & 0x00030003u) | 0x43004300u;
      __nv_bfloat162 v = *reinterpret_cast<const __nv_bfloat162*>(&bits);
      v = __hsub2(v, bias);
      h[p] = *reinterpret_cast<const uint32_t*>(&v);
    }
    // word wi holds columns 16 wi .. 16 wi + 15 = chunks 2 wi and 2 wi + 1
#pragma unroll
    for (int half = 0; half < 2; ++half) {
      const int c = 2 * wi + half;
      uint4 q = make_uint4(h[4 * half], h[4 * half + 1], h[4 * half + 2], h[4 * half + 3]);
      *reinterpret_cast<uint4*>(row + ((c ^ (r & 7)) << 4)) = q;
    }
  }
}

__device__ __forceinline__ bool bar_red_or(uint32_t id, uint32_t n, bool v) {
  uint32_t out;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "bar.red.or.pred q, %2, %3, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(out)
      : "r"(static_cast<uint32_t>(v)), "r"(id), "r"(n)
      : "memory");
  return out != 0;
}

template <int PHASE, int BN>
__global__ void __launch_bounds__(threads_for<PHASE>(), 1)
    tc_phase_kernel(const __grid_constant__ CUtensorMap tmA,
                    const __grid_constant__ CUtensorMap tmB, const PhaseArgs p) {
  using C = Cfg<BN>;
  constexpr int S_ = C::kStages;
  constexpr bool kCodes = PHASE == kCore;

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = sA + S_ * kATileBytes;
  uint8_t* sCodes = sB + S_ * C::kBTileBytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(sCodes + S_ * kCodeBytes);
  uint64_t* empty = full + S_;
  uint64_t* aready = empty + S_;
  uint64_t* tfull = aready + S_;
  uint64_t* tempty = tfull + 2;
  uint64_t* mma_done = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  int* ticket = reinterpret_cast<int*>(tmem_slot + 2);
  float* red = reinterpret_cast<float*>(tmem_slot + 4);       // [4][kChunk] cross-warp sums
  float* zsum_s = red + 4 * C::kChunk;                        // [BN] sum of z per token

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S_; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
      mbar_init(&aready[s], kBM);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], kBM);
    }
    mbar_init(mma_done, 1);
    *abort_flag = 0;
    fence_barrier_init();
    if (!kCodes) prefetch_tmap(&tmA);
    prefetch_tmap(&tmB);
  }
  if (warp == 1) tmem_alloc(tmem_slot, C::kTmemCols);
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem_base = *tmem_slot;

  // Let the next phase's CTAs launch as soon as SMs free up; they wait for this grid's
  // completion (griddepcontrol.wait) before reading what it writes.
  pdl_launch_dependents();

  const int first_unit = blockIdx.x;
  const int unit_step = gridDim.x;

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      const uint64_t pol_w = policy_evict_first();   // weights: streamed once
      const uint64_t pol_x = policy_evict_last();    // activations: re-read by other tiles
      if (PHASE != kAnalysis) {
        // Warm L2 with this CTA's first weight tiles while the previous phase finishes.
        if (first_unit < p.units) {
          int rt, tt, ks;
          unit_coords(p, first_unit, rt, tt, ks);
          const int k0 = ks * p.kb_per_split, k1 = min(p.KB, k0 + p.kb_per_split);
          for (int kb = k0; kb < k1; ++kb) {
            if (kCodes) {
              const uint32_t* src = p.words + (static_cast<int64_t>(rt) * p.KB + kb) * 512;
              asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src),
                           "r"(kCodeBytes)
                           : "memory");
            } else {
              asm volatile(
                  "cp.async.bulk.prefetch.tensor.2d.L2.global.tile [%0, {%1, %2}];" ::"l"(
                      reinterpret_cast<uint64_t>(&tmA)),
                  "r"(kb * kBK), "r"(rt * kBM)
                  : "memory");
            }
          }
        }
        pdl_wait();
      }
      int stage = 0;
      uint32_t phase = 0;
      uint32_t issued_parity[S_];
      bool issued[S_];
#pragma unroll
      for (int s = 0; s < S_; ++s) issued[s] = false, issued_parity[s] = 0;
      for (int u = first_unit; u < p.units && !*abort_flag; u += unit_step) {
        int rt, tt, ks;
        unit_coords(p, u, rt, tt, ks);
        const int k0 = ks * p.kb_per_split, k1 = min(p.KB, k0 + p.kb_per_split);
        for (int kb = k0; kb < k1; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1)) {
            report(p.status, FQ_ERR_TIMEOUT);
            *abort_flag = 1;
            break;
          }
          if (kCodes) {
            mbar_arrive_expect_tx(&full[stage], kCodeBytes + C::kBTileBytes);
            bulk_load(sCodes + stage * kCodeBytes,
                      p.words + (static_cast<int64_t>(rt) * p.KB + kb) * 512, kCodeBytes,
                      &full[stage], pol_w);
          } else {
            mbar_arrive_expect_tx(&full[stage], kATileBytes + C::kBTileBytes);
            tma_load_2d(sA + stage * kATileBytes, &tmA, &full[stage], kb * kBK, rt * kBM,
                        pol_w);
          }
          tma_load_2d(sB + stage * C::kBTileBytes, &tmB, &full[stage], kb * kBK, tt * BN,
                      pol_x);
          issued[stage] = true;
          issued_parity[stage] = phase;
          if (++stage == S_) stage = 0, phase ^= 1;
        }
      }
      // Never leave with copies in flight: wait (bounded) for the last round of each stage.
      for (int s = 0; s < S_; ++s)
        if (issued[s] && !mbar_wait(&full[s], issued_parity[s])) report(p.status, FQ_ERR_TIMEOUT);
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = umma_idesc_bf16(kBM, BN);
      int stage = 0;
      uint32_t phase = 0;
      int buf = 0;
      uint32_t acc_phase = 0;
      bool issued_any = false;
      for (int u = first_unit; u < p.units && !*abort_flag; u += unit_step) {
        int rt, tt, ks;
        unit_coords(p, u, rt, tt, ks);
        const int k0 = ks * p.kb_per_split, k1 = min(p.KB, k0 + p.kb_per_split);
        if (!mbar_wait(&tempty[buf], acc_phase ^ 1)) {
          report(p.status, FQ_ERR_TIMEOUT);
          *abort_flag = 1;
          break;
        }
        tc_fence_after_sync();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(buf * BN);
        bool ok = true;
        for (int kb = k0; kb < k1; ++kb) {
          ok = mbar_wait(&full[stage], phase) && (!kCodes || mbar_wait(&aready[stage], phase));
          if (!ok) break;
          tc_fence_after_sync();
          const uint64_t adesc = umma_desc_sw128(smem_u32(sA + stage * kATileBytes));
          const uint64_t bdesc = umma_desc_sw128(smem_u32(sB + stage * C::kBTileBytes));
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k) {
            // advance 16 bf16 = 32 bytes along K inside the swizzle atom
            umma_bf16(d_tmem, adesc + 2 * k, bdesc + 2 * k, idesc,
                      (kb > k0 || k > 0) ? 1u : 0u);
          }
          issued_any = true;
          umma_commit(&empty[stage]);
          if (++stage == S_) stage = 0, phase ^= 1;
        }
        if (!ok) {
          report(p.status, FQ_ERR_TIMEOUT);
          *abort_flag = 1;
          break;
        }
        umma_commit(&tfull[buf]);
        if (++buf == 2) buf = 0, acc_phase ^= 1;
      }
      // Drain: every MMA issued has completed before the TMEM is released.
      if (issued_any) {
        umma_commit(mma_done);
        if (!mbar_wait(mma_done, 0)) report(p.status, FQ_ERR_TIMEOUT);
      }
    }
  } else if (warp < 6) {
    // ---------------------------------------------------------------- epilogue (rows)
    const int quarter = warp & 3;                 // TMEM lanes 32*quarter .. +31
    const int r_in_tile = quarter * 32 + lane;
    const int et = threadIdx.x - 64;              // 0..127 within the epilogue group
    const int ew = warp - 2;
    if (PHASE != kAnalysis) pdl_wait();
    int buf = 0;
    uint32_t acc_phase = 0;
    for (int u = first_unit; u < p.units; u += unit_step) {
      int rt, tt, ks;
      unit_coords(p, u, rt, tt, ks);
      const int row = rt * kBM + r_in_tile;
      const int t0 = tt * BN;
      const bool row_ok = row < p.R;
      float s_i = 0.f, z_i = 0.f, g_i = 1.f;
      if (PHASE == kCore && row_ok) {
        s_i = __half2float(p.scale[row]);
        z_i = __half2float(p.zero[row]);
        if (p.gamma) g_i = p.gamma[row];
      }
      const bool fail = !mbar_wait(&tfull[buf], acc_phase);
      if (fail) report(p.status, FQ_ERR_TIMEOUT);
      if (bar_red_or(1, 128, fail || *abort_flag)) {
        if (threadIdx.x == 64) *abort_flag = 1;
        break;
      }
      tc_fence_after_sync();
      const uint32_t t_row = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) +
                             static_cast<uint32_t>(buf * BN);

      // Final value of this thread's row for tokens t0 + c .. + kChunk - 1 -> epilogue, store.
      auto finish_chunk = [&](int c, const float (&acc)[C::kChunk]) {
        float v[C::kChunk];
#pragma unroll
        for (int j = 0; j < C::kChunk; ++j) {
          float a = acc[j];
          if (PHASE == kCore) a = g_i * fmaf(s_i, a, z_i * zsum_s[c + j]);
          v[j] = a;
        }
#pragma unroll
        for (int j = 0; j < C::kChunk; ++j) {
          const int t = t0 + c + j;
          const __nv_bfloat16 b = __float2bfloat16_rn(v[j]);
          v[j] = __bfloat162float(b);
          if (row_ok && t < p.M) p.out[static_cast<int64_t>(t) * p.R + row] = b;
        }
        if (PHASE == kAnalysis) {
          // per-token sum over the tile's 128 rows of the bf16 z actually stored
#pragma unroll
          for (int j = 0; j < C::kChunk; ++j) {
            float s = row_ok ? v[j] : 0.f;
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
            v[j] = s;
          }
          if (lane == 0) {
#pragma unroll
            for (int j = 0; j < C::kChunk; ++j) red[ew * C::kChunk + j] = v[j];
          }
          named_barrier_sync(1, 128);
          if (et < C::kChunk) {
            const int t = t0 + c + et;
            // fixed order over the four warps (TMEM quarters 2, 3, 0, 1 -> rows 64.., 96.., 0.., 32..)
            const float s = (red[2 * C::kChunk + et] + red[3 * C::kChunk + et]) +
                            (red[0 * C::kChunk + et] + red[1 * C::kChunk + et]);
            if (t < p.M) p.zsum_part[static_cast<int64_t>(rt) * p.M + t] = s;
          }
          named_barrier_sync(1, 128);
        }
      };

      if (PHASE == kCore) {
        // sum_j z[t][j] for the tile's tokens, from the analysis phase's per-tile sums
        named_barrier_sync(1, 128);
        for (int j = et; j < BN; j += 128) {
          const int t = t0 + j;
          float s = 0.f;
          if (t < p.M)
            for (int q = 0; q < p.zsum_tiles; ++q)
              s += ldcg_f32(p.zsum_part + static_cast<int64_t>(q) * p.M + t);
          zsum_s[j] = s;
        }
        named_barrier_sync(1, 128);
      }

      if (p.S == 1) {
#pragma unroll 1
        for (int c = 0; c < BN; c += C::kChunk) {
          float acc[C::kChunk];
          tmem_ld16(t_row + c, acc);
          tmem_wait_ld();
          finish_chunk(c, acc);
        }
        tc_fence_before_sync();
        mbar_arrive(&tempty[buf]);
      } else {
        float* part = p.partial + static_cast<int64_t>(ks) * p.M * p.R;
#pragma unroll 1
        for (int c = 0; c < BN; c += C::kChunk) {
          float acc[C::kChunk];
          tmem_ld16(t_row + c, acc);
          tmem_wait_ld();
#pragma unroll
          for (int j = 0; j < C::kChunk; ++j) {
            const int t = t0 + c + j;
            if (row_ok && t < p.M) part[static_cast<int64_t>(t) * p.R + row] = acc[j];
          }
        }
        tc_fence_before_sync();
        mbar_arrive(&tempty[buf]);
        __threadfence();
        named_barrier_sync(1, 128);
        if (et == 0) {
          const unsigned old = atomicInc(&p.counters[rt * p.TT + tt], static_cast<unsigned>(p.S - 1));
          *ticket = (old == static_cast<unsigned>(p.S - 1)) ? 1 : 0;
        }
        named_barrier_sync(1, 128);
        if (*ticket) {
          __threadfence();
#pragma unroll 1
          for (int c = 0; c < BN; c += C::kChunk) {
            float acc[C::kChunk];
#pragma unroll
            for (int j = 0; j < C::kChunk; ++j) {
              const int t = t0 + c + j;
              float s = 0.f;
              if (row_ok && t < p.M)
                for (int q = 0; q < p.S; ++q)
                  s += ldcg_f32(p.partial + (static_cast<int64_t>(q) * p.M + t) * p.R + row);
              acc[j] = s;
            }
            finish_chunk(c, acc);
          }
        }
      }
      if (++buf == 2) buf = 0, acc_phase ^= 1;
    }
  } else {
    // ---------------------------------------------------------------- code decoders (core)
    if (kCodes) {
      const int r = threadIdx.x - 192;    // row of the tile this thread decodes
      int stage = 0;
      uint32_t phase = 0;
      for (int u = first_unit; u < p.units && !*abort_flag; u += unit_step) {
        int rt, tt, ks;
        unit_coords(p, u, rt, tt, ks);
        const int k0 = ks * p.kb_per_split, k1 = min(p.KB, k0 + p.kb_per_split);
        bool ok = true;
        for (int kb = k0; kb < k1; ++kb) {
          if (!mbar_wait(&full[stage], phase)) {
            ok = false;
            break;
          }
          const uint4 w4 = reinterpret_cast<const uint4*>(sCodes + stage * kCodeBytes)[r];
          decode_row(w4, sA + stage * kATileBytes, r);
          fence_proxy_async_smem();
          mbar_arrive(&aready[stage]);
          if (++stage == S_) stage = 0, phase ^= 1;
        }
        if (!ok) {
          report(p.status, FQ_ERR_TIMEOUT);
          *abort_flag = 1;
          break;
        }
      }
    }
  }

  tc_fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after_sync();
    tmem_dealloc(tmem_base, C::kTmemCols);
  }
}

// ---------------------------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------------------------
PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000,
                                         cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  });
  return fn;
}

// bf16 matrix rows x cols (row-major), boxes of 64 columns x box_rows rows, 128-byte swizzle.
bool make_tmap(CUtensorMap* m, const void* base, int64_t rows, int64_t cols, int box_rows) {
  auto enc = get_encode();
  if (!enc) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(cols) * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(kBK), static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
             estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int pick_bn(int M) {
  if (M <= 16) return 16;
  if (M <= 32) return 32;
  if (M <= 64) return 64;
  if (M <= 128) return 128;
  return 256;
}

// Largest split count the planner may choose (also sizes the workspace, so it must not
// depend on the device).
int max_splits(int RT, int TT, int KB) {
  if (static_cast<int64_t>(RT) * TT >= kMaxSMs) return 1;
  return std::max(1, std::min(kMaxSplits, KB));
}

// Split K so that RT*TT*S units spread evenly over the SMs: minimise the busiest CTA's
// K blocks plus a fixed per-unit overhead.
void plan_phase(PhaseArgs& a, int R, int K, int M, int BN, int sms) {
  a.R = R;
  a.K = K;
  a.M = M;
  a.RT = static_cast<int>(ceil_div(R, kBM));
  a.TT = static_cast<int>(ceil_div(M, BN));
  a.KB = static_cast<int>(ceil_div(K, kBK));
  const int base = a.RT * a.TT;
  const int smax = std::min(max_splits(a.RT, a.TT, a.KB), a.KB);
  int best_s = 1;
  double best = 1e30;
  for (int s = 1; s <= smax; ++s) {
    const int kbs = static_cast<int>(ceil_div(a.KB, s));
    const int seff = static_cast<int>(ceil_div(a.KB, kbs));
    if (seff != s) continue;
    const double waves = static_cast<double>(ceil_div(static_cast<int64_t>(base) * s, sms));
    const double cost = waves * (kbs + 3.0) + (s > 1 ? 2.0 : 0.0);
    if (cost < best - 1e-9) best = cost, best_s = s;
  }
  a.S = best_s;
  a.kb_per_split = static_cast<int>(ceil_div(a.KB, best_s));
  a.units = base * best_s;
}

struct WsLayout {
  size_t counters, z, u, zsum, partial, total;
};

WsLayout ws_layout(int M, int d_in, int n_in, int n_out, int d_out) {
  WsLayout L{};
  const int BN = pick_bn(M);
  const int TT = static_cast<int>(ceil_div(M, BN));
  size_t off = kWsHeader;
  L.counters = off;
  off += round_up(3 * kMaxCounterTiles * sizeof(unsigned), 256);
  L.z = off;
  off += round_up(static_cast<int64_t>(M) * n_in * 2, 256);
  L.u = off;
  off += round_up(static_cast<int64_t>(M) * n_out * 2, 256);
  L.zsum = off;
  off += round_up(ceil_div(n_in, kBM) * M * 4, 256);
  L.partial = off;
  const int R[3] = {n_in, n_out, d_out};
  const int K[3] = {d_in, n_in, n_out};
  int64_t part = 0;
  for (int ph = 0; ph < 3; ++ph) {
    const int RT = static_cast<int>(ceil_div(R[ph], kBM));
    const int KB = static_cast<int>(ceil_div(K[ph], kBK));
    const int s = max_splits(RT, TT, KB);
    if (s > 1) part = std::max<int64_t>(part, static_cast<int64_t>(s) * M * R[ph] * 4);
  }
  off += round_up(part, 256);
  L.total = off;
  return L;
}

int device_sms() {
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  return sms > 0 ? sms : 148;
}

template <int PHASE, int BN>
cudaError_t launch_phase(const CUtensorMap& tmA, const CUtensorMap& tmB, const PhaseArgs& a,
                         int sms, bool pdl, cudaStream_t s) {
  auto kern = tc_phase_kernel<PHASE, BN>;
  constexpr int smem = smem_bytes_for<BN>();
  static bool attr_set = false;   // per instantiation; harmless to repeat
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(static_cast<unsigned>(std::min(a.units, sms)));
  cfg.blockDim = dim3(threads_for<PHASE>());
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kern, tmA, tmB, a);
}

// maps: {T_in, x, z, T_out^T, u}.  The core phase's A operand is the packed codes, so it gets
// an unused map in that slot.
template <int BN>
cudaError_t launch_all(const CUtensorMap* maps, PhaseArgs* a, int sms, cudaStream_t s) {
  cudaError_t e = launch_phase<kAnalysis, BN>(maps[0], maps[1], a[0], sms, false, s);
  if (e != cudaSuccess) return e;
  e = launch_phase<kCore, BN>(maps[1], maps[2], a[1], sms, true, s);   // A map unused
  if (e != cudaSuccess) return e;
  return launch_phase<kSynthesis, BN>(maps[3], maps[4], a[2], sms, true, s);
}

}  // namespace

size_t tc_workspace_bytes(int M, int d_in, int n_in, int n_out, int d_out) {
  return ws_layout(M, d_in, n_in, n_out, d_out).total;
}

fq_status launch_tc_forward(const void* x, int M, int d_in, const void* T_in,
                            const fq_packed& Cq, const void* T_out_t, int d_out,
                            const float* gamma, void* y, char* ws, size_t ws_bytes,
                            cudaStream_t s) {
  const int n_in = Cq.n_in, n_out = Cq.n_out;
  const WsLayout L = ws_layout(M, d_in, n_in, n_out, d_out);
  if (ws_bytes < L.total) return FQ_ERR_WORKSPACE;
  const int BN = pick_bn(M);
  const int sms = device_sms();
  auto* status = reinterpret_cast<int32_t*>(ws);
  auto* counters = reinterpret_cast<unsigned*>(ws + L.counters);
  auto* z = reinterpret_cast<__nv_bfloat16*>(ws + L.z);
  auto* u = reinterpret_cast<__nv_bfloat16*>(ws + L.u);
  auto* zsum = reinterpret_cast<float*>(ws + L.zsum);
  auto* partial = reinterpret_cast<float*>(ws + L.partial);

  PhaseArgs a[3];
  const int R[3] = {n_in, n_out, d_out};
  const int K[3] = {d_in, n_in, n_out};
  __nv_bfloat16* outs[3] = {z, u, reinterpret_cast<__nv_bfloat16*>(y)};
  for (int ph = 0; ph < 3; ++ph) {
    a[ph] = PhaseArgs{};
    plan_phase(a[ph], R[ph], K[ph], M, BN, sms);
    if (a[ph].S > 1 && a[ph].RT * a[ph].TT > kMaxCounterTiles) return FQ_ERR_UNSUPPORTED;
    a[ph].out = outs[ph];
    a[ph].partial = partial;
    a[ph].counters = counters + ph * kMaxCounterTiles;
    a[ph].zsum_part = zsum;
    a[ph].zsum_tiles = static_cast<int>(ceil_div(n_in, kBM));
    a[ph].status = status;
  }
  a[1].words = Cq.words;
  a[1].scale = reinterpret_cast<const __half*>(Cq.scale);
  a[1].zero = reinterpret_cast<const __half*>(Cq.zero);
  a[1].gamma = gamma;

  // maps: T_in, x, z, T_out^T, u  (A maps use 128-row boxes, B maps BN-row boxes)
  CUtensorMap maps[5];
  if (!make_tmap(&maps[0], T_in, n_in, d_in, kBM) || !make_tmap(&maps[1], x, M, d_in, BN) ||
      !make_tmap(&maps[2], z, M, n_in, BN) || !make_tmap(&maps[3], T_out_t, d_out, n_out, kBM) ||
      !make_tmap(&maps[4], u, M, n_out, BN))
    return FQ_ERR_CUDA;
  if (cudaMemsetAsync(ws, 0, L.z, s) != cudaSuccess) return FQ_ERR_CUDA;

  cudaError_t e;
  switch (BN) {
    case 16: e = launch_all<16>(maps, a, sms, s); break;
    case 32: e = launch_all<32>(maps, a, sms, s); break;
    case 64: e = launch_all<64>(maps, a, sms, s); break;
    case 128: e = launch_all<128>(maps, a, sms, s); break;
    default: e = launch_all<256>(maps, a, sms, s); break;
  }
  return e == cudaSuccess ? FQ_OK : FQ_ERR_CUDA;
}

}  // namespace fq
