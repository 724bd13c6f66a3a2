// FQ_BF16 path: the three products of the frame-quantized layer on the sm_103a tensor cores.
//
// Every phase is one persistent, warp-specialised kernel computing
//     out[t][i] = epilogue( sum_k A[i][k] * B[t][k] )      (i < R rows, t < M tokens)
// with the weight-side operand A as the 128-row MMA operand and the tokens as the N operand
// (N = BN = 128 or 256).  It serves batches of more than 64 tokens (prefill); smaller ones take
// the fused decode kernel.  Phases (Sec. 3.2):
//   analysis   A = T_in (n_in x d_in),  B = x,  out = z (bf16)
//   core       A = 2-bit codes of C_hat (n_out x n_in) decoded to bf16 in shared memory,
//              B = z, out = u = gamma * (s * acc + zero * sum(z))   (bf16)
//   synthesis  A = T_out^T (d_out x n_out), B = u, out = y (bf16)
//
// Warp roles:  warp 0 TMA producer (one lane), warp 1 TMEM owner + MMA issuer (one lane),
//              warps 2-5 epilogue (thread = accumulator row), warps 6-9 code decoders (core).
// Operand tiles are 64 bf16 wide in K (one 128-byte swizzle atom) and staged through a ring
// of shared-memory stages guarded by mbarriers; accumulators are double-buffered in TMEM so
// the epilogue of one tile overlaps the MMAs of the next.
//
// Tiles are numbered token tile fastest (tile = row tile * TT + token tile) and CTA c takes tiles
// c, c + grid, ...: the CTAs of a wave share each weight tile across all token tiles, so a
// weight matrix larger than L2 (T_out^T of the up and gate layers, 267 MB) streams from HBM
// once per wave instead of once per token tile (measured 8.7% faster on the 2048-token block).
//
// sum(z), needed by the core's zero term, comes from the analysis epilogue as one sum per
// 128-row tile of z and token, taken over the bf16 values stored.  Decoder warps take whole
// stages in turn (stage i goes to warp i mod 4), so four stages are decoded at once.
//
// The three phases are chained with programmatic dependent launch (the analysis kernel too,
// so consecutive layers chain as well): a kernel's CTAs start on SMs as they free up, load
// weight tiles that do not depend on the previous kernel, and wait (griddepcontrol.wait)
// before reading activations or writing anything the previous kernel may still read.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <map>
#include <mutex>
#include <utility>

#include "fq_device.cuh"
#include "fq_internal.h"
#include "framequant_dense.h"

namespace fq {
namespace {

enum Phase : int { kAnalysis = 0, kCore = 1, kSynthesis = 2 };

constexpr int kBM = 128;                    // MMA M (rows of A per tile)
constexpr int kBK = 64;                     // K per stage (one 128-byte swizzle atom of bf16)
constexpr int kATileBytes = kBM * kBK * 2;  // 16 KiB
constexpr int kCodeBytes = kBM * kBK / 4;   // 2 KiB of packed codes per stage
constexpr int kSmemBudget = 200 * 1024;
constexpr int kEpi = 128;                   // epilogue threads
constexpr int kChunk = 16;                  // accumulator columns per TMEM load

struct PhaseArgs {
  int R, K, M;
  int RT, TT, KB, tiles;
  int KS, kbs, units;        // K splits per tile, K blocks per split, tiles * KS work units
  float* part;               // KS > 1: fp32 partial tiles [tile][split][BN][128]
  uint32_t* cnt;             // KS > 1: arrivals per tile (the last resets it to 0)
  const uint32_t* words;     // core: packed codes
  __nv_bfloat16* out;        // [M][R]
  float* zsum_part;          // analysis writes [RT][M] sums of z; the core reads them
  int zsum_tiles;
  const __half* scale;
  const __half* zero;
  const float* gamma;
  int32_t* status;
  // Rounding of the frame representation of the activations (Appendix F), else all null:
  float* out32;              // analysis: z in fp32 (the bf16 z is then the rounded one)
  uint32_t* amax;            // analysis: running max |z| as float bits; the core resets it
  const float* delta;        // core: the rounding step Delta, which scales the product
};

template <int PHASE, int BN>
struct Layout {
  static constexpr bool kCodes = PHASE == kCore;
  static constexpr int kBTileBytes = BN * kBK * 2;
  static constexpr int kCodesStage = kCodes ? kCodeBytes : 0;
  static constexpr int kStageBytes = kATileBytes + kBTileBytes + kCodesStage;
  // Code rounds are decoded by warp (round mod 4), which waits for a stage's codes only in the
  // rounds it owns; that is exact only when every phase of a stage's barrier belongs to the
  // same warp, i.e. when the ring depth is a multiple of 4.
  static constexpr int kStagesRaw = std::min(12, kSmemBudget / kStageBytes);
  static constexpr int kStages = kCodes ? (kStagesRaw & ~3) : kStagesRaw;
  // double-buffered accumulators [0, 2 BN)
  static constexpr int kAccCols = 2 * BN;
  static constexpr uint32_t kTmemCols = kAccCols <= 256 ? 256 : 512;
  // byte offsets from the 1024-aligned base
  static constexpr int oA = 0;
  static constexpr int oB = oA + kStages * kATileBytes;
  static constexpr int oCodes = oB + kStages * kBTileBytes;
  static constexpr int oBar = oCodes + kStages * kCodesStage;
  static constexpr int kNumBars = 4 * kStages + 2 + 2 + 1;
  static constexpr int oMisc = oBar + kNumBars * 8;
  static constexpr int oRedSmall = oMisc + 16;                      // [4][kChunk] + 4 floats
  static constexpr int oZsum = oRedSmall + (4 * kChunk + 4) * 4;    // [2][BN] floats
  static constexpr int kBytes = oZsum + 2 * BN * 4 + 1024;          // + alignment slack
  static_assert(BN == 128 || BN == 256, "prefill tile widths");
  static_assert(kBTileBytes % 1024 == 0, "B tiles must keep 1024-byte alignment");
  static_assert(kBytes <= 227 * 1024, "shared memory");
  static_assert(kStages >= 2 && (!kCodes || kStages % 4 == 0), "ring depth");
};

template <int PHASE>
constexpr int threads_for() { return PHASE == kCore ? 320 : 192; }

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
  using Lo = Layout<PHASE, BN>;
  constexpr int S_ = Lo::kStages;
  constexpr bool kCodes = Lo::kCodes;
  constexpr int kBTile = Lo::kBTileBytes;

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem + Lo::oA;
  uint8_t* sB = smem + Lo::oB;
  uint8_t* sCodes = smem + Lo::oCodes;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + Lo::oBar);   // A (+B) landed / B landed
  uint64_t* empty = full + S_;      // stage consumed by the MMAs
  uint64_t* aready = empty + S_;    // decoded A tile written (core)
  uint64_t* cfull = aready + S_;    // codes landed (core)
  uint64_t* tfull = cfull + S_;     // accumulator ready
  uint64_t* tempty = tfull + 2;     // accumulator drained
  uint64_t* mma_done = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + Lo::oMisc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  float* red = reinterpret_cast<float*>(smem + Lo::oRedSmall);     // [4][kChunk], flag
  float* zsum_s = reinterpret_cast<float*>(smem + Lo::oZsum);      // [2][BN]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t cid = blockIdx.x, ncl = gridDim.x;
  // work unit u = split * tiles + tile: K blocks [split * kbs, min(KB, (split + 1) * kbs))
  auto unit_tile = [&](int u) { return u % p.tiles; };
  auto unit_k0 = [&](int u) { return (u / p.tiles) * p.kbs; };
  auto unit_k1 = [&](int u) { return min(p.KB, (u / p.tiles + 1) * p.kbs); };

  if (threadIdx.x == 0) {
    for (int s = 0; s < S_; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
      mbar_init(&aready[s], 32);     // one decoder warp per stage
      mbar_init(&cfull[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], kEpi);
    }
    mbar_init(mma_done, 1);
    *abort_flag = 0;
    fence_barrier_init();
    if (!kCodes) prefetch_tmap(&tmA);
    prefetch_tmap(&tmB);
  }
  if (warp == 1) tmem_alloc(tmem_slot, Lo::kTmemCols);
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem_base = *tmem_slot;

  // Let the next kernel's CTAs launch as soon as SMs free up; they wait for this grid's
  // completion (griddepcontrol.wait) before reading what it writes.
  pdl_launch_dependents();

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      const uint64_t pol_w = policy_evict_first();   // weights: streamed once
      const uint64_t pol_x = policy_evict_last();    // activations: re-read by other tiles
      // Weight tiles of the first tile do not depend on the previous kernel: issue up to a
      // full ring of them before waiting for it, and warm L2 with the rest.
      int pre = 0;
      if (static_cast<int>(cid) < p.units) {
        const int rt = unit_tile(static_cast<int>(cid)) / p.TT;
        const int k0 = unit_k0(static_cast<int>(cid)), k1 = unit_k1(static_cast<int>(cid));
        pre = min(S_, k1 - k0);
        for (int i = 0; i < pre; ++i) {
          const int kb = k0 + i;
          if (kCodes) {
            mbar_arrive_expect_tx(&cfull[i], kCodeBytes);
            bulk_load(sCodes + i * kCodeBytes,
                      p.words + (static_cast<int64_t>(rt) * p.KB + kb) * 512, kCodeBytes,
                      &cfull[i], pol_w);
          } else {
            mbar_arrive_expect_tx(&full[i], kATileBytes + kBTile);
            tma_load_2d(sA + i * kATileBytes, &tmA, &full[i], kb * kBK, rt * kBM, pol_w);
          }
        }
        for (int kb = k0 + pre; kb < k1; ++kb) {
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
      pdl_wait();   // the previous kernel is complete and its writes are visible
      if (PHASE == kAnalysis && blockIdx.x == 0) *p.status = 0;   // new call: clear status
      // the rounding kernel before this one has read the maximum: ready for the next call
      if (PHASE == kCore && p.amax && blockIdx.x == 0) *p.amax = 0u;
      int stage = 0;
      uint32_t phase = 0;
      int it = 0;
      uint32_t issued_parity[S_];
      bool issued[S_];
#pragma unroll
      for (int s = 0; s < S_; ++s) issued[s] = false, issued_parity[s] = 0;
      for (int unit = static_cast<int>(cid); unit < p.units && !*abort_flag;
           unit += static_cast<int>(ncl)) {
        const int tile = unit_tile(unit), k0 = unit_k0(unit), k1 = unit_k1(unit);
        const int rt = tile / p.TT, tt = tile % p.TT;
        for (int kb = k0; kb < k1; ++kb, ++it) {
          if (it >= pre) {
            if (!mbar_wait(&empty[stage], phase ^ 1, abort_flag)) {
              report(p.status, FQ_ERR_TIMEOUT);
              *abort_flag = 1;
              break;
            }
            if (kCodes) {
              mbar_arrive_expect_tx(&cfull[stage], kCodeBytes);
              bulk_load(sCodes + stage * kCodeBytes,
                        p.words + (static_cast<int64_t>(rt) * p.KB + kb) * 512, kCodeBytes,
                        &cfull[stage], pol_w);
            } else {
              mbar_arrive_expect_tx(&full[stage], kATileBytes + kBTile);
              tma_load_2d(sA + stage * kATileBytes, &tmA, &full[stage], kb * kBK, rt * kBM,
                          pol_w);
            }
          }
          if (kCodes) mbar_arrive_expect_tx(&full[stage], kBTile);
          tma_load_2d(sB + stage * kBTile, &tmB, &full[stage], kb * kBK, tt * BN, pol_x);
          issued[stage] = true;
          issued_parity[stage] = phase;
          if (++stage == S_) stage = 0, phase ^= 1;
        }
      }
      // Never leave with copies in flight: wait (bounded) for the last round of each stage.
      for (int s = 0; s < S_; ++s) {
        if (!issued[s]) continue;
        if (!mbar_wait(&full[s], issued_parity[s], nullptr) ||
            (kCodes && !mbar_wait(&cfull[s], issued_parity[s], nullptr)))
          report(p.status, FQ_ERR_TIMEOUT);
      }
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
      for (int unit = static_cast<int>(cid); unit < p.units && !*abort_flag;
           unit += static_cast<int>(ncl)) {
        const int k0 = unit_k0(unit), k1 = unit_k1(unit);
        if (!mbar_wait(&tempty[buf], acc_phase ^ 1, abort_flag)) {
          report(p.status, FQ_ERR_TIMEOUT);
          *abort_flag = 1;
          break;
        }
        tc_fence_after_sync();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(buf * BN);
        bool ok = true;
        for (int kb = k0; kb < k1; ++kb) {
          ok = mbar_wait(&full[stage], phase, abort_flag) &&
               (!kCodes || mbar_wait(&aready[stage], phase, abort_flag));
          if (!ok) break;
          tc_fence_after_sync();
          const uint64_t adesc = umma_desc_sw128(smem_u32(sA + stage * kATileBytes));
          const uint64_t bdesc = umma_desc_sw128(smem_u32(sB + stage * kBTile));
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k)   // 16 bf16 = 32 bytes along K per step
            umma_bf16(d_tmem, adesc + 2 * k, bdesc + 2 * k, idesc, (kb > k0 || k > 0) ? 1u : 0u);
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
        if (!mbar_wait(mma_done, 0, nullptr)) report(p.status, FQ_ERR_TIMEOUT);
      }
    }
  } else if (warp < 6) {
    // ---------------------------------------------------------------- epilogue (rows)
    const int quarter = warp & 3;                 // TMEM lanes 32*quarter .. +31
    const int r_in_tile = quarter * 32 + lane;
    const int et = threadIdx.x - 64;              // 0..127 within the epilogue group
    const int ew = warp - 2;
    pdl_wait();
    int buf = 0;
    uint32_t acc_phase = 0;
    for (int unit = static_cast<int>(cid); unit < p.units; unit += static_cast<int>(ncl)) {
      const int tile = unit_tile(unit), split = unit / p.tiles;
      const int rt = tile / p.TT, tt = tile % p.TT;
      const int row = rt * kBM + r_in_tile;
      const int t0 = tt * BN;
      const bool row_ok = row < p.R;
      float s_i = 0.f, z_i = 0.f;
      if (PHASE == kCore && row_ok) {
        s_i = __half2float(p.scale[row]);
        z_i = __half2float(p.zero[row]);
      }
      if (PHASE == kCore) {
        // sum_j z[t][j] for the tile's tokens, from the analysis phase's per-tile sums
        named_barrier_sync(1, kEpi);
        for (int q = et; q < BN; q += kEpi) {
          const int t = t0 + q;
          float s = 0.f;
          if (t < p.M)
            for (int g = 0; g < p.zsum_tiles; ++g)
              s += ldcg_f32(p.zsum_part + static_cast<int64_t>(g) * p.M + t);
          zsum_s[buf * BN + q] = s;
        }
        named_barrier_sync(1, kEpi);
      }
      const bool fail = !mbar_wait(&tfull[buf], acc_phase, abort_flag);
      if (fail) report(p.status, FQ_ERR_TIMEOUT);
      if (bar_red_or(1, kEpi, fail || *abort_flag)) {
        if (et == 0) *abort_flag = 1;
        break;
      }
      tc_fence_after_sync();
      const uint32_t t_row = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) +
                             static_cast<uint32_t>(buf * BN);
      const float* zs = zsum_s + buf * BN;
      const float g_i = (PHASE == kCore && row_ok && p.gamma) ? p.gamma[row] : 1.f;
      // with rounded activations the accumulator is the exact integer sum_j q_ij zbar_j, and
      // u = Delta gamma (s acc + zero sum_j zbar_j)
      const float dl = (PHASE == kCore && p.delta) ? ldcg_f32(p.delta) : 1.f;
      float amax_t = 0.f;                         // analysis with rounding: this row's max |z|
      // the finished values of columns c .. c + 15 of this thread's row
      auto emit = [&](int c, float* v) {
        if (PHASE == kAnalysis && p.out32) {
          // fp32 z for the rounding kernel, and the running maximum of |z|
#pragma unroll
          for (int q = 0; q < kChunk; ++q) {
            const int t = t0 + c + q;
            if (row_ok && t < p.M) {
              p.out32[static_cast<int64_t>(t) * p.R + row] = v[q];
              amax_t = fmaxf(amax_t, fabsf(v[q]));
            }
          }
          return;
        }
#pragma unroll
        for (int q = 0; q < kChunk; ++q) {
          if (PHASE == kCore) v[q] = g_i * fmaf(s_i, v[q], z_i * zs[c + q]) * dl;
          const __nv_bfloat16 b = __float2bfloat16_rn(v[q]);
          v[q] = __bfloat162float(b);
          const int t = t0 + c + q;
          if (row_ok && t < p.M) p.out[static_cast<int64_t>(t) * p.R + row] = b;
        }
        if (PHASE == kAnalysis) {
          // per-token sum over the tile's 128 rows of the bf16 z actually stored
#pragma unroll
          for (int q = 0; q < kChunk; ++q) {
            float s = row_ok ? v[q] : 0.f;
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
            v[q] = s;
          }
          if (lane == 0) {
#pragma unroll
            for (int q = 0; q < kChunk; ++q) red[ew * kChunk + q] = v[q];
          }
          named_barrier_sync(1, kEpi);
          if (et < kChunk) {
            const int t = t0 + c + et;
            // fixed order over the TMEM quarters (rows 0.., 32.., 64.., 96..)
            const float s = (red[2 * kChunk + et] + red[3 * kChunk + et]) +
                            (red[0 * kChunk + et] + red[1 * kChunk + et]);
            if (t < p.M) p.zsum_part[static_cast<int64_t>(rt) * p.M + t] = s;
          }
          named_barrier_sync(1, kEpi);
        }
      };
      if (p.KS == 1) {
#pragma unroll 1
        for (int c = 0; c < BN; c += kChunk) {
          float v[kChunk];
          tmem_ld16(t_row + c, v);
          tmem_wait_ld();
          emit(c, v);
        }
        tc_fence_before_sync();
        mbar_arrive(&tempty[buf]);
      } else {
        // Split K: store this split's partial tile (column-major, so a warp's 32 rows are one
        // 128-byte line), release the accumulator, and count the split in.  The tile's last
        // split to arrive adds the partials in split order and finishes the tile.
        float* mine = p.part + (static_cast<int64_t>(tile) * p.KS + split) * BN * kBM;
#pragma unroll 1
        for (int c = 0; c < BN; c += kChunk) {
          float v[kChunk];
          tmem_ld16(t_row + c, v);
          tmem_wait_ld();
#pragma unroll
          for (int q = 0; q < kChunk; ++q) mine[(c + q) * kBM + r_in_tile] = v[q];
        }
        tc_fence_before_sync();
        mbar_arrive(&tempty[buf]);
        __threadfence();
        named_barrier_sync(1, kEpi);
        if (et == 0) {
          const uint32_t old = atomicAdd(&p.cnt[tile], 1u);
          const bool last = old == static_cast<uint32_t>(p.KS - 1);
          if (last) p.cnt[tile] = 0;                 // ready for the next call
          __threadfence();
          red[4 * kChunk] = last ? 1.f : 0.f;
        }
        named_barrier_sync(1, kEpi);
        if (red[4 * kChunk] != 0.f) {
          const float* all = p.part + static_cast<int64_t>(tile) * p.KS * BN * kBM;
#pragma unroll 1
          for (int c = 0; c < BN; c += kChunk) {
            float v[kChunk];
#pragma unroll
            for (int q = 0; q < kChunk; ++q) v[q] = 0.f;
            for (int sp = 0; sp < p.KS; ++sp) {
#pragma unroll
              for (int q = 0; q < kChunk; ++q)
                v[q] += ldcg_f32(all + (static_cast<int64_t>(sp) * BN + c + q) * kBM + r_in_tile);
            }
            emit(c, v);
          }
        }
        named_barrier_sync(1, kEpi);                 // the flag is read before it is reused
      }
      if (PHASE == kAnalysis && p.out32) {
        // one atomic per warp and tile: the tensor's max |z| (non-negative floats order like
        // their bit patterns)
#pragma unroll
        for (int off = 16; off > 0; off >>= 1)
          amax_t = fmaxf(amax_t, __shfl_xor_sync(0xffffffffu, amax_t, off));
        if (lane == 0 && amax_t > 0.f) atomicMax(p.amax, __float_as_uint(amax_t));
      }
      if (++buf == 2) buf = 0, acc_phase ^= 1;
    }
  } else {
    // ---------------------------------------------------------------- code decoders (core)
    if (kCodes) {
      // stage i of this CTA is decoded by decoder warp i mod 4, four rows per lane
      const int dw = warp - 6;
      int stage = 0;
      uint32_t phase = 0;
      int it = 0;
      bool ok = true;
      for (int unit = static_cast<int>(cid); unit < p.units && ok && !*abort_flag;
           unit += static_cast<int>(ncl)) {
        for (int kb = unit_k0(unit); kb < unit_k1(unit); ++kb, ++it) {
          if ((it & 3) == dw) {
            if (!mbar_wait(&cfull[stage], phase, abort_flag)) {
              ok = false;
              break;
            }
            const uint4* codes = reinterpret_cast<const uint4*>(sCodes + stage * kCodeBytes);
            uint8_t* tile_a = sA + stage * kATileBytes;
#pragma unroll
            for (int rr = 0; rr < 4; ++rr) decode_row(codes[lane + 32 * rr], tile_a, lane + 32 * rr);
            fence_proxy_async_smem();
            mbar_arrive(&aready[stage]);
          }
          if (++stage == S_) stage = 0, phase ^= 1;
        }
      }
      if (!ok) {
        report(p.status, FQ_ERR_TIMEOUT);
        *abort_flag = 1;
      }
    }
  }

  tc_fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after_sync();
    tmem_dealloc(tmem_base, Lo::kTmemCols);
  }
}

// Rounding of the frame representation of the activations (Appendix F): with the tensor's
// step Delta = max |z| / L, L = 2^(N-1) - 1, zq = nearest integer to z / Delta (ties to even,
// clamped to [-L, L]) as bf16 (exact: |zq| <= 127 needs 7 significant bits), and the per-token
// sum of zq for the zero term (exact in fp32: at most 127 * 81920 < 2^24).  One block per
// token row and round.
constexpr int kQuantThreads = 256;

__global__ void __launch_bounds__(kQuantThreads) ff_round_kernel(
    const float* __restrict__ z32, int M, int n, float L, const uint32_t* __restrict__ amax,
    float* __restrict__ delta, __nv_bfloat16* __restrict__ zq, float* __restrict__ zsum) {
  __shared__ float red[kQuantThreads / 32];
  pdl_launch_dependents();
  pdl_wait();                                   // the analysis is complete
  const float d = __uint_as_float(*reinterpret_cast<const volatile uint32_t*>(amax)) / L;
  if (blockIdx.x == 0 && threadIdx.x == 0) *delta = d;
  for (int t = blockIdx.x; t < M; t += gridDim.x) {
    const float* zr = z32 + static_cast<int64_t>(t) * n;
    __nv_bfloat16* qr = zq + static_cast<int64_t>(t) * n;
    float s = 0.f;
    for (int j = threadIdx.x; j < n; j += kQuantThreads) {
      float q = d > 0.f ? rintf(__fdiv_rn(__ldcg(zr + j), d)) : 0.f;
      q = fminf(fmaxf(q, -L), L);
      qr[j] = __float2bfloat16_rn(q);
      s += q;
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
    __syncthreads();
    if (threadIdx.x == 0) {
      float tot = 0.f;
      for (int w = 0; w < kQuantThreads / 32; ++w) tot += red[w];
      zsum[t] = tot;
    }
    __syncthreads();
  }
}

// The analysis of the d_in unit vectors, for the weight reconstruction: unit vector e_t has
// z = T_in e_t = column t of T_in, exact in bf16, so the analysis product is a transpose,
// z[t][j] = T_in[j][t], through 32 x 32 shared-memory tiles.
__global__ void unit_analysis_kernel(const __nv_bfloat16* __restrict__ T_in, int n_in, int d_in,
                                     __nv_bfloat16* __restrict__ z) {
  __shared__ __nv_bfloat16 tile[32][34];
  const int t0 = blockIdx.x * 32, j0 = blockIdx.y * 32;
  for (int dy = threadIdx.y; dy < 32; dy += 8) {
    const int j = j0 + dy, t = t0 + threadIdx.x;
    if (j < n_in && t < d_in) tile[dy][threadIdx.x] = T_in[static_cast<int64_t>(j) * d_in + t];
  }
  __syncthreads();
  for (int dy = threadIdx.y; dy < 32; dy += 8) {
    const int t = t0 + dy, j = j0 + threadIdx.x;
    if (t < d_in && j < n_in) z[static_cast<int64_t>(t) * n_in + j] = tile[threadIdx.x][dy];
  }
}

// sum_j z[t][j] of unit vector t (the column sums of T_in), for the code product's zero term.
// Block of 32 columns x 32 row groups: thread (x, y) adds rows j = y, y + 32, ... of column
// t0 + x (coalesced across the warp), then the 32 partial sums of a column are added in row
// group order.  Block 0 clears the status word of the new call.
__global__ void __launch_bounds__(1024) unit_zsum_kernel(const __nv_bfloat16* __restrict__ T_in,
                                                         int n_in, int d_in,
                                                         float* __restrict__ zsum,
                                                         int32_t* __restrict__ status) {
  __shared__ float part[32][33];
  if (blockIdx.x == 0 && threadIdx.x == 0 && threadIdx.y == 0) *status = 0;
  const int t = blockIdx.x * 32 + threadIdx.x;
  float s = 0.f;
  if (t < d_in)
    for (int j = threadIdx.y; j < n_in; j += 32)
      s += __bfloat162float(T_in[static_cast<int64_t>(j) * d_in + t]);
  part[threadIdx.y][threadIdx.x] = s;
  __syncthreads();
  if (threadIdx.y == 0 && t < d_in) {
    float tot = 0.f;
    for (int y = 0; y < 32; ++y) tot += part[y][threadIdx.x];
    zsum[t] = tot;
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

int pick_bn(int M) { return M <= 128 ? 128 : 256; }

struct DeviceInfo {
  int dev = -1;
  int sms = 0;
};

DeviceInfo device_info() {
  DeviceInfo d;
  cudaGetDevice(&d.dev);
  cudaDeviceGetAttribute(&d.sms, cudaDevAttrMultiProcessorCount, d.dev);
  if (d.sms <= 0) d.sms = 148;
  return d;
}

template <int PHASE, int BN>
cudaError_t prepare_kernel(int dev) {
  static std::mutex mu;
  static std::map<int, bool> done;
  std::lock_guard<std::mutex> g(mu);
  if (done[dev]) return cudaSuccess;
  cudaError_t e = cudaFuncSetAttribute(tc_phase_kernel<PHASE, BN>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       Layout<PHASE, BN>::kBytes);
  if (e == cudaSuccess) done[dev] = true;
  return e;
}

// One work unit per CTA and round, at most one CTA per SM.  A phase with fewer tiles than SMs
// splits each tile's K range (up to kMaxSplits ways, at least kMinSplitBlocks K blocks each)
// so that it fills the GPU: at 128 tokens a 8192-row phase has only 64 tiles.
constexpr int kMaxSplits = 4;
constexpr int kMinSplitBlocks = 4;
constexpr int kMaxSplitSms = 256;      // bound on the SM count used for split-K planning

int split_for(int tiles, int KB, int sms) {
  sms = std::min(sms, kMaxSplitSms);
  if (tiles >= sms) return 1;
  int ks = std::min({kMaxSplits, sms / tiles, KB / kMinSplitBlocks});
  return std::max(ks, 1);
}

template <int PHASE, int BN>
void plan_phase(PhaseArgs& a, const DeviceInfo& d, int& grid) {
  a.RT = static_cast<int>(ceil_div(a.R, kBM));
  a.TT = static_cast<int>(ceil_div(a.M, BN));
  a.KB = static_cast<int>(ceil_div(a.K, kBK));
  a.tiles = a.RT * a.TT;
  a.KS = split_for(a.tiles, a.KB, d.sms);
  a.kbs = static_cast<int>(ceil_div(a.KB, a.KS));
  a.KS = static_cast<int>(ceil_div(a.KB, a.kbs));     // every split non-empty
  a.units = a.tiles * a.KS;
  grid = std::min(a.units, d.sms);
}

struct WsLayout {
  size_t z, u, zsum, cnt, part, z32, total;
};

// Partial tiles for split K, sized for any device with at most kMaxSplitSms SMs: a phase with
// t < kMaxSplitSms tiles keeps at most min(kMaxSplitSms, t * kMaxSplits) partial tiles.
WsLayout ws_layout(int M, int d_in, int n_in, int n_out, int d_out, int act_bits) {
  WsLayout L{};
  size_t off = kWsHeader;
  L.z = off;
  off += round_up(static_cast<int64_t>(M) * n_in * 2, 256);
  L.u = off;
  off += round_up(static_cast<int64_t>(M) * n_out * 2, 256);
  L.zsum = off;
  off += round_up(ceil_div(n_in, kBM) * M * 4, 256);
  const int BN = pick_bn(M);
  const int64_t TT = ceil_div(M, BN);
  const int64_t rows[3] = {n_in, n_out, d_out};
  int64_t slots = 0, max_tiles = 0;
  for (int64_t r : rows) {
    const int64_t tiles = ceil_div(r, kBM) * TT;
    if (tiles < kMaxSplitSms) {
      slots = std::max(slots, std::min<int64_t>(kMaxSplitSms, tiles * kMaxSplits));
      max_tiles = std::max(max_tiles, tiles);
    }
  }
  (void)d_in;
  L.cnt = off;
  off += round_up(max_tiles * 4, 256);
  L.part = off;
  off += static_cast<size_t>(slots) * BN * kBM * 4;
  L.z32 = off;
  if (act_bits > 0) off += round_up(static_cast<int64_t>(M) * n_in * 4, 256);
  L.total = off;
  return L;
}

template <int PHASE, int BN>
cudaError_t launch_phase(const CUtensorMap& tmA, const CUtensorMap& tmB, const PhaseArgs& a,
                         int grid, cudaStream_t s) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(static_cast<unsigned>(grid));
  cfg.blockDim = dim3(threads_for<PHASE>());
  cfg.dynamicSmemBytes = Layout<PHASE, BN>::kBytes;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, tc_phase_kernel<PHASE, BN>, tmA, tmB, a);
}

// maps: {T_in, x, z, T_out^T, u}.  The core phase's A operand is the packed codes, so it gets
// an unused map in that slot.
cudaError_t launch_round(const PhaseArgs& an, int n_in, int act_bits, const DeviceInfo& d,
                         float* delta, __nv_bfloat16* zq, float* zsum, cudaStream_t s) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(static_cast<unsigned>(std::max(1, std::min(an.M, 4 * d.sms))));
  cfg.blockDim = dim3(kQuantThreads);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const float L = static_cast<float>((1 << (act_bits - 1)) - 1);
  return cudaLaunchKernelEx(&cfg, ff_round_kernel, static_cast<const float*>(an.out32), an.M,
                            n_in, L, static_cast<const uint32_t*>(an.amax), delta, zq, zsum);
}

template <int BN>
fq_status run_forward(const CUtensorMap* maps, PhaseArgs* a, int max_sms, int act_bits,
                      float* delta, cudaStream_t s) {
  DeviceInfo d = device_info();
  if (max_sms > 0) d.sms = std::min(d.sms, max_sms);
  if (prepare_kernel<kAnalysis, BN>(d.dev) != cudaSuccess ||
      prepare_kernel<kCore, BN>(d.dev) != cudaSuccess ||
      prepare_kernel<kSynthesis, BN>(d.dev) != cudaSuccess)
    return FQ_ERR_CUDA;
  int g[3];
  plan_phase<kAnalysis, BN>(a[0], d, g[0]);
  plan_phase<kCore, BN>(a[1], d, g[1]);
  plan_phase<kSynthesis, BN>(a[2], d, g[2]);
  a[1].zsum_tiles = act_bits > 0 ? 1 : a[0].RT;      // rounded: one exact sum per token
  if (launch_phase<kAnalysis, BN>(maps[0], maps[1], a[0], g[0], s) != cudaSuccess)
    return FQ_ERR_CUDA;
  if (act_bits > 0 && launch_round(a[0], a[1].K, act_bits, d, delta, a[0].out, a[0].zsum_part,
                                   s) != cudaSuccess)
    return FQ_ERR_CUDA;
  if (launch_phase<kCore, BN>(maps[1], maps[2], a[1], g[1], s) != cudaSuccess ||
      launch_phase<kSynthesis, BN>(maps[3], maps[4], a[2], g[2], s) != cudaSuccess)
    return FQ_ERR_CUDA;
  return FQ_OK;
}

// The dense product of the weight-reconstruction path: one analysis-phase kernel with the
// reconstructed weight as its A operand (the per-tile sums of the output it also writes go to
// the workspace and are not used).
WsLayout dense_ws_layout(int M, int d_out) {
  WsLayout L{};
  size_t off = kWsHeader;
  L.zsum = off;
  off += round_up(ceil_div(d_out, kBM) * M * 4, 256);
  const int BN = pick_bn(M);
  const int64_t tiles = ceil_div(d_out, kBM) * ceil_div(M, BN);
  int64_t slots = 0, max_tiles = 0;
  if (tiles < kMaxSplitSms) {
    slots = std::min<int64_t>(kMaxSplitSms, tiles * kMaxSplits);
    max_tiles = tiles;
  }
  L.cnt = off;
  off += round_up(max_tiles * 4, 256);
  L.part = off;
  off += static_cast<size_t>(slots) * BN * kBM * 4;
  L.total = off;
  return L;
}

template <int BN>
fq_status run_dense(const CUtensorMap& tmW, const CUtensorMap& tmX, PhaseArgs& a,
                    cudaStream_t s) {
  const DeviceInfo d = device_info();
  if (prepare_kernel<kAnalysis, BN>(d.dev) != cudaSuccess) return FQ_ERR_CUDA;
  int grid = 0;
  plan_phase<kAnalysis, BN>(a, d, grid);
  return launch_phase<kAnalysis, BN>(tmW, tmX, a, grid, s) == cudaSuccess ? FQ_OK : FQ_ERR_CUDA;
}

fq_status launch_tc_dense(const void* x, int M, int d_in, const void* W, int d_out, void* y,
                          char* ws, size_t ws_bytes, cudaStream_t s) {
  const WsLayout L = dense_ws_layout(M, d_out);
  if (ws_bytes < L.total) return FQ_ERR_WORKSPACE;
  const int BN = pick_bn(M);
  PhaseArgs a{};
  a.R = d_out;
  a.K = d_in;
  a.M = M;
  a.out = reinterpret_cast<__nv_bfloat16*>(y);
  a.zsum_part = reinterpret_cast<float*>(ws + L.zsum);
  a.status = reinterpret_cast<int32_t*>(ws);
  a.cnt = reinterpret_cast<uint32_t*>(ws + L.cnt);
  a.part = reinterpret_cast<float*>(ws + L.part);
  CUtensorMap mW, mX;
  if (!make_tmap(&mW, W, d_out, d_in, kBM) || !make_tmap(&mX, x, M, d_in, BN)) return FQ_ERR_CUDA;
  return BN == 128 ? run_dense<128>(mW, mX, a, s) : run_dense<256>(mW, mX, a, s);
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

size_t tc_workspace_bytes(int M, int d_in, int n_in, int n_out, int d_out, int act_bits) {
  return ws_layout(M, d_in, n_in, n_out, d_out, act_bits).total;
}

fq_status launch_tc_forward(const void* x, int M, int d_in, const void* T_in,
                            const fq_packed& Cq, const void* T_out_t, int d_out,
                            const float* gamma, void* y, char* ws, size_t ws_bytes,
                            int max_sms, int act_bits, cudaStream_t s) {
  const int n_in = Cq.n_in, n_out = Cq.n_out;
  const WsLayout L = ws_layout(M, d_in, n_in, n_out, d_out, act_bits);
  if (ws_bytes < L.total) return FQ_ERR_WORKSPACE;
  const int BN = pick_bn(M);
  auto* status = reinterpret_cast<int32_t*>(ws);
  auto* z = reinterpret_cast<__nv_bfloat16*>(ws + L.z);
  auto* u = reinterpret_cast<__nv_bfloat16*>(ws + L.u);
  auto* zsum = reinterpret_cast<float*>(ws + L.zsum);

  PhaseArgs a[3];
  const int R[3] = {n_in, n_out, d_out};
  const int K[3] = {d_in, n_in, n_out};
  __nv_bfloat16* outs[3] = {z, u, reinterpret_cast<__nv_bfloat16*>(y)};
  for (int ph = 0; ph < 3; ++ph) {
    a[ph] = PhaseArgs{};
    a[ph].R = R[ph];
    a[ph].K = K[ph];
    a[ph].M = M;
    a[ph].out = outs[ph];
    a[ph].zsum_part = zsum;
    a[ph].status = status;
    a[ph].cnt = reinterpret_cast<uint32_t*>(ws + L.cnt);
    a[ph].part = reinterpret_cast<float*>(ws + L.part);
  }
  a[1].words = Cq.words;
  a[1].scale = reinterpret_cast<const __half*>(Cq.scale_f16);
  a[1].zero = reinterpret_cast<const __half*>(Cq.zero_f16);
  a[1].gamma = gamma;
  float* delta = nullptr;
  if (act_bits > 0) {
    a[0].out32 = reinterpret_cast<float*>(ws + L.z32);
    a[0].amax = reinterpret_cast<uint32_t*>(ws + kWsAmax);
    delta = reinterpret_cast<float*>(ws + kWsDelta);
    a[1].amax = a[0].amax;
    a[1].delta = delta;
  }

  // maps: T_in, x, z, T_out^T, u  (A maps use 128-row boxes, B maps BN-row boxes)
  CUtensorMap maps[5];
  if (!make_tmap(&maps[0], T_in, n_in, d_in, kBM) || !make_tmap(&maps[1], x, M, d_in, BN) ||
      !make_tmap(&maps[2], z, M, n_in, BN) || !make_tmap(&maps[3], T_out_t, d_out, n_out, kBM) ||
      !make_tmap(&maps[4], u, M, n_out, BN))
    return FQ_ERR_CUDA;

  return BN == 128 ? run_forward<128>(maps, a, max_sms, act_bits, delta, s)
                   : run_forward<256>(maps, a, max_sms, act_bits, delta, s);
}

namespace {
// The code product and the synthesis of the tensor-core chain, after z and one sum of z per
// token have been written to the workspace (a[1].zsum_tiles = 1).
template <int BN>
fq_status run_core_synthesis(const CUtensorMap* maps, PhaseArgs* a, cudaStream_t s) {
  const DeviceInfo d = device_info();
  if (prepare_kernel<kCore, BN>(d.dev) != cudaSuccess ||
      prepare_kernel<kSynthesis, BN>(d.dev) != cudaSuccess)
    return FQ_ERR_CUDA;
  int g[2];
  plan_phase<kCore, BN>(a[1], d, g[0]);
  plan_phase<kSynthesis, BN>(a[2], d, g[1]);
  a[1].zsum_tiles = 1;
  if (launch_phase<kCore, BN>(maps[0], maps[0], a[1], g[0], s) != cudaSuccess ||
      launch_phase<kSynthesis, BN>(maps[1], maps[2], a[2], g[1], s) != cudaSuccess)
    return FQ_ERR_CUDA;
  return FQ_OK;
}
}  // namespace

fq_status launch_tc_unit_forward(const void* T_in, int d_in, const fq_packed& Cq,
                                 const void* T_out_t, int d_out, const float* gamma, void* y,
                                 char* ws, size_t ws_bytes, cudaStream_t s) {
  const int M = d_in, n_in = Cq.n_in, n_out = Cq.n_out;
  const WsLayout L = ws_layout(M, d_in, n_in, n_out, d_out, 0);
  if (ws_bytes < L.total) return FQ_ERR_WORKSPACE;
  const int BN = pick_bn(M);
  auto* status = reinterpret_cast<int32_t*>(ws);
  auto* z = reinterpret_cast<__nv_bfloat16*>(ws + L.z);
  auto* u = reinterpret_cast<__nv_bfloat16*>(ws + L.u);
  auto* zsum = reinterpret_cast<float*>(ws + L.zsum);
  const auto* Tin = static_cast<const __nv_bfloat16*>(T_in);

  PhaseArgs a[3];
  const int R[3] = {n_in, n_out, d_out};
  const int K[3] = {d_in, n_in, n_out};
  __nv_bfloat16* outs[3] = {z, u, reinterpret_cast<__nv_bfloat16*>(y)};
  for (int ph = 1; ph < 3; ++ph) {
    a[ph] = PhaseArgs{};
    a[ph].R = R[ph];
    a[ph].K = K[ph];
    a[ph].M = M;
    a[ph].out = outs[ph];
    a[ph].zsum_part = zsum;
    a[ph].status = status;
    a[ph].cnt = reinterpret_cast<uint32_t*>(ws + L.cnt);
    a[ph].part = reinterpret_cast<float*>(ws + L.part);
  }
  a[1].words = Cq.words;
  a[1].scale = reinterpret_cast<const __half*>(Cq.scale_f16);
  a[1].zero = reinterpret_cast<const __half*>(Cq.zero_f16);
  a[1].gamma = gamma;

  // maps: z (the code product's B; also the unused A slot), T_out^T, u
  CUtensorMap maps[3];
  if (!make_tmap(&maps[0], z, M, n_in, BN) || !make_tmap(&maps[1], T_out_t, d_out, n_out, kBM) ||
      !make_tmap(&maps[2], u, M, n_out, BN))
    return FQ_ERR_CUDA;

  unit_analysis_kernel<<<dim3(static_cast<unsigned>(ceil_div(d_in, 32)),
                              static_cast<unsigned>(ceil_div(n_in, 32))),
                         dim3(32, 8), 0, s>>>(Tin, n_in, d_in, z);
  if (cudaGetLastError() != cudaSuccess) return FQ_ERR_CUDA;
  unit_zsum_kernel<<<static_cast<unsigned>(ceil_div(d_in, 32)), dim3(32, 32), 0, s>>>(
      Tin, n_in, d_in, zsum, status);
  if (cudaGetLastError() != cudaSuccess) return FQ_ERR_CUDA;
  return BN == 128 ? run_core_synthesis<128>(maps, a, s) : run_core_synthesis<256>(maps, a, s);
}

}  // namespace fq

extern "C" {

size_t fq_dense_workspace_bytes(int M, int d_in, int d_out) {
  if (M <= 0 || d_in <= 0 || d_out <= 0) return 0;
  return fq::dense_ws_layout(M, d_out).total;
}

fq_status fq_dense_forward(const void* x, int M, int d_in, const void* W_hat, int d_out, void* y,
                           void* ws, size_t ws_bytes, fq_stream_t stream) {
  if (!x || !W_hat || !y || M <= 0 || d_in <= 0 || d_out <= 0) return FQ_ERR_INVALID_ARG;
  if (d_in % 8 || d_out % 8 || !fq::aligned16(x) || !fq::aligned16(W_hat) || !fq::aligned16(y))
    return FQ_ERR_ALIGNMENT;
  if (!ws) return FQ_ERR_WORKSPACE;
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return FQ_ERR_ALIGNMENT;
  if (ws_bytes < fq_dense_workspace_bytes(M, d_in, d_out)) return FQ_ERR_WORKSPACE;
  int dev = 0, major = 0, minor = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess)
    return FQ_ERR_CUDA;
  if (major * 10 + minor != 103) return FQ_ERR_UNSUPPORTED;
  return fq::launch_tc_dense(x, M, d_in, W_hat, d_out, y, static_cast<char*>(ws), ws_bytes,
                             reinterpret_cast<cudaStream_t>(stream));
}

}  // extern "C"
