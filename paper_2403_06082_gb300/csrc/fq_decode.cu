// FQ_BF16 forward for small batches (M <= 64 tokens): the whole layer in one persistent
// dataflow kernel.
//
// The three products of the layer (Sec. 3.2)
//     analysis   z = T_in x              A = T_in   (n_in x d_in),   B = x
//     core       u = gamma (C_hat z)     A = codes  (n_out x n_in),  B = z
//     synthesis  y = T_out^T u           A = T_out^T (d_out x n_out), B = u
// are cut into tasks = (phase, 128-row tile, K split).  CTA b of G runs tasks b, b + G, ... in
// order; since task indices grow with the phase, every CTA finishes its analysis tasks before
// its core tasks and those before its synthesis tasks, so no CTA ever waits on work that is
// queued behind a wait.  A task reads its activations only after the tiles it needs are
// final: when the last split of a tile has been reduced, its finaliser stamps the tile's
// ready flag with this call's generation (release), and the activation producer of a
// dependent task waits for exactly those flags (acquire, bounded).  No phase waits for the
// whole grid, a split's reduction overlaps other tasks, and the weight producer runs ahead
// into the next tasks (and warms L2 with this CTA's later weight tiles) while activations
// are still being produced.
//
// sum(z), needed by the core's zero term, is produced by the analysis finaliser as one sum
// per 64-column block of z and token, from the bf16 values it stores; a core split adds the
// blocks of its own K range.
//
// The workspace header holds the generation counter, the tiles' ready flags and the split
// tickets; they must start at zero (a zero-filled workspace) and every call leaves them ready
// for the next: tickets wrap back to zero, flags keep generations that are all in the past,
// and the last CTA to finish advances the generation.
//
// Warps: 0 weight (A) producer, 1 TMEM owner + MMA issuer, 2-5 epilogue (thread = tile row),
// 6 activation (B) producer, 7-10 code decoders (core stages, stage i -> warp i mod 4).
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <map>
#include <mutex>

#include "fq_device.cuh"
#include "fq_internal.h"

namespace fq {
namespace {

constexpr int kBM = 128;
constexpr int kBK = 64;
constexpr int kATile = kBM * kBK * 2;      // 16 KiB
constexpr int kCodeBytes = kBM * kBK / 4;  // 2 KiB
constexpr int kMaxSplit = 8;
constexpr int kEpi = 128;
constexpr int kChunk = 16;
constexpr int kThreads = 352;
constexpr int64_t kL2PrefetchBudget = 64ll << 20;

struct DecPhase {
  int R, K, RT, S, KB, kbs, tasks, base;
  __nv_bfloat16* out;     // [M][R]
  float* partial;         // [S][M][R] when S > 1
  uint32_t* flags;        // [RT] tile final in this call when == generation + 1
  uint32_t* tickets;      // [RT] split arrivals (wrap to zero)
};

struct DecArgs {
  int M, total;
  DecPhase ph[3];
  const uint32_t* words;
  const __half* scale;
  const __half* zero;
  const float* gamma;
  float* zsum64;          // [nblk][M] sums of z over 64-column blocks
  int nblk;
  int32_t* status;
  uint32_t* gen;
  uint32_t* done;
  int prefetch_later;     // 0: none, 1: codes, 2: codes and T_out^T tiles
};

template <int BN>
struct DecLayout {
  static constexpr int kBTile = BN * kBK * 2;
  static constexpr int kStage = kATile + kBTile + kCodeBytes;
  static constexpr int kStages = std::min(12, (200 * 1024 - 4096) / kStage);
  static constexpr uint32_t kTmemCols = 2 * BN < 32 ? 32 : 2 * BN;
  static constexpr int oA = 0;
  static constexpr int oB = oA + kStages * kATile;
  static constexpr int oC = oB + kStages * kBTile;
  static constexpr int oBar = oC + kStages * kCodeBytes;
  static constexpr int kBars = 4 * kStages + 5;
  static constexpr int oMisc = oBar + kBars * 8;
  static constexpr int oRed = oMisc + 16;            // [4][BN] floats
  static constexpr int oZs = oRed + 4 * BN * 4;      // [BN] floats
  static constexpr int kBytes = oZs + BN * 4 + 1024;
  static_assert(kBTile % 1024 == 0, "B tiles keep 1024-byte alignment");
};

struct Task {
  int p, tile, ks;
};

__device__ __forceinline__ DecPhase phase_of(const DecArgs& a, int p) {
  return p == 0 ? a.ph[0] : (p == 1 ? a.ph[1] : a.ph[2]);
}

__device__ __forceinline__ Task task_of(const DecArgs& a, int i) {
  const int p = (i >= a.ph[1].base) + (i >= a.ph[2].base);
  const DecPhase ph = phase_of(a, p);
  const int j = i - ph.base;
  return {p, j / ph.S, j % ph.S};
}

// Same code decoding as the three-kernel path: q -> bf16(128 + q) - 128, swizzled row store.
__device__ __forceinline__ void decode_row_dec(const uint4 w4, uint8_t* tile, int r) {
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
#pragma unroll
    for (int half = 0; half < 2; ++half) {
      const int c = 2 * wi + half;
      *reinterpret_cast<uint4*>(row + ((c ^ (r & 7)) << 4)) =
          make_uint4(h[4 * half], h[4 * half + 1], h[4 * half + 2], h[4 * half + 3]);
    }
  }
}

__device__ __forceinline__ bool bar_red_or_dec(uint32_t id, uint32_t n, bool v) {
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

// First timeout of a call: role, task, stage and a detail word go to status[4..7] (the rest
// of the header's first 64 bytes), for diagnosis with the status word.
__device__ __forceinline__ void note_timeout(int32_t* status, int role, int task, int stage,
                                             int detail) {
  report(status, FQ_ERR_TIMEOUT);
  if (atomicCAS(reinterpret_cast<int*>(status) + 4, 0, role) == 0) {
    status[5] = task;
    status[6] = stage;
    status[7] = detail;
  }
}

template <int BN>
__global__ void __launch_bounds__(kThreads, 1)
    decode_layer_kernel(const __grid_constant__ CUtensorMap tmTin,
                        const __grid_constant__ CUtensorMap tmX,
                        const __grid_constant__ CUtensorMap tmZ,
                        const __grid_constant__ CUtensorMap tmTout,
                        const __grid_constant__ CUtensorMap tmU, const DecArgs a) {
  using Lo = DecLayout<BN>;
  constexpr int S_ = Lo::kStages;
  constexpr int kBTile = Lo::kBTile;

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem + Lo::oA;
  uint8_t* sB = smem + Lo::oB;
  uint8_t* sC = smem + Lo::oC;
  // fullA completes every round of a stage (a weight tile or, for core tasks, its codes);
  // aready only in core rounds, so its parity is tracked per stage
  uint64_t* fullA = reinterpret_cast<uint64_t*>(smem + Lo::oBar);
  uint64_t* fullB = fullA + S_;
  uint64_t* empty = fullB + S_;
  uint64_t* aready = empty + S_;
  uint64_t* tfull = aready + S_;
  uint64_t* tempty = tfull + 2;
  uint64_t* mma_done = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + Lo::oMisc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  uint32_t* gen_s = tmem_slot + 2;
  int* ticket_s = reinterpret_cast<int*>(tmem_slot + 3);
  float* red = reinterpret_cast<float*>(smem + Lo::oRed);
  float* zs_s = reinterpret_cast<float*>(smem + Lo::oZs);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = gridDim.x;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S_; ++s) {
      mbar_init(&fullA[s], 1);
      mbar_init(&fullB[s], 1);
      mbar_init(&empty[s], 1);
      mbar_init(&aready[s], 32);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], kEpi);
    }
    mbar_init(mma_done, 1);
    *abort_flag = 0;
    fence_barrier_init();
    prefetch_tmap(&tmTin);
    prefetch_tmap(&tmX);
    prefetch_tmap(&tmZ);
    prefetch_tmap(&tmTout);
    prefetch_tmap(&tmU);
  }
  if (warp == 1) tmem_alloc(tmem_slot, Lo::kTmemCols);
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem_base = *tmem_slot;
  pdl_launch_dependents();

  if (warp == 0) {
    // -------------------------------------------------------------- weight (A) producer
    if (lane == 0) {
      const uint64_t pol_w = policy_evict_first();
      int stage = 0;
      uint32_t phase = 0;
      bool first = true;
      uint32_t last_par[S_];
      bool used[S_];
#pragma unroll
      for (int s = 0; s < S_; ++s) last_par[s] = 0, used[s] = false;
      for (int i = blockIdx.x; i < a.total && !*abort_flag; i += G) {
        const Task t = task_of(a, i);
        const DecPhase ph = phase_of(a, t.p);
        const int k0 = t.ks * ph.kbs, k1 = min(ph.KB, k0 + ph.kbs);
        for (int kb = k0; kb < k1; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1, abort_flag)) {
            if (!*abort_flag) note_timeout(a.status, 1, i, stage, static_cast<int>(phase));
            *abort_flag = 1;
            break;
          }
          if (t.p == 1) {
            mbar_arrive_expect_tx(&fullA[stage], kCodeBytes);
            bulk_load(sC + stage * kCodeBytes,
                      a.words + (static_cast<int64_t>(t.tile) * ph.KB + kb) * 512, kCodeBytes,
                      &fullA[stage], pol_w);
          } else {
            mbar_arrive_expect_tx(&fullA[stage], kATile);
            tma_load_2d(sA + stage * kATile, t.p == 0 ? &tmTin : &tmTout, &fullA[stage],
                        kb * kBK, t.tile * kBM, pol_w);
          }
          used[stage] = true;
          last_par[stage] = phase;
          if (++stage == S_) stage = 0, phase ^= 1;
        }
        if (first) {
          first = false;
          // warm L2 with the weight tiles of this CTA's later tasks
          for (int j = i + G; j < a.total && a.prefetch_later > 0; j += G) {
            const Task u = task_of(a, j);
            const DecPhase q = phase_of(a, u.p);
            const int u0 = u.ks * q.kbs, u1 = min(q.KB, u0 + q.kbs);
            if (u.p == 1) {
              const uint32_t* src = a.words + (static_cast<int64_t>(u.tile) * q.KB + u0) * 512;
              asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src),
                           "r"(static_cast<uint32_t>((u1 - u0) * kCodeBytes))
                           : "memory");
            } else if (u.p == 2 && a.prefetch_later > 1) {
              for (int kb = u0; kb < u1; ++kb)
                asm volatile(
                    "cp.async.bulk.prefetch.tensor.2d.L2.global.tile [%0, {%1, %2}];" ::"l"(
                        reinterpret_cast<uint64_t>(&tmTout)),
                    "r"(kb * kBK), "r"(u.tile * kBM)
                    : "memory");
            }
          }
        }
      }
      for (int s = 0; s < S_; ++s)
        if (used[s] && !mbar_wait(&fullA[s], last_par[s], nullptr))
          report(a.status, FQ_ERR_TIMEOUT);
    }
  } else if (warp == 6) {
    // -------------------------------------------------------------- activation (B) producer
    if (lane == 0) {
      const uint64_t pol_x = policy_evict_last();
      pdl_wait();
      if (blockIdx.x == 0) *a.status = 0;      // a new call
      const uint32_t g = ld_acquire_gpu(a.gen) + 1;
      int stage = 0;
      uint32_t phase = 0;
      uint32_t last_par[S_];
      bool used[S_];
#pragma unroll
      for (int s = 0; s < S_; ++s) last_par[s] = 0, used[s] = false;
      for (int i = blockIdx.x; i < a.total && !*abort_flag; i += G) {
        const Task t = task_of(a, i);
        const DecPhase ph = phase_of(a, t.p);
        const int k0 = t.ks * ph.kbs, k1 = min(ph.KB, k0 + ph.kbs);
        if (t.p > 0) {
          // every source tile covering this task's K range must be final
          const DecPhase src = phase_of(a, t.p - 1);
          const int lo = (k0 * kBK) / kBM, hi = (min(ph.K, k1 * kBK) - 1) / kBM;
          bool ok = true;
          int bad = -1;
          for (int s = lo; s <= hi && ok; ++s) {
            ok = wait_flag(&src.flags[s], g, abort_flag);
            if (!ok) bad = s;
          }
          if (!ok) {
            if (!*abort_flag)
              note_timeout(a.status, 2, i, bad,
                           static_cast<int>(ld_acquire_gpu(&src.flags[bad]) - g) * 1000 + t.p);
            *abort_flag = 1;
            break;
          }
        }
        const CUtensorMap* tm = t.p == 0 ? &tmX : (t.p == 1 ? &tmZ : &tmU);
        bool ok = true;
        for (int kb = k0; kb < k1; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1, abort_flag)) {
            if (!*abort_flag) note_timeout(a.status, 3, i, stage, static_cast<int>(phase));
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&fullB[stage], kBTile);
          tma_load_2d(sB + stage * kBTile, tm, &fullB[stage], kb * kBK, 0, pol_x);
          used[stage] = true;
          last_par[stage] = phase;
          if (++stage == S_) stage = 0, phase ^= 1;
        }
        if (!ok) {
          report(a.status, FQ_ERR_TIMEOUT);
          *abort_flag = 1;
          break;
        }
      }
      for (int s = 0; s < S_; ++s)
        if (used[s] && !mbar_wait(&fullB[s], last_par[s], nullptr))
          report(a.status, FQ_ERR_TIMEOUT);
    }
  } else if (warp == 1) {
    // -------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = umma_idesc_bf16(kBM, BN);
      int stage = 0;
      uint32_t phase = 0;
      int buf = 0;
      uint32_t acc_phase = 0;
      uint32_t apar = 0;     // bit s: parity of the next aready[s] phase
      bool issued_any = false;
      for (int i = blockIdx.x; i < a.total && !*abort_flag; i += G) {
        const Task t = task_of(a, i);
        const DecPhase ph = phase_of(a, t.p);
        const int k0 = t.ks * ph.kbs, k1 = min(ph.KB, k0 + ph.kbs);
        if (!mbar_wait(&tempty[buf], acc_phase ^ 1, abort_flag)) {
          if (!*abort_flag) note_timeout(a.status, 4, i, buf, static_cast<int>(acc_phase));
          *abort_flag = 1;
          break;
        }
        tc_fence_after_sync();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(buf * BN);
        bool ok = true;
        for (int kb = k0; kb < k1; ++kb) {
          if (t.p == 1) {
            ok = mbar_wait(&aready[stage], (apar >> stage) & 1u, abort_flag);
            apar ^= 1u << stage;
          } else {
            ok = mbar_wait(&fullA[stage], phase, abort_flag);
          }
          if (!ok && !*abort_flag) note_timeout(a.status, 5, i, stage, kb * 2 + static_cast<int>(phase));
          if (ok) {
            ok = mbar_wait(&fullB[stage], phase, abort_flag);
            if (!ok && !*abort_flag) note_timeout(a.status, 6, i, stage, kb * 2 + static_cast<int>(phase));
          }
          if (!ok) break;
          tc_fence_after_sync();
          const uint64_t adesc = umma_desc_sw128(smem_u32(sA + stage * kATile));
          const uint64_t bdesc = umma_desc_sw128(smem_u32(sB + stage * kBTile));
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k)
            umma_bf16(d_tmem, adesc + 2 * k, bdesc + 2 * k, idesc, (kb > k0 || k > 0) ? 1u : 0u);
          issued_any = true;
          umma_commit(&empty[stage]);
          if (++stage == S_) stage = 0, phase ^= 1;
        }
        if (!ok) {
          report(a.status, FQ_ERR_TIMEOUT);
          *abort_flag = 1;
          break;
        }
        umma_commit(&tfull[buf]);
        if (++buf == 2) buf = 0, acc_phase ^= 1;
      }
      if (issued_any) {
        umma_commit(mma_done);
        if (!mbar_wait(mma_done, 0, nullptr)) report(a.status, FQ_ERR_TIMEOUT);
      }
    }
  } else if (warp >= 7) {
    // -------------------------------------------------------------- code decoders
    const int dw = warp - 7;
    int stage = 0;
    uint32_t phase = 0;
    int it = 0;
    bool ok = true;
    for (int i = blockIdx.x; i < a.total && ok && !*abort_flag; i += G) {
      const Task t = task_of(a, i);
      const DecPhase ph = phase_of(a, t.p);
      const int k0 = t.ks * ph.kbs, k1 = min(ph.KB, k0 + ph.kbs);
      for (int kb = k0; kb < k1; ++kb, ++it) {
        // every decoder warp follows every round of the ring (a parity wait is only exact
        // when the waiter is at most one phase ahead), and decodes the code rounds it owns
        if (!mbar_wait(&fullA[stage], phase, abort_flag)) {
          if (!*abort_flag && lane == 0) note_timeout(a.status, 7, i, stage, static_cast<int>(phase));
          ok = false;
          break;
        }
        if (t.p == 1 && (it & 3) == dw) {
          const uint4* codes = reinterpret_cast<const uint4*>(sC + stage * kCodeBytes);
          uint8_t* tile_a = sA + stage * kATile;
#pragma unroll
          for (int rr = 0; rr < 4; ++rr)
            decode_row_dec(codes[lane + 32 * rr], tile_a, lane + 32 * rr);
          fence_proxy_async_smem();
          mbar_arrive(&aready[stage]);
        }
        if (++stage == S_) stage = 0, phase ^= 1;
      }
    }
    if (!ok) {
      report(a.status, FQ_ERR_TIMEOUT);
      *abort_flag = 1;
    }
  } else {
    // -------------------------------------------------------------- epilogue (warps 2-5)
    const int quarter = warp & 3;                 // TMEM lanes 32 * quarter .. + 31
    const int r_in_tile = quarter * 32 + lane;
    const int et = threadIdx.x - 64;
    pdl_wait();
    if (et == 0) *gen_s = ld_acquire_gpu(a.gen) + 1;
    named_barrier_sync(1, kEpi);
    const uint32_t g = *gen_s;
    int buf = 0;
    uint32_t acc_phase = 0;
    for (int i = blockIdx.x; i < a.total; i += G) {
      const Task t = task_of(a, i);
      const DecPhase ph = phase_of(a, t.p);
      const int k0 = t.ks * ph.kbs, k1 = min(ph.KB, k0 + ph.kbs);
      const int row = t.tile * kBM + r_in_tile;
      const bool row_ok = row < ph.R;
      float s_i = 0.f, z_i = 0.f, g_i = 1.f;
      bool fail = false;
      if (t.p == 1) {
        if (row_ok) {
          s_i = __half2float(a.scale[row]);
          z_i = __half2float(a.zero[row]);
          if (a.gamma) g_i = a.gamma[row];
        }
        // sum of z over this split's K range, from the 64-column block sums of the analysis
        if (et == 0) {
          const int lo = (k0 * kBK) / kBM, hi = (min(ph.K, k1 * kBK) - 1) / kBM;
          for (int s = lo; s <= hi && !fail; ++s) {
            fail = !wait_flag(&a.ph[0].flags[s], g, abort_flag);
            if (fail && !*abort_flag) note_timeout(a.status, 8, i, s, 0);
          }
        }
        named_barrier_sync(1, kEpi);
        for (int q = et; q < BN; q += kEpi) {
          float s = 0.f;
          if (q < a.M)
            for (int b = k0; b < k1 && b < a.nblk; ++b) s += ldcg_f32(a.zsum64 + b * a.M + q);
          zs_s[q] = s;
        }
      }
      if (!fail && !mbar_wait(&tfull[buf], acc_phase, abort_flag)) {
        fail = true;
        if (!*abort_flag && et == 0) note_timeout(a.status, 9, i, buf, static_cast<int>(acc_phase));
      }
      if (fail) report(a.status, FQ_ERR_TIMEOUT);
      if (bar_red_or_dec(1, kEpi, fail || *abort_flag)) {
        if (et == 0) *abort_flag = 1;
        break;
      }
      tc_fence_after_sync();
      const uint32_t t_row = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) +
                             static_cast<uint32_t>(buf * BN);

      // final values of this row for tokens c .. c + 15: store, and for the analysis the
      // per-token sums over the tile's two 64-row blocks
      auto finish = [&](int c, float (&v)[kChunk]) {
#pragma unroll
        for (int j = 0; j < kChunk; ++j) {
          float val = v[j];
          if (t.p == 1) val *= g_i;
          const __nv_bfloat16 b = __float2bfloat16_rn(val);
          if (row_ok && c + j < a.M) ph.out[static_cast<int64_t>(c + j) * ph.R + row] = b;
          v[j] = row_ok ? __bfloat162float(b) : 0.f;
        }
        if (t.p == 0) {
#pragma unroll
          for (int j = 0; j < kChunk; ++j) {
            float s = v[j];
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
            if (lane == 0) red[quarter * BN + c + j] = s;
          }
          named_barrier_sync(1, kEpi);
          if (et < 2 * kChunk) {
            const int blk = et / kChunk, tok = c + et % kChunk;
            const float s = red[(2 * blk) * BN + tok] + red[(2 * blk + 1) * BN + tok];
            const int gb = t.tile * 2 + blk;
            if (gb < a.nblk && tok < a.M) a.zsum64[gb * a.M + tok] = s;
          }
          named_barrier_sync(1, kEpi);
        }
      };

      if (ph.S == 1) {
        float vals[BN];
#pragma unroll
        for (int c = 0; c < BN; c += kChunk) {
          float v[kChunk];
          tmem_ld16(t_row + c, v);
          tmem_wait_ld();
#pragma unroll
          for (int j = 0; j < kChunk; ++j)
            vals[c + j] = t.p == 1 ? fmaf(s_i, v[j], z_i * zs_s[c + j]) : v[j];
        }
        tc_fence_before_sync();
        mbar_arrive(&tempty[buf]);
#pragma unroll
        for (int c = 0; c < BN; c += kChunk) {
          float v[kChunk];
#pragma unroll
          for (int j = 0; j < kChunk; ++j) v[j] = vals[c + j];
          finish(c, v);
        }
      } else {
        float* part = ph.partial + static_cast<int64_t>(t.ks) * a.M * ph.R;
#pragma unroll
        for (int c = 0; c < BN; c += kChunk) {
          float v[kChunk];
          tmem_ld16(t_row + c, v);
          tmem_wait_ld();
#pragma unroll
          for (int j = 0; j < kChunk; ++j) {
            const float val = t.p == 1 ? fmaf(s_i, v[j], z_i * zs_s[c + j]) : v[j];
            if (row_ok && c + j < a.M) part[static_cast<int64_t>(c + j) * ph.R + row] = val;
          }
        }
        tc_fence_before_sync();
        mbar_arrive(&tempty[buf]);
        __threadfence();
        named_barrier_sync(1, kEpi);
        if (et == 0) {
          const unsigned old =
              atomicInc(&ph.tickets[t.tile], static_cast<unsigned>(ph.S - 1));
          *ticket_s = old == static_cast<unsigned>(ph.S - 1) ? 1 : 0;
        }
        named_barrier_sync(1, kEpi);
        if (*ticket_s == 0) {
          if (++buf == 2) buf = 0, acc_phase ^= 1;
          continue;                     // another CTA finishes this tile
        }
        __threadfence();
#pragma unroll
        for (int c = 0; c < BN; c += kChunk) {
          float v[kChunk];
#pragma unroll
          for (int j = 0; j < kChunk; ++j) v[j] = 0.f;
#pragma unroll 2
          for (int q = 0; q < ph.S; ++q) {
            const float* src = ph.partial + (static_cast<int64_t>(q) * a.M + c) * ph.R + row;
            float w[kChunk];
#pragma unroll
            for (int j = 0; j < kChunk; ++j)
              w[j] = (row_ok && c + j < a.M) ? ldcg_f32(src + static_cast<int64_t>(j) * ph.R)
                                              : 0.f;
#pragma unroll
            for (int j = 0; j < kChunk; ++j) v[j] += w[j];
          }
          finish(c, v);
        }
      }
      // the tile is final: publish it to dependent tasks
      if (t.p < 2) {
        __threadfence();
        named_barrier_sync(1, kEpi);
        if (et == 0) st_release_gpu(&ph.flags[t.tile], g);
      }
      if (++buf == 2) buf = 0, acc_phase ^= 1;
    }
  }

  tc_fence_before_sync();
  __syncthreads();
  if (threadIdx.x == 0) {
    // the last CTA to finish moves the workspace to the next call's generation
    __threadfence();
    const unsigned old = atomicInc(a.done, static_cast<unsigned>(G - 1));
    if (old == static_cast<unsigned>(G - 1)) {
      __threadfence();
      atomicAdd(a.gen, 1u);
    }
  }
  if (warp == 1) {
    tc_fence_after_sync();
    tmem_dealloc(tmem_base, Lo::kTmemCols);
  }
}

// ---------------------------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------------------------
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
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

bool tmap_bf16(CUtensorMap* m, const void* base, int64_t rows, int64_t cols, int box_rows) {
  auto enc = encode_fn();
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

int decode_bn(int M) { return M <= 16 ? 16 : (M <= 32 ? 32 : 64); }

struct DecWs {
  size_t z, u, zsum, part[3], total;
};

DecWs dec_ws(int M, int d_in, int n_in, int n_out, int d_out) {
  (void)d_in;
  DecWs L{};
  size_t off = kWsHeader;
  L.z = off;
  off += round_up(static_cast<int64_t>(M) * n_in * 2, 256);
  L.u = off;
  off += round_up(static_cast<int64_t>(M) * n_out * 2, 256);
  L.zsum = off;
  off += round_up(ceil_div(n_in, kBK) * M * 4, 256);
  const int R[3] = {n_in, n_out, d_out};
  for (int p = 0; p < 3; ++p) {
    L.part[p] = off;
    off += round_up(static_cast<int64_t>(kMaxSplit) * M * R[p] * 4, 256);
  }
  L.total = off;
  return L;
}

template <int BN>
cudaError_t prepare(int dev) {
  static std::mutex mu;
  static std::map<int, bool> done;
  std::lock_guard<std::mutex> g(mu);
  if (done[dev]) return cudaSuccess;
  const cudaError_t e = cudaFuncSetAttribute(decode_layer_kernel<BN>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             DecLayout<BN>::kBytes);
  if (e == cudaSuccess) done[dev] = true;
  return e;
}

// K splits of one phase: the busiest CTA's K blocks plus a fixed cost per task (pipeline
// fill, epilogue) and a small cost for a split's reduction, minimised over S.
void plan(DecPhase& ph, int G) {
  ph.RT = static_cast<int>(ceil_div(ph.R, kBM));
  ph.KB = static_cast<int>(ceil_div(ph.K, kBK));
  int best_s = 1;
  double best = 1e30;
  for (int s = 1; s <= std::min(kMaxSplit, ph.KB); ++s) {
    const int kbs = static_cast<int>(ceil_div(ph.KB, s));
    if (ceil_div(ph.KB, kbs) != s) continue;
    const double per_cta = static_cast<double>(ceil_div(static_cast<int64_t>(ph.RT) * s, G));
    const double cost = per_cta * (kbs + 3.0) + (s > 1 ? 2.0 : 0.0);
    if (cost < best - 1e-9) best = cost, best_s = s;
  }
  ph.S = best_s;
  ph.kbs = static_cast<int>(ceil_div(ph.KB, best_s));
  ph.tasks = ph.RT * ph.S;
}

template <int BN>
fq_status run(const CUtensorMap* m, DecArgs& a, int G, cudaStream_t s) {
  int dev = 0;
  cudaGetDevice(&dev);
  if (prepare<BN>(dev) != cudaSuccess) return FQ_ERR_CUDA;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(static_cast<unsigned>(G));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = DecLayout<BN>::kBytes;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, decode_layer_kernel<BN>, m[0], m[1], m[2], m[3], m[4], a) ==
                 cudaSuccess
             ? FQ_OK
             : FQ_ERR_CUDA;
}

}  // namespace

size_t decode_workspace_bytes(int M, int d_in, int n_in, int n_out, int d_out) {
  return dec_ws(M, d_in, n_in, n_out, d_out).total;
}

fq_status launch_decode_forward(const void* x, int M, int d_in, const void* T_in,
                                const fq_packed& Cq, const void* T_out_t, int d_out,
                                const float* gamma, void* y, char* ws, size_t ws_bytes,
                                cudaStream_t s) {
  const int n_in = Cq.n_in, n_out = Cq.n_out;
  const DecWs L = dec_ws(M, d_in, n_in, n_out, d_out);
  if (ws_bytes < L.total) return FQ_ERR_WORKSPACE;
  const int BN = decode_bn(M);
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (sms <= 0) return FQ_ERR_CUDA;

  DecArgs a{};
  a.M = M;
  const int R[3] = {n_in, n_out, d_out};
  const int K[3] = {d_in, n_in, n_out};
  void* outs[3] = {ws + L.z, ws + L.u, y};
  int base = 0;
  for (int p = 0; p < 3; ++p) {
    DecPhase& ph = a.ph[p];
    ph.R = R[p];
    ph.K = K[p];
    plan(ph, sms);
    if (ph.RT > kWsMaxTiles) return FQ_ERR_UNSUPPORTED;
    ph.base = base;
    base += ph.tasks;
    ph.out = static_cast<__nv_bfloat16*>(outs[p]);
    ph.partial = reinterpret_cast<float*>(ws + L.part[p]);
    ph.flags = reinterpret_cast<uint32_t*>(ws + kWsFlags) + p * kWsMaxTiles;
    ph.tickets = reinterpret_cast<uint32_t*>(ws + kWsTickets) + p * kWsMaxTiles;
  }
  a.total = base;
  a.words = Cq.words;
  a.scale = reinterpret_cast<const __half*>(Cq.scale);
  a.zero = reinterpret_cast<const __half*>(Cq.zero);
  a.gamma = gamma;
  a.zsum64 = reinterpret_cast<float*>(ws + L.zsum);
  a.nblk = static_cast<int>(ceil_div(n_in, kBK));
  a.status = reinterpret_cast<int32_t*>(ws);
  a.gen = reinterpret_cast<uint32_t*>(ws + kWsGen);
  a.done = reinterpret_cast<uint32_t*>(ws + kWsDone);
  const int64_t code_bytes = static_cast<int64_t>(fq_packed_words(n_out, n_in)) * 4;
  const int64_t tout_bytes = static_cast<int64_t>(d_out) * n_out * 2;
  a.prefetch_later = code_bytes + tout_bytes <= kL2PrefetchBudget ? 2
                     : (code_bytes <= kL2PrefetchBudget ? 1 : 0);

  CUtensorMap m[5];
  if (!tmap_bf16(&m[0], T_in, n_in, d_in, kBM) || !tmap_bf16(&m[1], x, M, d_in, BN) ||
      !tmap_bf16(&m[2], ws + L.z, M, n_in, BN) ||
      !tmap_bf16(&m[3], T_out_t, d_out, n_out, kBM) || !tmap_bf16(&m[4], ws + L.u, M, n_out, BN))
    return FQ_ERR_CUDA;
  const int G = std::min(sms, a.total);
  switch (BN) {
    case 16: return run<16>(m, a, G, s);
    case 32: return run<32>(m, a, G, s);
    default: return run<64>(m, a, G, s);
  }
}

}  // namespace fq
