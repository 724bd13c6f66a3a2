// FQ_BF16 forward for small batches (M <= 64 tokens): the whole layer in one persistent
// dataflow kernel.
//
// The three products of the layer (Sec. 3.2)
//     analysis   z = T_in x              A = T_in   (n_in x d_in),   B = x
//     core       u = gamma (C_hat z)     A = codes  (n_out x n_in),  B = z
//     synthesis  y = T_out^T u           A = T_out^T (d_out x n_out), B = u
// are cut into tasks = (phase, 128-row tile).  The kernel runs as clusters of S CTAs; CTA r of
// a cluster takes K split r of every task of its cluster and reduces slice r (128/S rows) of
// the task's output tile.  The split-K exchange is one-way: every epilogue thread pushes its
// row of fp32 partial sums from registers into the receive buffer of the CTA that owns the
// row (st.async into distributed shared memory, counted by that CTA's own mbarrier), and each
// CTA adds the S partials of its slice in rank order (deterministic; no global partials, no
// atomics, no remote arrivals).  Receive buffers alternate between consecutive tasks; a buffer
// is only written again after its owner has sent the next task's partials, which it does only
// after reading the buffer, so no back-pressure signal is needed.  Each cluster runs its own
// list of tasks, in phase order (so no cluster waits on work queued behind a wait); the
// lists are built on the host (tiles dealt round-robin, each phase's tiles ordered by where
// they fall in the next phase's K splits, so that every consumer's first K blocks are
// produced first).  Each CTA stamps the ready flag of its slice with this
// call's generation (release) once the slice is stored, and the activation producer of a
// dependent task waits for exactly the slices its K range reads (acquire, bounded, one lane
// per flag).  No phase waits for the whole grid, and the weight producer runs ahead into the
// next tasks (and warms L2 with this CTA's later code blocks, and with its synthesis tiles when
// the layer is small enough) while activations are still being produced.
//
// sum(z), needed by the core's zero term, is taken by the core's epilogue over the bf16 z of its
// own K range, read from global memory once the slices' ready flags are seen (this runs while
// the task's MMAs are in flight, and keeps the analysis epilogue, which every core task waits
// for, short).
//
// The workspace header holds the generation counter and the tiles' ready flags; a zero-filled
// header is a valid start and every call leaves it valid for the next (flags keep
// generations that are all in the past; the last CTA to finish advances the generation).
//
// Warps: 0 weight (A) producer, 1 TMEM owner + MMA issuer 0, 2-5 epilogue (thread = tile row),
// 6 activation (B) producer, 7-10 code decoders (ring stage s -> decoder s mod 4; one per SM
// sub-partition, since the decode is issue-bound), and for 16 or 32 tokens 12, 14, 15 MMA
// issuers 1-3 (one issuer per SM sub-partition).
//
// Ring protocol.  A parity wait on an mbarrier is only exact when its waiter is neither ahead
// of the barrier nor two or more phases behind it, so each barrier's waiters take part in
// every one of its phases that follows a phase they wait for:
//   empty[s]  (the round's MMAs completed)  the weight and the activation producers, which
//             both fill every round of the stage;
//   cfull[s]  (a core round's code block landed)  decoder s mod 4, whose arrival on fullA[s]
//             the round's MMAs (and so the next code load into the stage) wait for;
//   fullA[s]  (the A tile is in place: the weight tile's bytes, or the decoder's arrival in
//             core rounds), fullB[s]  the issuer that owns s, which commits empty[s].
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <array>
#include <map>
#include <mutex>
#include <utility>
#include <vector>

#include "fq_device.cuh"
#include "fq_internal.h"

namespace fq {
namespace {

constexpr int kBM = 128;
constexpr int kBK = 64;
constexpr int kATile = kBM * kBK * 2;      // 16 KiB
constexpr int kCodeBytes = kBM * kBK / 4;  // 2 KiB
constexpr int kMaxSplit = 8;
static_assert(kMaxSplit <= kWsSlices, "one ready flag per slice");
constexpr int kEpi = 128;
constexpr int kChunk = 16;
// MMA issuers per CTA.  A tcgen05.mma with N = 16 or 32 tokens is short, and one thread cannot
// issue K blocks (waits, MMAs, commit) as fast as the tensor core retires them; NI issuers, one
// per SM sub-partition, each own the ring stages s = q (mod NI) and accumulate their K blocks
// into their own accumulator, which the epilogue adds.  Owning stages (not K blocks) keeps
// every barrier of a stage waited for by one thread, in phase order.  With 64 tokens the
// epilogue's registers do not leave room for the extra warps: one issuer.
// With four issuers the code decode also gets a second warp per stage (warps 16-19), each of
// a stage's two decoders expanding half of its rows; with 64 tokens neither fits.
template <int BN>
struct DecCfg {
  static constexpr int NI = BN <= 32 ? 4 : 1;
  static constexpr bool kPairs = NI == 4;
  static constexpr int kThreads = NI == 4 ? 640 : 384;
};
// warp -> issuer index (warps 1, 12, 14, 15: sub-partitions 1, 0, 2, 3), -1 for other roles
__host__ __device__ constexpr int issuer_of(int warp, int ni) {
  return warp == 1 ? 0
                   : (ni == 4 ? (warp == 12 ? 1 : (warp == 14 ? 2 : (warp == 15 ? 3 : -1))) : -1);
}
// L2 warming.  When a layer's code blocks fit kL2PrefetchBudget, each CTA prefetches the code
// blocks of its later tasks after issuing its first task's loads.  When the code blocks and
// T_out^T fit together, it also prefetches the T_out^T tiles of its synthesis tasks, once it
// reaches its first code-product task: by then its analysis loads are out, and the code
// product, bounded by the decode, leaves HBM mostly idle (prefetching them earlier competes with
// the analysis stream; prefetching part of a larger layer's T_out^T measured no faster).
constexpr int64_t kL2PrefetchBudget = 64ll << 20;

struct DecPhase {
  int R, K, RT, KB, kbs;
  __nv_bfloat16* out;     // [M][R]
  uint32_t* flags;        // [RT][kWsSlices] slice final in this call when == generation + 1
  // A block-sparse weight operand (frames in structured form), else null: row tile t reads
  // only K blocks aidx[3t] .. aidx[3t+1]-1, stored as contiguous pre-swizzled 16 KiB tiles
  // from tile aidx[3t+2] of atiles on
  const uint8_t* atiles;
  const int32_t* aidx;
  int acount;             // stored tiles of atiles
};

// One launch runs up to kMaxGroup independent layers (no layer reads another's output), e.g.
// q, k and v of an attention block, or gate and up of an MLP; a single layer is a group of 1.
constexpr int kMaxGroup = FQ_MAX_GROUP;

struct DecLayer {
  DecPhase ph[3];
  const uint32_t* words;
  const __half* scale;
  const __half* zero;
  const float* gamma;
  int pf_tout;            // prefetch the T_out^T tiles of this CTA's synthesis tasks into L2
};

// Tensor maps per layer: T_in, x, z, T_out^T, u.
enum { kMapTin = 0, kMapX = 1, kMapZ = 2, kMapTout = 3, kMapU = 4, kMapsPerLayer = 5 };
struct DecMaps {
  CUtensorMap m[kMaxGroup][kMapsPerLayer];
};

struct DecArgs {
  int M, S, total, G;
  DecLayer L[kMaxGroup];
  int32_t* status;
  uint32_t* gen;
  uint32_t* done;
  int pf_codes;           // prefetch this CTA's later code blocks into L2
  int ext_in;             // bit p: phase p's input was written before the launch (no flags)
  const char* pf_next;    // a range to warm in L2 from the first synthesis task (next layer)
  int64_t pf_next_bytes;  // its length, a multiple of 16 (0: none)
  // Test hook (0 in normal use): > 0 makes the activation producer's waits for another
  // phase's slices expect a stamp no call ever writes and give up after this many cycles, so
  // that the timeout path can be exercised without a fault (one-CTA launches only).
  int64_t inject_wait;
};

// Per-cluster task lists, a kernel parameter: cluster c runs task[off[c]] .. task[off[c+1]-1].
constexpr int kMaxClusters = 160;
constexpr int kMaxSched = 3 * kWsMaxTiles;
constexpr int kTileBits = 12;                  // row tiles per phase < 4096
struct DecSched {
  uint16_t off[kMaxClusters + 1];
  uint16_t task[kMaxSched];          // layer << 14 | phase << 12 | row tile
};

template <int BN>
struct DecLayout {
  static constexpr int kBTile = BN * kBK * 2;
  static constexpr int kStage = kATile + kBTile + kCodeBytes;
  static constexpr int kRecvRow = BN + 4;                     // floats per received row
  static constexpr int kRecv = kBM * kRecvRow * 4;            // [S][128/S][BN + 4] fp32
  static constexpr int NI = DecCfg<BN>::NI;
  // a multiple of NI: issuer q owns stages q, q + NI, ...
  static constexpr int kStages =
      std::min(12, (216 * 1024 - 4096 - 2 * kRecv) / kStage) / NI * NI;
  static constexpr int kAccCols = 2 * NI * BN;               // [2 buffers][NI issuers][BN]
  static constexpr uint32_t kTmemCols =
      kAccCols <= 32 ? 32 : (kAccCols <= 64 ? 64 : (kAccCols <= 128 ? 128 : 256));
  static constexpr int oA = 0;
  static constexpr int oB = oA + kStages * kATile;
  static constexpr int oC = oB + kStages * kBTile;
  static constexpr int oRecv = oC + kStages * kCodeBytes;    // two receive buffers
  static constexpr int oBar = oRecv + 2 * kRecv;
  static constexpr int kBars = 4 * kStages + 10;
  static constexpr int oMisc = oBar + kBars * 8;
  static constexpr int oZs = oMisc + 32;                     // [BN] floats
  static constexpr int oZsPart = oZs + BN * 4;               // [128] floats
  static constexpr int kBytes = oZsPart + kEpi * 4 + 1024;
  static_assert(kBTile % 1024 == 0, "B tiles keep 1024-byte alignment");
  static_assert(kStages >= 3 && kStages % NI == 0, "pipeline depth, stage ownership");
  static_assert(kAccCols <= 256, "accumulator columns");
  static_assert(kBytes <= 227 * 1024, "shared memory per CTA");
};

__device__ __forceinline__ uint4 ldcg_u4(const __nv_bfloat16* p) {
  return __ldcg(reinterpret_cast<const uint4*>(p));
}

struct Task {
  int l, p, tile;
};

// by value: the roles keep a task's phase constants in registers (loads from the parameter
// space with a dynamic index are not free in the flag-polling and copy loops)
__device__ __forceinline__ DecPhase phase_of(const DecArgs& a, int l, int p) {
  return a.L[l].ph[p];
}

__device__ __forceinline__ Task task_at(const DecSched& sc, int ti) {
  const uint32_t e = sc.task[ti];
  return {static_cast<int>(e >> 14), static_cast<int>((e >> kTileBits) & 3u),
          static_cast<int>(e & ((1u << kTileBits) - 1))};
}

// q -> bf16(4 + q) (exact: 4 .. 7 need 3 significant bits), one 128-byte row of a K-major tile
// with the 128-byte swizzle (16-byte chunk c of row r lands at chunk c ^ (r mod 8)).  Columns
// 2p and 2p + 1 of a word sit at bits 2p and 2p + 16; one shift puts them at bits 5 and 21, the
// two mantissa bits below the leading one of 4.0 (0x4080), and one AND-OR adds the exponent.
// The MMA then yields sum_j (4 + q_j) z_j, and the epilogue subtracts 4 sum_j z_j.
template <int P>
__device__ __forceinline__ uint32_t code_pair_bf16(uint32_t w) {
  const uint32_t x = P <= 2 ? (w << (5 - 2 * P)) : (w >> (2 * P - 5));
  return (x & 0x00600060u) | 0x40804080u;
}

__device__ __forceinline__ void decode_row_dec(const uint4 w4, uint8_t* tile, int r) {
  const uint32_t wv[4] = {w4.x, w4.y, w4.z, w4.w};
  uint8_t* row = tile + r * 128;
#pragma unroll
  for (int wi = 0; wi < 4; ++wi) {
    const uint32_t w = wv[wi];
    const uint4 lo = make_uint4(code_pair_bf16<0>(w), code_pair_bf16<1>(w), code_pair_bf16<2>(w),
                                code_pair_bf16<3>(w));
    const uint4 hi = make_uint4(code_pair_bf16<4>(w), code_pair_bf16<5>(w), code_pair_bf16<6>(w),
                                code_pair_bf16<7>(w));
    *reinterpret_cast<uint4*>(row + (((2 * wi) ^ (r & 7)) << 4)) = lo;
    *reinterpret_cast<uint4*>(row + (((2 * wi + 1) ^ (r & 7)) << 4)) = hi;
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
// of the header's first 32 bytes), for diagnosis together with the status word.
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
__global__ void __launch_bounds__(DecCfg<BN>::kThreads, 1)
    decode_layer_kernel(const __grid_constant__ DecMaps maps, const __grid_constant__ DecArgs a,
                        const __grid_constant__ DecSched sched) {
  using Lo = DecLayout<BN>;
  constexpr int S_ = Lo::kStages;
  constexpr int kBTile = Lo::kBTile;
  constexpr int NI = Lo::NI;

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem + Lo::oA;
  uint8_t* sB = smem + Lo::oB;
  uint8_t* sC = smem + Lo::oC;
  float* recv_buf = reinterpret_cast<float*>(smem + Lo::oRecv);
  // fullA, fullB and empty complete once in every round of their stage, cfull[s] in core
  // rounds only (its waiters keep one parity bit per stage)
  uint64_t* fullA = reinterpret_cast<uint64_t*>(smem + Lo::oBar);
  uint64_t* fullB = fullA + S_;
  uint64_t* empty = fullB + S_;
  uint64_t* cfull = empty + S_;
  uint64_t* tfull = cfull + S_;
  uint64_t* tempty = tfull + 2;
  uint64_t* mma_done = tempty + 2;     // [4] one per issuer
  uint64_t* recv_bar = mma_done + 4;   // [2] the peers' partials of this CTA's slice arrived
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + Lo::oMisc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  uint32_t* gen_s = tmem_slot + 2;
  float* zs_s = reinterpret_cast<float*>(smem + Lo::oZs);
  float* zs_part = reinterpret_cast<float*>(smem + Lo::oZsPart);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int S = a.S;
  const bool clustered = S > 1;
  uint32_t rank = 0, cid = blockIdx.x, ncl = gridDim.x;
  if (clustered) {
    rank = cluster_ctarank();
    cid = cluster_id_x();
    ncl = cluster_count_x();
  }
  const int ks = static_cast<int>(rank);
  const int t_lo = sched.off[cid], t_hi = sched.off[cid + 1];   // this cluster's tasks

  if (warp == 0) {
    // the barriers, initialised lane-parallel: fullA, fullB, empty, cfull (count 1), tfull[2]
    // (one commit per issuer), tempty[2] (kEpi), mma_done[4] (1), recv_bar[2] (1)
    // fullA takes two arrivals per round when a stage has two decoders: the weight
    // producer's two (with the tile's bytes), or one from each decoder
    constexpr uint32_t kFullA = DecCfg<BN>::kPairs ? 2u : 1u;
    for (int b = lane; b < Lo::kBars; b += 32) {
      const int r = b - 4 * S_;
      const uint32_t cnt = b < S_ ? kFullA
                                  : (r < 0 ? 1u
                                           : (r < 2 ? static_cast<uint32_t>(NI)
                                                    : (r < 4 ? static_cast<uint32_t>(kEpi)
                                                             : 1u)));
      mbar_init(&fullA[b], cnt);
    }
    fence_barrier_init();
    __syncwarp();
    if (lane == 0) {
      *abort_flag = 0;
      if (clustered) {
        // arm the receive buffers for this CTA's first two tasks (later tasks re-arm them)
        const uint32_t bytes = static_cast<uint32_t>((S - 1) * (kBM / S) * BN * 4);
        for (int b = 0; b < 2; ++b)
          if (t_lo + b < t_hi) mbar_arrive_expect_tx(&recv_bar[b], bytes);
      }
    }
    if (lane < a.G * kMapsPerLayer)
      prefetch_tmap(&maps.m[lane / kMapsPerLayer][lane % kMapsPerLayer]);
  }
  if (warp == 1) tmem_alloc(tmem_slot, Lo::kTmemCols);
  tc_fence_before_sync();
  __syncthreads();
  // Every CTA's barriers must exist before a peer pushes partial sums into it: all threads
  // arrive here, and the epilogue (the only role that writes into other CTAs) waits before its
  // first push; the other roles wait at the end.
  if (clustered) cluster_arrive();
  tc_fence_after_sync();
  const uint32_t tmem_base = *tmem_slot;
  pdl_launch_dependents();

  // this CTA's K range of a task of phase ph
  // this CTA's K range of row tile `tile` of phase ph (its own range for a block-sparse
  // operand, split over the cluster like a dense one)
  auto krange = [&](const DecPhase& ph, int tile, int& k0, int& k1) {
    if (ph.aidx) {
      const int lo = __ldg(ph.aidx + 3 * tile), hi = __ldg(ph.aidx + 3 * tile + 1);
      const int per = (hi - lo + S - 1) / S;
      k0 = lo + ks * per;
      k1 = min(hi, k0 + per);
    } else {
      k0 = ks * ph.kbs;
      k1 = min(ph.KB, k0 + ph.kbs);
    }
  };

  if (warp == 0) {
    // -------------------------------------------------------------- weight (A) producer
    {
      const uint64_t pol_w = policy_evict_first();
      int stage = 0;
      uint32_t phase = 0;
      bool tout_pf = false;
      for (int l = 0; l < a.G; ++l) tout_pf |= a.L[l].pf_tout > 0;
      bool first = true, next_pf = a.pf_next_bytes > 0;
      // this CTA's share of the next layer's range, into L2 (64 KiB per prefetch)
      auto prefetch_next = [&]() {
        next_pf = false;
        if (lane != 0) return;
        const int64_t per = ((a.pf_next_bytes + gridDim.x - 1) / gridDim.x + 15) & ~15ll;
        const int64_t b0 = static_cast<int64_t>(blockIdx.x) * per;
        const int64_t b1 = min(a.pf_next_bytes, b0 + per);
        for (int64_t o = b0; o < b1; o += 65536)
          asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(a.pf_next + o),
                       "r"(static_cast<uint32_t>(b1 - o < 65536 ? b1 - o : 65536))
                       : "memory");
      };
      // bit s: stage s filled / its last fill a code block / parity of that fill's phase of
      // fullA (weight tile) or cfull (code block)
      uint32_t used = 0, last_code = 0, last_par = 0, cpar = 0;
      bool wok = true;
      for (int i = t_lo; i < t_hi && wok; ++i) {
        if (__any_sync(0xffffffffu, *abort_flag != 0)) break;
        const Task t = task_at(sched, i);
        const DecPhase ph = phase_of(a, t.l, t.p);
        const uint32_t* words = a.L[t.l].words;
        const CUtensorMap* tmA = &maps.m[t.l][t.p == 0 ? kMapTin : kMapTout];
        int k0, k1;
        krange(ph, t.tile, k0, k1);
        // a block-sparse operand: the tile's first K block and its first stored tile
        const int a_lo = ph.aidx ? __ldg(ph.aidx + 3 * t.tile) : 0;
        const int a_off = ph.aidx ? __ldg(ph.aidx + 3 * t.tile + 2) : 0;
        if (next_pf && t.p == 2) prefetch_next();
        if (tout_pf && t.p >= 1) {
          tout_pf = false;
          // this CTA's synthesis tiles of the layers warmed in L2, in the order they will be
          // read, into L2
          for (int j = i; j < t_hi && lane == 0; ++j) {
            const Task u = task_at(sched, j);
            if (u.p != 2 || !a.L[u.l].pf_tout) continue;
            const DecPhase q = phase_of(a, u.l, u.p);
            int u0, u1;
            krange(q, u.tile, u0, u1);
            if (q.atiles) {
              const int lo = __ldg(q.aidx + 3 * u.tile), off = __ldg(q.aidx + 3 * u.tile + 2);
              if (u1 > u0)
                asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(
                                 q.atiles + static_cast<int64_t>(off + u0 - lo) * kATile),
                             "r"(static_cast<uint32_t>((u1 - u0) * kATile))
                             : "memory");
            } else {
              for (int kb = u0; kb < u1; ++kb)
                asm volatile(
                    "cp.async.bulk.prefetch.tensor.2d.L2.global.tile [%0, {%1, %2}];" ::"l"(
                        reinterpret_cast<uint64_t>(&maps.m[u.l][kMapTout])),
                    "r"(kb * kBK), "r"(u.tile * kBM)
                    : "memory");
            }
          }
        }
        for (int kb = k0; kb < k1; ++kb) {
          const bool got = mbar_wait(&empty[stage], phase ^ 1, abort_flag);
          if (!__all_sync(0xffffffffu, got)) {
            if (lane == 0) {
              if (!*abort_flag) note_timeout(a.status, 1, i, stage, static_cast<int>(phase));
              *abort_flag = 1;
            }
            wok = false;
            break;
          }
          const uint32_t bit = 1u << stage;
          used |= bit;
          if (t.p == 1) {
            if (lane == 0) {
              mbar_arrive_expect_tx(&cfull[stage], kCodeBytes);
              bulk_load(sC + stage * kCodeBytes,
                        words + (static_cast<int64_t>(t.tile) * ph.KB + kb) * 512,
                        kCodeBytes, &cfull[stage], pol_w);
            }
            last_code |= bit;
            last_par = (last_par & ~bit) | (cpar & bit);
            cpar ^= bit;
          } else {
            if (lane == 0) {
              mbar_arrive_expect_tx(&fullA[stage], kATile);
              if (DecCfg<BN>::kPairs) mbar_arrive(&fullA[stage]);
              if (ph.atiles)
                bulk_load(sA + stage * kATile,
                          ph.atiles + static_cast<int64_t>(a_off + kb - a_lo) * kATile, kATile,
                          &fullA[stage], pol_w);
              else
                tma_load_2d(sA + stage * kATile, tmA, &fullA[stage], kb * kBK, t.tile * kBM,
                            pol_w);
            }
            last_code &= ~bit;
            last_par = (last_par & ~bit) | (phase << stage);
          }
          if (++stage == S_) stage = 0, phase ^= 1;
        }
        if (first && wok) {
          first = false;
          // warm L2 with the code blocks of this CTA's later tasks
          for (int j = i + 1; j < t_hi && a.pf_codes && lane == 0; ++j) {
            const Task u = task_at(sched, j);
            const DecPhase q = phase_of(a, u.l, u.p);
            int u0, u1;
            krange(q, u.tile, u0, u1);
            if (u.p == 1 && u1 > u0) {
              const uint32_t* src =
                  a.L[u.l].words + (static_cast<int64_t>(u.tile) * q.KB + u0) * 512;
              asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src),
                           "r"(static_cast<uint32_t>((u1 - u0) * kCodeBytes))
                           : "memory");
            }
          }
        }
      }
      if (next_pf) prefetch_next();      // a CTA without synthesis tasks still takes its share
      // no copy may still be landing when the CTA leaves: the last fill of every stage (no
      // later phase of its barrier exists, so the parity wait is exact)
      for (int s = 0; s < S_ && lane == 0; ++s)
        if (((used >> s) & 1u) &&
            !mbar_wait(((last_code >> s) & 1u) ? &cfull[s] : &fullA[s], (last_par >> s) & 1u,
                       nullptr))
          report(a.status, FQ_ERR_TIMEOUT);
    }
  } else if (warp == 6) {
    // -------------------------------------------------------------- activation (B) producer
    // the whole warp polls ready flags (one lane per slice); lane 0 issues the loads
    const uint64_t pol_x = policy_evict_last();
    pdl_wait();
    if (blockIdx.x == 0 && lane == 0) {
      // a new call: clear the status word and the previous call's timeout details
      *a.status = 0;
      for (int w = 4; w < 8; ++w) a.status[w] = 0;
    }
    const uint32_t g = ld_acquire_gpu(a.gen) + 1;
    const uint32_t g_want = a.inject_wait > 0 ? g + 0x40000000u : g;
    const long long wait_limit = a.inject_wait > 0 ? a.inject_wait : kWaitLimitCycles;
    const int rows_per = kBM / S;
    int stage = 0;
    uint32_t phase = 0;
    uint32_t used = 0, last_par = 0;   // bit s: stage s filled, parity of its last fill
    for (int i = t_lo; i < t_hi; ++i) {
      if (__shfl_sync(0xffffffffu, *abort_flag != 0, 0)) break;   // warp-uniform
      const Task t = task_at(sched, i);
      const DecPhase ph = phase_of(a, t.l, t.p);
      int k0, k1;
      krange(ph, t.tile, k0, k1);
      // Loads go out in K order as soon as the slices of the previous phase's output that a K
      // block reads are final: the lanes poll the not-yet-final slices of the K range, and
      // the ready prefix decides how far lane 0 may issue.
      const DecPhase src = phase_of(a, t.l, t.p > 0 ? t.p - 1 : 0);
      const int sl1 = k1 > k0 ? (min(ph.K, k1 * kBK) - 1) / rows_per : 0;
      int ready = k1 > k0 ? (k0 * kBK) / rows_per : 0;   // slices below `ready` are final
      const long long t_start = clock64();
      bool ok = true;
      int kb = k0;
      const CUtensorMap* tm = &maps.m[t.l][t.p == 0 ? kMapX : (t.p == 1 ? kMapZ : kMapU)];
      while (kb < k1 && ok) {
        int kb_end = k1;
        if (t.p > 0 && !((a.ext_in >> t.p) & 1) && ready <= sl1) {
          // first slice (from `ready`) that is not final yet, over the whole warp
          int first_missing = sl1 + 1;
          for (int gs = ready + lane; gs <= sl1; gs += 32)
            if (ld_acquire_gpu(&src.flags[(gs / S) * kWsSlices + gs % S]) != g_want) {
              first_missing = gs;
              break;
            }
#pragma unroll
          for (int off = 16; off > 0; off >>= 1)
            first_missing = min(first_missing, __shfl_xor_sync(0xffffffffu, first_missing, off));
          ready = first_missing;
          // K blocks whose rows all lie below the first missing slice
          kb_end = ready > sl1 ? k1 : min(k1, (ready * rows_per) / kBK);
          if (kb_end <= kb) {
            // lane 0 decides for the warp, so that every lane leaves the loop together
            if (__shfl_sync(0xffffffffu, clock64() - t_start > wait_limit || *abort_flag, 0)) {
              if (lane == 0 && !*abort_flag) {
                const uint32_t* f = &src.flags[(ready / S) * kWsSlices + ready % S];
                note_timeout(a.status, 2, i, ready, static_cast<int>(ld_acquire_gpu(f) - g) * 1000 + t.p);
              }
              ok = false;
              break;
            }
            __nanosleep(64);
            continue;
          }
        }
        for (; kb < kb_end; ++kb) {
          const bool got = mbar_wait(&empty[stage], phase ^ 1, abort_flag);
          if (!__all_sync(0xffffffffu, got)) {
            if (lane == 0 && !*abort_flag) note_timeout(a.status, 3, i, stage, static_cast<int>(phase));
            ok = false;
            break;
          }
          if (lane == 0) {
            mbar_arrive_expect_tx(&fullB[stage], kBTile);
            tma_load_2d(sB + stage * kBTile, tm, &fullB[stage], kb * kBK, 0, pol_x);
          }
          used |= 1u << stage;
          last_par = (last_par & ~(1u << stage)) | (phase << stage);
          if (++stage == S_) stage = 0, phase ^= 1;
        }
      }
      if (!ok && lane == 0) *abort_flag = 1;
      if (!__shfl_sync(0xffffffffu, ok, 0)) break;
    }
    if (lane == 0)
      for (int s = 0; s < S_; ++s)
        if (((used >> s) & 1u) && !mbar_wait(&fullB[s], (last_par >> s) & 1u, nullptr))
          report(a.status, FQ_ERR_TIMEOUT);
  } else if (issuer_of(warp, NI) >= 0) {
    // -------------------------------------------------------------- MMA issuers
    // issuer q: the K blocks that land in ring stages s = q (mod NI), into accumulator q of
    // the task's buffer; every issuer walks every round to follow the ring
    const int q = issuer_of(warp, NI);
    if (lane == 0) {
      constexpr uint32_t idesc = umma_idesc_bf16(kBM, BN);
      int stage = 0;
      uint32_t phase = 0;
      int buf = 0;
      uint32_t acc_phase = 0;
      bool issued_any = false;
      for (int i = t_lo; i < t_hi && !*abort_flag; ++i) {
        const Task t = task_at(sched, i);
        const DecPhase ph = phase_of(a, t.l, t.p);
        int k0, k1;
        krange(ph, t.tile, k0, k1);
        if (!mbar_wait(&tempty[buf], acc_phase ^ 1, abort_flag)) {
          if (!*abort_flag) note_timeout(a.status, 4, i, buf, static_cast<int>(acc_phase));
          *abort_flag = 1;
          break;
        }
        tc_fence_after_sync();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>((buf * NI + q) * BN);
        bool ok = true;
        bool acc = false;      // this issuer has accumulated a K block of the task
        for (int kb = k0; kb < k1; ++kb) {
          if (stage % NI == q) {
            ok = mbar_wait(&fullA[stage], phase, abort_flag);
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
              umma_bf16(d_tmem, adesc + 2 * k, bdesc + 2 * k, idesc, (acc || k > 0) ? 1u : 0u);
            acc = true;
            issued_any = true;
            umma_commit(&empty[stage]);
          }
          if (++stage == S_) stage = 0, phase ^= 1;
        }
        if (!ok) {
          *abort_flag = 1;
          break;
        }
        umma_commit(&tfull[buf]);      // with no K block of its own this arrives at once
        if (++buf == 2) buf = 0, acc_phase ^= 1;
      }
      if (issued_any) {
        umma_commit(&mma_done[q]);
        if (!mbar_wait(&mma_done[q], 0, nullptr)) report(a.status, FQ_ERR_TIMEOUT);
      }
    }
  } else if ((warp >= 7 && warp <= 10) || (DecCfg<BN>::kPairs && warp >= 16 && warp <= 19)) {
    // -------------------------------------------------------------- code decoders
    // Decoder d (warps 7-10, and 16-19 with decoder pairs) expands the code blocks of the core
    // rounds that land in ring stages s = d (mod 4) into the stage's A slot (with pairs, rows
    // 0-63 by warp 7 + d and rows 64-127 by warp 16 + d); it waits for nothing else.  All lanes
    // wait (measured: one polling lane with the others parked in a shuffle wakes later).
    const int dw = warp <= 10 ? warp - 7 : warp - 16;
    constexpr int kRR = DecCfg<BN>::kPairs ? 2 : 4;         // 32-row groups per decoder
    const int rr0 = warp <= 10 ? 0 : 2;
    int stage = 0;
    uint32_t cpar = 0;     // bit s: parity of the next cfull[s] phase
    bool ok = true;
    for (int i = t_lo; i < t_hi && ok; ++i) {
      if (__shfl_sync(0xffffffffu, *abort_flag != 0, 0)) break;   // warp-uniform
      const Task t = task_at(sched, i);
      const DecPhase ph = phase_of(a, t.l, t.p);
      int k0, k1;
      krange(ph, t.tile, k0, k1);
      const int n = max(0, k1 - k0);
      if (t.p != 1) {
        stage = (stage + n) % S_;
        continue;
      }
      for (int kb = 0; kb < n; ++kb) {
        if ((stage & 3) == dw) {
          const bool got = mbar_wait(&cfull[stage], (cpar >> stage) & 1u, abort_flag);
          if (!got && lane == 0 && !*abort_flag) note_timeout(a.status, 7, i, stage, static_cast<int>(cpar));
          cpar ^= 1u << stage;
          if (!__all_sync(0xffffffffu, got)) {
            ok = false;
            break;
          }
          const uint4* codes = reinterpret_cast<const uint4*>(sC + stage * kCodeBytes);
          uint8_t* tile_a = sA + stage * kATile;
#pragma unroll
          for (int rr = rr0; rr < rr0 + kRR; ++rr)
            decode_row_dec(codes[lane + 32 * rr], tile_a, lane + 32 * rr);
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) mbar_arrive(&fullA[stage]);
        }
        if (++stage == S_) stage = 0;
      }
    }
    if (!ok && lane == 0) {
      report(a.status, FQ_ERR_TIMEOUT);
      *abort_flag = 1;
    }
  } else if (warp >= 2 && warp <= 5) {
    // -------------------------------------------------------------- epilogue (warps 2-5)
    const int quarter = warp & 3;                 // TMEM lanes 32 * quarter .. + 31
    const int r_in_tile = quarter * 32 + lane;
    const int et = threadIdx.x - 64;
    const int rows_per = kBM / S;                 // rows of a tile per slice (one per CTA)
    const int dest = r_in_tile / rows_per;        // CTA that reduces this thread's row
    const int rl_own = r_in_tile % rows_per;
    constexpr int kRow = Lo::kRecvRow;
    const uint32_t recv_bytes = static_cast<uint32_t>((S - 1) * rows_per * BN * 4);
    pdl_wait();
    if (et == 0) *gen_s = ld_acquire_gpu(a.gen) + 1;
    named_barrier_sync(1, kEpi);
    if (clustered) cluster_wait();
    const uint32_t g = *gen_s;
    int buf = 0;
    uint32_t acc_phase = 0;
    int ring_pos = 0;                             // ring stage of the next task's first K block
    int j = 0;                                    // tasks finished by this CTA
    for (int i = t_lo; i < t_hi; ++i, ++j) {
      const Task t = task_at(sched, i);
      const DecPhase ph = phase_of(a, t.l, t.p);
      const DecPhase ph_z = phase_of(a, t.l, 0);      // the layer's z and its ready flags
      const __half* l_scale = a.L[t.l].scale;
      const __half* l_zero = a.L[t.l].zero;
      const float* l_gamma = a.L[t.l].gamma;
      int k0, k1;
      krange(ph, t.tile, k0, k1);
      const bool has_k = k1 > k0;
      const int row = t.tile * kBM + r_in_tile;
      const bool row_ok = row < ph.R;
      float s_i = 0.f, z_i = 0.f, g_row = 1.f;
      if (t.p == 1 && row_ok) {
        s_i = __half2float(l_scale[row]);
        z_i = __half2float(l_zero[row]);
        if (l_gamma) g_row = l_gamma[row];
      }
      const float zb_i = z_i - 4.f * s_i;          // the decoded codes carry an offset of 4
      bool fail = false;
      if (t.p == 1) {
        // sum of z over this CTA's K range: first the ready flags of the slices it reads
        if (has_k && !(a.ext_in & 2)) {
          const int sl0 = (k0 * kBK) / rows_per, sl1 = (min(ph.K, k1 * kBK) - 1) / rows_per;
          for (int gs = sl0 + et; gs <= sl1 && !fail; gs += kEpi) {
            fail = !wait_flag(&ph_z.flags[(gs / S) * kWsSlices + gs % S], g, abort_flag);
            if (fail && !*abort_flag) note_timeout(a.status, 8, i, gs, 0);
          }
        }
        if (bar_red_or_dec(1, kEpi, fail)) {
          if (et == 0) *abort_flag = 1;
          break;
        }
        {
          // 128 / BN threads per token each add a strided share of the token's z, then one
          // thread per token adds the shares in a fixed order
          constexpr int kPer = kEpi / BN;
          const int q = et % BN, part = et / BN;
          float sz = 0.f;
          if (q < a.M && has_k) {
            // z columns k0 * 64 .. of token q: multiples of 8 (n_in is a multiple of 16), so
            // 16-byte loads from L2, each thread a strided share
            const int c0 = k0 * kBK, c1 = min(ph.K, k1 * kBK);
            const __nv_bfloat16* zr = ph_z.out + static_cast<int64_t>(q) * ph.K;
            for (int c = c0 + 8 * part; c < c1; c += 8 * kPer) {
              const uint4 w = ldcg_u4(zr + c);
              const uint32_t wv[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&wv[e]));
                sz += f.x + f.y;
              }
            }
          }
          zs_part[part * BN + q] = sz;
          named_barrier_sync(1, kEpi);
          if (et < BN) {
            float tot = 0.f;
#pragma unroll
            for (int r = 0; r < kPer; ++r) tot += zs_part[r * BN + et];
            zs_s[et] = tot;
          }
        }
      }
      // one thread waits, the others block in the named barrier below
      if (et == 0 && !mbar_wait(&tfull[buf], acc_phase, abort_flag)) {
        fail = true;
        if (!*abort_flag) note_timeout(a.status, 9, i, buf, static_cast<int>(acc_phase));
      }
      if (bar_red_or_dec(1, kEpi, fail || *abort_flag)) {
        if (et == 0) *abort_flag = 1;
        break;
      }
      tc_fence_after_sync();
      const uint32_t t_row = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) +
                             static_cast<uint32_t>(buf * NI * BN);
      // issuers that accumulated K blocks of this task: those owning the task's first
      // min(NI, K blocks) ring stages
      const int nkb = max(0, k1 - k0);
      const int ring0 = ring_pos % NI;
      ring_pos = (ring_pos + nkb) % S_;
      // this thread's row of the accumulator (for the core: gamma (s Q z + zero sum z) over the
      // CTA's K range), the issuers' accumulators added in issuer order
      float vals[BN];
#pragma unroll
      for (int c = 0; c < BN; c += kChunk) {
        float v[kChunk];
#pragma unroll
        for (int q = 0; q < kChunk; ++q) v[q] = 0.f;
        for (int qa = 0; qa < NI; ++qa) {
          if ((qa - ring0 + NI) % NI >= nkb) continue;       // uniform across the warp
          float w[kChunk];
          tmem_ld16(t_row + static_cast<uint32_t>(qa * BN + c), w);
          tmem_wait_ld();
#pragma unroll
          for (int q = 0; q < kChunk; ++q) v[q] += w[q];
        }
#pragma unroll
        for (int q = 0; q < kChunk; ++q)
          vals[c + q] = t.p == 1 ? g_row * fmaf(s_i, v[q], zb_i * zs_s[c + q]) : v[q];
      }
      tc_fence_before_sync();
      mbar_arrive(&tempty[buf]);

      if (!clustered) {
        // one CTA per task: this thread owns one row of the tile
#pragma unroll
        for (int c = 0; c < BN; ++c) {
          const __nv_bfloat16 b = __float2bfloat16_rn(vals[c]);
          if (row_ok && c < a.M) ph.out[static_cast<int64_t>(c) * ph.R + row] = b;
        }
        if (t.p < 2) {
          named_barrier_sync(1, kEpi);
          if (et == 0) st_release_gpu(&ph.flags[t.tile * kWsSlices], g);
        }
      } else {
        // ---- push this row into slot `ks` of the owning CTA's receive buffer
        const int rb = j & 1;
        float* recv = recv_buf + rb * (kBM * kRow);
        const int slot_row = ks * rows_per + rl_own;
        if (dest == ks) {
          float4* dst = reinterpret_cast<float4*>(recv + slot_row * kRow);
#pragma unroll
          for (int c4 = 0; c4 < BN / 4; ++c4)
            dst[c4] = make_float4(vals[4 * c4], vals[4 * c4 + 1], vals[4 * c4 + 2], vals[4 * c4 + 3]);
        } else {
          const uint32_t rdst = mapa(smem_u32(recv + slot_row * kRow), static_cast<uint32_t>(dest));
          const uint32_t rbar = mapa(smem_u32(&recv_bar[rb]), static_cast<uint32_t>(dest));
#pragma unroll
          for (int c4 = 0; c4 < BN / 4; ++c4)
            st_async_v4(rdst + 16 * c4, vals[4 * c4], vals[4 * c4 + 1], vals[4 * c4 + 2],
                        vals[4 * c4 + 3], rbar);
        }
        // ---- the S - 1 peers' partials of this CTA's slice
        bool ok = true;
        if (et == 0) {
          ok = mbar_wait(&recv_bar[rb], static_cast<uint32_t>(j >> 1) & 1u, abort_flag);
          if (!ok && !*abort_flag) note_timeout(a.status, 11, i, j, 0);
        }
        if (bar_red_or_dec(1, kEpi, !ok)) {   // also orders this CTA's own slot writes
          if (et == 0) *abort_flag = 1;
          break;
        }
        // re-arm the buffer for this CTA's task after next; its peers write it only after
        // this CTA has sent them the next task's partials, i.e. after the reads below
        if (et == 0 && i + 2 < t_hi)
          mbar_arrive_expect_tx(&recv_bar[rb], recv_bytes);
        // ---- reduce the slice in rank order; item = (row of the slice, 4 tokens), so 16-row
        // groups sit in 16 consecutive lanes (items per warp are all valid or all not)
        const int items = rows_per * (BN / 4);
        for (int w = et; w < items; w += kEpi) {
          const int rl = w % rows_per, tg = w / rows_per;
          float4 acc = *reinterpret_cast<const float4*>(recv + rl * kRow + 4 * tg);
          for (int q = 1; q < S; ++q) {
            const float4 v = *reinterpret_cast<const float4*>(recv + (q * rows_per + rl) * kRow + 4 * tg);
            acc.x += v.x;
            acc.y += v.y;
            acc.z += v.z;
            acc.w += v.w;
          }
          const int orow = t.tile * kBM + ks * rows_per + rl;
          const bool ok_r = orow < ph.R;
          const float o[4] = {acc.x, acc.y, acc.z, acc.w};
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int tok = 4 * tg + u;
            const __nv_bfloat16 b = __float2bfloat16_rn(o[u]);
            if (ok_r && tok < a.M) ph.out[static_cast<int64_t>(tok) * ph.R + orow] = b;
          }
        }
        if (t.p < 2) {
          // the slice is stored: publish it
          named_barrier_sync(1, kEpi);
          if (et == 0) st_release_gpu(&ph.flags[t.tile * kWsSlices + ks], g);
        }
      }
      if (++buf == 2) buf = 0, acc_phase ^= 1;
    }
  }

  tc_fence_before_sync();
  __syncthreads();
  // No CTA leaves while a peer may still write into its shared memory (after a wait that gave
  // up, the exchange can be cut short); every wait above is bounded, so all CTAs get here.
  if (clustered) {
    if (warp < 2 || warp > 5) cluster_wait();    // the epilogue waited before its first push
    cluster_sync();
  }
  if (threadIdx.x == 0) {
    // the last CTA to finish moves the workspace to the next call's generation
    __threadfence();
    const unsigned old = atomicInc(a.done, gridDim.x - 1);
    if (old == gridDim.x - 1) {
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
  size_t z, u, total;
};

DecWs dec_ws(int M, int n_in, int n_out) {
  DecWs L{};
  size_t off = kWsHeader;
  L.z = off;
  off += round_up(static_cast<int64_t>(M) * n_in * 2, 256);
  L.u = off;
  off += round_up(static_cast<int64_t>(M) * n_out * 2, 256);
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

// Co-resident clusters of S CTAs of this kernel on the current device (0 if none).
template <int BN>
int max_clusters(int dev, int S) {
  static std::mutex mu;
  static std::map<std::pair<int, int>, int> cache;
  std::lock_guard<std::mutex> g(mu);
  const auto key = std::make_pair(dev, S);
  const auto it = cache.find(key);
  if (it != cache.end()) return it->second;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(static_cast<unsigned>(S * 64));
  cfg.blockDim = dim3(DecCfg<BN>::kThreads);
  cfg.dynamicSmemBytes = DecLayout<BN>::kBytes;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = static_cast<unsigned>(S);
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, decode_layer_kernel<BN>, &cfg) != cudaSuccess) {
    cudaGetLastError();
    n = 0;
  }
  cache[key] = n;
  return n;
}

// One phase of one layer of a launch: rows R of its output, reduction length K, and the K of
// the layer's next phase (0 if none), whose splits its tiles are ordered by.
struct Block {
  int l, p, R, K, K_next;
};

// Launch order of the (layer, phase) blocks.  A single layer runs its three phases in order.  A
// group runs them along diagonals, block (l, p) at position l + p and lower phases first:
//     A0 A1 C0 A2 C1 S0 C2 S1 S2   (three layers; A analysis, C code product, S synthesis),
// so that each layer's phase boundaries have another layer's streaming behind them, and every
// block still comes after the block it reads (same layer, previous phase).
std::vector<Block> launch_order(int G, const int (*R)[3], const int (*K)[3]) {
  std::vector<Block> v;
  for (int l = 0; l < G; ++l)
    for (int p = 0; p < 3; ++p)
      if (R[l][p] > 0) v.push_back({l, p, R[l][p], K[l][p], p < 2 ? K[l][p + 1] : 0});
  std::stable_sort(v.begin(), v.end(), [](const Block& x, const Block& y) {
    return x.l + x.p != y.l + y.p ? x.l + x.p < y.l + y.p : x.p < y.p;
  });
  return v;
}

// Task lists for `ncl` clusters of S CTAs: the blocks' tiles, concatenated in launch order, dealt
// round-robin (each block spreads evenly and starts on the clusters the previous one left least
// busy).  Within a block whose layer has a next phase, tiles are ordered by their offset inside
// that phase's K splits, so that every split of the next phase finds its first K blocks among
// the first tiles produced.
void build_schedule(const std::vector<Block>& blocks, int S, int ncl, DecSched* out) {
  std::vector<std::vector<uint16_t>> lists(ncl);
  std::vector<int> order;
  int pos = 0;
  for (const Block& b : blocks) {
    const int RT = static_cast<int>(ceil_div(b.R, kBM));
    order.resize(RT);
    for (int t = 0; t < RT; ++t) order[t] = t;
    const int kbs_next = static_cast<int>(ceil_div(ceil_div(b.K_next, kBK), S));
    if (kbs_next > 0) {
      const int64_t split_rows = static_cast<int64_t>(kbs_next) * kBK;
      std::stable_sort(order.begin(), order.end(), [&](int x, int y) {
        return (static_cast<int64_t>(x) * kBM) % split_rows <
               (static_cast<int64_t>(y) * kBM) % split_rows;
      });
    }
    for (int t : order)
      lists[pos++ % ncl].push_back(
          static_cast<uint16_t>((b.l << 14) | (b.p << kTileBits) | t));
  }
  int n = 0;
  for (int c = 0; c < ncl; ++c) {
    out->off[c] = static_cast<uint16_t>(n);
    for (uint16_t e : lists[c]) out->task[n++] = e;
  }
  out->off[ncl] = static_cast<uint16_t>(n);
}

struct Plan {
  int S = 0, ncl = 0;
  DecSched sched{};
};

// Cluster size and task lists for a launch's blocks, cached.  Cluster size: the busiest
// cluster's K blocks over the blocks, with a fixed cost per task (pipeline fill and drain,
// reduction) and code blocks weighted by their smaller bytes.
template <int BN>
const Plan* plan_for(int dev, int sms, int budget, const std::vector<Block>& blocks) {
  static std::mutex mu;
  static std::map<std::vector<int>, Plan> cache;
  std::vector<int> key{dev, budget};
  for (const Block& b : blocks) key.insert(key.end(), {b.l, b.p, b.R, b.K, b.K_next});
  std::lock_guard<std::mutex> g(mu);
  const auto it = cache.find(key);
  if (it != cache.end()) return &it->second;
  int total = 0;
  for (const Block& b : blocks) total += static_cast<int>(ceil_div(b.R, kBM));
  Plan best;
  double best_cost = 1e30;
  for (int S : {1, 2, 4, 8}) {
    // A budget below the SM count takes its share of the device's resident clusters, so
    // that calls whose budgets add up to at most the SM count are resident together.
    int ncl = budget;
    if (S > 1) {
      const int mc = max_clusters<BN>(dev, S);
      ncl = budget >= sms ? mc : static_cast<int>(static_cast<int64_t>(mc) * budget / sms);
    }
    ncl = std::min({ncl, total, kMaxClusters});
    if (ncl <= 0) continue;
    double cost = 0;
    for (const Block& b : blocks) {
      const int RT = static_cast<int>(ceil_div(b.R, kBM));
      const int KB = static_cast<int>(ceil_div(b.K, kBK));
      const double w = b.p == 1 ? 0.35 : 1.0;
      cost += static_cast<double>(ceil_div(RT, ncl)) * (w * ceil_div(KB, S) + 4.0);
    }
    if (cost < best_cost - 1e-9) {
      best_cost = cost;
      best.S = S;
      best.ncl = ncl;
    }
  }
  if (best.S == 0) return nullptr;
  build_schedule(blocks, best.S, best.ncl, &best.sched);
  return &(cache[key] = best);
}

template <int BN>
fq_status run(const DecMaps& maps, DecArgs& a, const std::vector<Block>& blocks, int sms,
              int budget, cudaStream_t s) {
  int dev = 0;
  cudaGetDevice(&dev);
  if (prepare<BN>(dev) != cudaSuccess) return FQ_ERR_CUDA;
  int total = 0;
  for (const Block& b : blocks) total += static_cast<int>(ceil_div(b.R, kBM));
  if (total > kMaxSched) return FQ_ERR_UNSUPPORTED;
  const Plan* plan = plan_for<BN>(dev, sms, budget, blocks);
  if (!plan) return FQ_ERR_CUDA;
  a.S = plan->S;
  for (int l = 0; l < a.G; ++l)
    for (int p = 0; p < 3; ++p) {
      DecPhase& ph = a.L[l].ph[p];
      ph.RT = static_cast<int>(ceil_div(ph.R, kBM));
      ph.KB = static_cast<int>(ceil_div(ph.K, kBK));
      ph.kbs = static_cast<int>(ceil_div(ph.KB, plan->S));
    }
  a.total = total;
  {
    // L2 warming within one budget for the whole launch: the code blocks of every layer, then
    // the T_out^T of as many layers (in order) as fit with them
    int64_t code_bytes = 0;
    for (int l = 0; l < a.G; ++l)
      code_bytes += static_cast<int64_t>(a.L[l].ph[1].R) * a.L[l].ph[1].K / 4;
    a.pf_codes = code_bytes <= kL2PrefetchBudget;
    int64_t warm = code_bytes;
    bool any_tout = false;
    for (int l = 0; l < a.G; ++l) {
      const DecPhase& sy = a.L[l].ph[2];
      warm += sy.atiles ? static_cast<int64_t>(sy.acount) * kATile
                        : static_cast<int64_t>(sy.R) * sy.K * 2;
      a.L[l].pf_tout = a.L[l].ph[2].R > 0 && warm <= kL2PrefetchBudget;
      any_tout |= a.L[l].pf_tout != 0;
    }
    // the next layer's range only when this launch's last synthesis reads from L2 (HBM idle),
    // and at most the warming budget
    a.pf_next_bytes = any_tout && a.L[a.G - 1].pf_tout
                          ? std::min<int64_t>(a.pf_next_bytes, kL2PrefetchBudget)
                          : 0;
  }
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(static_cast<unsigned>(plan->ncl * plan->S));
  cfg.blockDim = dim3(DecCfg<BN>::kThreads);
  cfg.dynamicSmemBytes = DecLayout<BN>::kBytes;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = static_cast<unsigned>(plan->S);
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = plan->S > 1 ? 2 : 1;
  return cudaLaunchKernelEx(&cfg, decode_layer_kernel<BN>, maps, a, plan->sched) == cudaSuccess
             ? FQ_OK
             : FQ_ERR_CUDA;
}

// Workspace of a launch: the 64 KiB header, then z and u of every layer.
struct DecWsGroup {
  size_t z[kMaxGroup], u[kMaxGroup], total;
};

DecWsGroup dec_ws_group(int M, int G, const DecGroupLayer* Ls) {
  DecWsGroup W{};
  size_t off = kWsHeader;
  for (int l = 0; l < G; ++l) {
    W.z[l] = off;
    off += round_up(static_cast<int64_t>(M) * Ls[l].C.n_in * 2, 256);
    W.u[l] = off;
    off += round_up(static_cast<int64_t>(M) * Ls[l].C.n_out * 2, 256);
  }
  W.total = off;
  return W;
}

}  // namespace

size_t decode_workspace_bytes(int M, int d_in, int n_in, int n_out, int d_out) {
  (void)d_in;
  (void)d_out;
  return dec_ws(M, n_in, n_out).total;
}

size_t decode_group_workspace_bytes(int M, int G, const DecGroupLayer* layers) {
  if (G < 1 || G > kMaxGroup) return 0;
  return dec_ws_group(M, G, layers).total;
}

// The fused kernel over a group of G independent layers (G = 1: one layer), or (core_only,
// G = 1) over the code product alone with z already in the workspace and u left there.
fq_status launch_decode_group(int M, int G, const DecGroupLayer* Ls, char* ws, size_t ws_bytes,
                              int max_sms, bool core_only, const void* pf, size_t pf_bytes,
                              int64_t inject_wait, cudaStream_t s) {
  if (G < 1 || G > kMaxGroup || (core_only && G != 1)) return FQ_ERR_INVALID_ARG;
  const DecWsGroup W = dec_ws_group(M, G, Ls);
  if (ws_bytes < W.total) return FQ_ERR_WORKSPACE;
  const int BN = decode_bn(M);
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (sms <= 0) return FQ_ERR_CUDA;
  const int budget = max_sms > 0 ? std::min(sms, max_sms) : sms;
  if (inject_wait > 0 && budget != 1) return FQ_ERR_INVALID_ARG;   // one CTA, no cluster peers

  DecArgs a{};
  a.M = M;
  a.G = G;
  int R[kMaxGroup][3], K[kMaxGroup][3], Keff[kMaxGroup][3];
  uint32_t* flag_base = reinterpret_cast<uint32_t*>(ws + kWsFlags);
  const int64_t flag_words = static_cast<int64_t>(kWsHeader - kWsFlags) / 4;
  int64_t flag_off = 0;
  DecMaps maps;
  for (int l = 0; l < G; ++l) {
    const DecGroupLayer& Ly = Ls[l];
    const int n_in = Ly.C.n_in, n_out = Ly.C.n_out;
    const int Rl[3] = {core_only ? 0 : n_in, n_out, core_only ? 0 : Ly.d_out};
    const int Kl[3] = {core_only ? 0 : Ly.d_in, n_in, core_only ? 0 : n_out};
    void* outs[3] = {ws + W.z[l], ws + W.u[l], core_only ? static_cast<void*>(ws + W.u[l]) : Ly.y};
    const SparseOperand* sp[3] = {&Ly.tin, nullptr, &Ly.tout};
    for (int p = 0; p < 3; ++p) {
      R[l][p] = Rl[p];
      K[l][p] = Kl[p];
      Keff[l][p] = Kl[p];
      const int RT = static_cast<int>(ceil_div(Rl[p], kBM));
      if (RT > kWsMaxTiles || RT >= (1 << kTileBits)) return FQ_ERR_UNSUPPORTED;
      DecPhase& ph = a.L[l].ph[p];
      ph.R = Rl[p];
      ph.K = Kl[p];
      ph.out = static_cast<__nv_bfloat16*>(outs[p]);
      if (sp[p] && sp[p]->tiles && Rl[p] > 0) {
        ph.atiles = sp[p]->tiles;
        ph.aidx = sp[p]->idx;
        ph.acount = sp[p]->count;
        // the cost model's K: the operand's stored K blocks per row tile
        Keff[l][p] = static_cast<int>(ceil_div(static_cast<int64_t>(sp[p]->count) * kBK, RT));
      }
      if (G == 1) {
        // one layer: the phases' flags at fixed places of the header
        ph.flags = flag_base + p * kWsMaxTiles * kWsSlices;
      } else if (p < 2) {
        // a group: the flags of the analysis and code-product slices, packed in layer order
        // (the synthesis publishes none); every flag of the header only ever holds a past
        // generation, whichever layout wrote it
        ph.flags = flag_base + flag_off;
        flag_off += static_cast<int64_t>(RT) * kWsSlices;
        if (flag_off > flag_words) return FQ_ERR_UNSUPPORTED;
      } else {
        ph.flags = flag_base;
      }
    }
    a.L[l].words = Ly.C.words;
    a.L[l].scale = reinterpret_cast<const __half*>(Ly.C.scale_f16);
    a.L[l].zero = reinterpret_cast<const __half*>(Ly.C.zero_f16);
    a.L[l].gamma = Ly.gamma;
    CUtensorMap* m = maps.m[l];
    if (!tmap_bf16(&m[kMapZ], ws + W.z[l], M, n_in, BN) ||
        !tmap_bf16(&m[kMapU], ws + W.u[l], M, n_out, BN))
      return FQ_ERR_CUDA;
    if (core_only) {
      // no analysis or synthesis tasks: their maps are never used for a copy
      m[kMapTin] = m[kMapZ];
      m[kMapX] = m[kMapZ];
      m[kMapTout] = m[kMapU];
    } else {
      // block-sparse operands are copied whole tiles at a time: their maps are never used
      if (!tmap_bf16(&m[kMapX], Ly.x, M, Ly.d_in, BN)) return FQ_ERR_CUDA;
      if (Ly.tin.tiles)
        m[kMapTin] = m[kMapX];
      else if (!tmap_bf16(&m[kMapTin], Ly.T_in, n_in, Ly.d_in, kBM))
        return FQ_ERR_CUDA;
      if (Ly.tout.tiles)
        m[kMapTout] = m[kMapU];
      else if (!tmap_bf16(&m[kMapTout], Ly.T_out_t, Ly.d_out, n_out, kBM))
        return FQ_ERR_CUDA;
    }
  }
  for (int l = G; l < kMaxGroup; ++l)
    for (int k = 0; k < kMapsPerLayer; ++k) maps.m[l][k] = maps.m[0][k];
  a.status = reinterpret_cast<int32_t*>(ws);
  a.gen = reinterpret_cast<uint32_t*>(ws + kWsGen);
  a.done = reinterpret_cast<uint32_t*>(ws + kWsDone);
  a.ext_in = core_only ? 2 : 0;
  a.pf_next = static_cast<const char*>(pf);
  a.pf_next_bytes = pf ? static_cast<int64_t>(pf_bytes) : 0;
  a.inject_wait = inject_wait;
  const std::vector<Block> blocks = launch_order(G, R, Keff);
  switch (BN) {
    case 16: return run<16>(maps, a, blocks, sms, budget, s);
    case 32: return run<32>(maps, a, blocks, sms, budget, s);
    default: return run<64>(maps, a, blocks, sms, budget, s);
  }
}

fq_status launch_decode_forward(const void* x, int M, int d_in, const void* T_in,
                                const fq_packed& Cq, const void* T_out_t, int d_out,
                                const float* gamma, void* y, char* ws, size_t ws_bytes,
                                int max_sms, const void* pf, size_t pf_bytes,
                                int64_t inject_wait, cudaStream_t s) {
  const DecGroupLayer L{x, d_in, T_in, Cq, T_out_t, d_out, gamma, y};
  return launch_decode_group(M, 1, &L, ws, ws_bytes, max_sms, false, pf, pf_bytes, inject_wait,
                             s);
}

fq_status launch_decode_core(int M, const fq_packed& Cq, const float* gamma, char* ws,
                             size_t ws_bytes, int max_sms, cudaStream_t s) {
  const DecGroupLayer L{nullptr, 0, nullptr, Cq, nullptr, 0, gamma, nullptr};
  return launch_decode_group(M, 1, &L, ws, ws_bytes, max_sms, true, nullptr, 0, 0, s);
}

size_t decode_core_z_offset() { return kWsHeader; }

size_t decode_core_u_offset(int M, int n_in) {
  return kWsHeader + round_up(static_cast<int64_t>(M) * n_in * 2, 256);
}

}  // namespace fq
