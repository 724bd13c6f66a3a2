// Host-side declarations shared by the translation units of libframequant.
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

#include <vector>

#include "framequant.h"

namespace fq {

constexpr int kRowTile = 128;   // rows per packed tile and per MMA tile
constexpr int kColBlock = 64;   // columns per packed block and per K stage

inline int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }
inline int64_t round_up(int64_t a, int64_t b) { return ceil_div(a, b) * b; }

// Workspace header (64 KiB, at fixed offsets whatever the layer's sizes, so that one workspace
// can serve layers of different shapes): [0] device status word, [4] generation counter,
// [8] end-of-call ticket, [12] the activation-rounding maximum, [16..31] the first timeout's
// role, task, stage and detail words (cleared by each call), [32] the activation-rounding step,
// [kWsFlags] ready flags, kWsSlices per row tile of up to kWsMaxTiles
// row tiles per phase.  A zero-filled header is a valid initial state and every completed call
// leaves it valid for the next one.
constexpr size_t kWsHeader = 64 * 1024;
constexpr size_t kWsGen = 4;
constexpr size_t kWsDone = 8;
constexpr size_t kWsAmax = 12;    // activation rounding: max |z| of the call (float bits)
constexpr size_t kWsDelta = 32;   // activation rounding: the call's step Delta (float)
constexpr size_t kWsFlags = 1024;
constexpr int kWsSlices = 8;
constexpr int kWsMaxTiles = 640;
static_assert(kWsFlags + 3 * kWsMaxTiles * kWsSlices * 4 <= kWsHeader, "flags fit the header");
constexpr int kDecodeMaxM = 64;   // batches up to this size take the fused decode kernel

// ---- fq_api.cu
}  // namespace fq
extern "C" size_t fq_packed_words(int n_out, int n_in);
namespace fq {
// The checks every entry point makes on a packed descriptor: pointers set and 16-byte aligned,
// n_in and n_out positive multiples of 16, ld_words = 4 ceil(n_in / 64) (FQ_ERR_INVALID_ARG /
// FQ_ERR_ALIGNMENT), bits = 2 (FQ_ERR_UNSUPPORTED).
fq_status check_packed(const fq_packed* C);

// ---- fq_pack.cu
// Dense frame operand (rows x cols bf16, row-major, cols % 8 == 0) -> out: ceil(rows/128) x
// ceil(cols/64) pre-swizzled 16 KiB tiles (row tile major, zero padded), then the block-sparse
// index {0, KB, t * KB} of each row tile at frame_tiles_index_offset().
size_t frame_tiles_index_offset(int rows, int cols);
cudaError_t launch_frame_tile(const void* T, int rows, int cols, void* out, cudaStream_t s);
cudaError_t launch_pack(const uint8_t* codes, const uint16_t* scale, const uint16_t* zero,
                        int n_out, int n_in, uint32_t* words, int32_t* status, cudaStream_t s);

// ---- fq_debug.cu: fp32 path
size_t debug_workspace_bytes(int M, int n_in, int n_out);
cudaError_t launch_debug_forward(const float* x, int M, int d_in, const float* T_in,
                                 const fq_packed& C, const float* T_out_t, int d_out,
                                 const float* gamma, float* y, char* ws, cudaStream_t s);

// ---- fq_decode.cu: bf16 path for small batches (one fused persistent kernel)
size_t decode_workspace_bytes(int M, int d_in, int n_in, int n_out, int d_out);
// max_sms > 0 caps the SMs a call's kernels occupy (the grid and the plan); pf/pf_bytes is an
// optional device range (16-byte aligned, multiple of 16 bytes) to warm in L2 during the
// synthesis when this layer's T_out^T is itself warmed during the code product; inject_wait > 0
// is the timeout test hook of fq_forward_opts (requires max_sms == 1)
fq_status launch_decode_forward(const void* x, int M, int d_in, const void* T_in,
                                const fq_packed& C, const void* T_out_t, int d_out,
                                const float* gamma, void* y, char* ws, size_t ws_bytes,
                                int max_sms, const void* pf, size_t pf_bytes,
                                int64_t inject_wait, cudaStream_t s);

// A block-sparse frame operand (frames in structured form): for every 128-row tile of the
// operand, the K blocks [idx[3t], idx[3t+1]) it has non-zero entries in, stored from tile
// idx[3t+2] of `tiles` on as contiguous 16 KiB tiles already in the 128-byte-swizzled shared
// memory image; `count` stored tiles in all.
struct SparseOperand {
  const uint8_t* tiles;
  const int32_t* idx;
  int count;
};

// One layer of a fused launch over independent layers (the M <= 64 kernel).  With tin.tiles
// (tout.tiles) set, the analysis (synthesis) reads that block-sparse operand instead of T_in
// (T_out_t).
struct DecGroupLayer {
  const void* x;
  int d_in;
  const void* T_in;
  fq_packed C;
  const void* T_out_t;
  int d_out;
  const float* gamma;
  void* y;
  SparseOperand tin{};
  SparseOperand tout{};
};
// Workspace of a launch over G layers (header, then z and u of each layer); 0 for G out of range.
size_t decode_group_workspace_bytes(int M, int G, const DecGroupLayer* layers);
// The fused kernel over G <= 4 independent layers; arguments checked by the caller.
fq_status launch_decode_group(int M, int G, const DecGroupLayer* layers, char* ws,
                              size_t ws_bytes, int max_sms, bool core_only, const void* pf,
                              size_t pf_bytes, int64_t inject_wait, cudaStream_t s);

// The code product alone (z already in the workspace at decode_core_z_offset(), u left at
// decode_core_u_offset()), for the structured-frame forward.
fq_status launch_decode_core(int M, const fq_packed& C, const float* gamma, char* ws,
                             size_t ws_bytes, int max_sms, cudaStream_t s);
size_t decode_core_z_offset();
size_t decode_core_u_offset(int M, int n_in);

// ---- fq_prep.cu: Q of the Householder QR of the a x a row-major G, columns signed so that R
// has a positive diagonal (row-major output)
void haar_q(const double* G, int a, std::vector<double>& Q);

// ---- fq_tc.cu: bf16 tensor-core path
// act_bits > 0: the analysis output is rounded to act_bits-bit integers with one step per call
// (Appendix F) before the code product
size_t tc_workspace_bytes(int M, int d_in, int n_in, int n_out, int d_out, int act_bits);
fq_status launch_tc_forward(const void* x, int M, int d_in, const void* T_in,
                            const fq_packed& C, const void* T_out_t, int d_out,
                            const float* gamma, void* y, char* ws, size_t ws_bytes,
                            int max_sms, int act_bits, cudaStream_t s);
// The same chain for the d_in unit vectors as tokens (M = d_in; y is d_in x d_out, row t the
// forward of e_t), with the analysis product replaced by its exact result: z[t] = column t of
// T_in (a transpose) and sum_j z[t][j] (column sums).  Workspace: tc_workspace_bytes(d_in, ...).
fq_status launch_tc_unit_forward(const void* T_in, int d_in, const fq_packed& C,
                                 const void* T_out_t, int d_out, const float* gamma, void* y,
                                 char* ws, size_t ws_bytes, cudaStream_t s);

}  // namespace fq
