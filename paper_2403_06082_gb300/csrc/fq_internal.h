// Host-side declarations shared by the translation units of libframequant.
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

#include "framequant.h"

namespace fq {

constexpr int kRowTile = 128;   // rows per packed tile and per MMA tile
constexpr int kColBlock = 64;   // columns per packed block and per K stage

inline int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }
inline int64_t round_up(int64_t a, int64_t b) { return ceil_div(a, b) * b; }

// Workspace header: [0, 4) status word, [4, 256) reserved; counters follow.
constexpr size_t kWsHeader = 256;

// ---- fq_api.cu
}  // namespace fq
extern "C" size_t fq_packed_words(int n_out, int n_in);
namespace fq {

// ---- fq_pack.cu
cudaError_t launch_pack(const uint8_t* codes, int n_out, int n_in, uint32_t* words,
                        int32_t* status, cudaStream_t s);

// ---- fq_debug.cu: fp32 path
size_t debug_workspace_bytes(int M, int n_in, int n_out);
cudaError_t launch_debug_forward(const float* x, int M, int d_in, const float* T_in,
                                 const fq_packed& C, const float* T_out_t, int d_out,
                                 const float* gamma, float* y, char* ws, cudaStream_t s);

// ---- fq_tc.cu: bf16 tensor-core path
size_t tc_workspace_bytes(int M, int d_in, int n_in, int n_out, int d_out);
fq_status launch_tc_forward(const void* x, int M, int d_in, const void* T_in,
                            const fq_packed& C, const void* T_out_t, int d_out,
                            const float* gamma, void* y, char* ws, size_t ws_bytes,
                            cudaStream_t s);

}  // namespace fq
