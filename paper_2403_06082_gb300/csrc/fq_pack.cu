// fq_pack: 2-bit codes (uint8, row-major) -> the tiled packed layout of framequant.h, with a
// check of the per-row scale and zero the descriptor will carry.
// Memory-bound: one thread writes one 16-byte group of 4 words (64 codes of one row).
// fq_frame_tile (below): a dense frame operand -> pre-swizzled contiguous tiles.
#include <algorithm>

#include "fq_device.cuh"
#include "fq_internal.h"

namespace fq {
namespace {

// an fp16 bit pattern with the exponent field all ones is an infinity or a NaN
__device__ __forceinline__ bool f16_nonfinite(uint16_t h) { return (h & 0x7C00u) == 0x7C00u; }

__global__ void __launch_bounds__(256) pack_kernel(const uint8_t* __restrict__ codes,
                                                   const uint16_t* __restrict__ scale,
                                                   const uint16_t* __restrict__ zero, int n_out,
                                                   int n_in, int KB, int64_t groups,
                                                   uint4* __restrict__ out,
                                                   int32_t* __restrict__ status) {
  const int64_t g = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (g >= groups) return;
  // group g = ((tile * KB + kb) * 128 + r): 4 words for row tile*128+r, columns kb*64 .. +63
  const int r = static_cast<int>(g % kRowTile);
  const int64_t tk = g / kRowTile;
  const int kb = static_cast<int>(tk % KB);
  const int tile = static_cast<int>(tk / KB);
  const int row = tile * kRowTile + r;
  uint32_t w[4] = {0u, 0u, 0u, 0u};
  bool bad = false;
  if (row < n_out) {
    // the row's scale and zero, once per row (by its first column block)
    if (kb == 0) bad |= f16_nonfinite(scale[row]) || f16_nonfinite(zero[row]);
    const uint8_t* src = codes + static_cast<int64_t>(row) * n_in;
    const int c0 = kb * kColBlock;
#pragma unroll
    for (int c = 0; c < kColBlock; ++c) {
      const int col = c0 + c;
      uint32_t q = 0;
      if (col < n_in) {
        q = src[col];
        bad |= q > 3u;
      }
      const int cc = c & 15;
      w[c >> 4] |= (q & 3u) << (2 * (cc >> 1) + 16 * (cc & 1));
    }
  }
  if (bad) report(status, FQ_ERR_DEVICE_CHECK);
  out[g] = make_uint4(w[0], w[1], w[2], w[3]);
}

}  // namespace

cudaError_t launch_pack(const uint8_t* codes, const uint16_t* scale, const uint16_t* zero,
                        int n_out, int n_in, uint32_t* words, int32_t* status, cudaStream_t s) {
  const int KB = static_cast<int>(ceil_div(n_in, kColBlock));
  const int64_t groups = ceil_div(n_out, kRowTile) * kRowTile * KB;
  const int threads = 256;
  const int64_t blocks = ceil_div(groups, threads);
  pack_kernel<<<static_cast<unsigned>(blocks), threads, 0, s>>>(
      codes, scale, zero, n_out, n_in, KB, groups, reinterpret_cast<uint4*>(words), status);
  return cudaGetLastError();
}

}  // namespace fq

// ------------------------------------------------------------------------------------------
// fq_frame_tile: a dense bf16 frame operand (rows x cols, row-major) -> contiguous pre-swizzled
// 128 x 64 tiles, the layout the M <= 64 kernel's weight copies read whole (one 16 KiB bulk
// copy per K block instead of a 2-D box of 128 rows of 128 bytes).  Memory-bound: one thread
// moves one 16-byte chunk (8 elements of one row).
namespace fq {
namespace {

constexpr int kTileRows = 128, kTileCols = 64;

__global__ void __launch_bounds__(256) frame_tile_kernel(const uint4* __restrict__ T, int rows,
                                                         int cols, int KB, int64_t chunks,
                                                         uint4* __restrict__ tiles,
                                                         int32_t* __restrict__ idx, int RT) {
  const int64_t g = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (g < 3ll * RT) {
    // row tile t reads K blocks 0 .. KB-1 from tile t * KB on (the block-sparse index form)
    const int t = static_cast<int>(g / 3), f = static_cast<int>(g % 3);
    idx[g] = f == 0 ? 0 : (f == 1 ? KB : t * KB);
  }
  if (g >= chunks) return;
  // chunk g of the output = (tile t, K block kb, row r, stored position h); it holds the
  // row's 16-byte group c = h ^ (r & 7) (128-byte swizzle within each 8-row group)
  const int h = static_cast<int>(g & 7);
  const int r = static_cast<int>((g >> 3) % kTileRows);
  const int64_t tk = g / (8 * kTileRows);
  const int kb = static_cast<int>(tk % KB);
  const int t = static_cast<int>(tk / KB);
  const int row = t * kTileRows + r;
  const int c = h ^ (r & 7);
  const int col = kb * kTileCols + c * 8;
  uint4 v = make_uint4(0u, 0u, 0u, 0u);
  if (row < rows && col < cols) v = __ldg(T + (static_cast<int64_t>(row) * cols + col) / 8);
  tiles[g] = v;
}

}  // namespace

size_t frame_tiles_index_offset(int rows, int cols) {
  return static_cast<size_t>(ceil_div(rows, kTileRows) * ceil_div(cols, kTileCols)) *
         (kTileRows * kTileCols * 2);
}

cudaError_t launch_frame_tile(const void* T, int rows, int cols, void* out, cudaStream_t s) {
  const int RT = static_cast<int>(ceil_div(rows, kTileRows));
  const int KB = static_cast<int>(ceil_div(cols, kTileCols));
  const int64_t chunks = static_cast<int64_t>(RT) * KB * kTileRows * 8;
  auto* tiles = static_cast<uint4*>(out);
  auto* idx = reinterpret_cast<int32_t*>(static_cast<char*>(out) +
                                         frame_tiles_index_offset(rows, cols));
  const int threads = 256;
  const int64_t blocks = ceil_div(std::max<int64_t>(chunks, 3ll * RT), threads);
  frame_tile_kernel<<<static_cast<unsigned>(blocks), threads, 0, s>>>(
      static_cast<const uint4*>(T), rows, cols, KB, chunks, tiles, idx, RT);
  return cudaGetLastError();
}

}  // namespace fq
