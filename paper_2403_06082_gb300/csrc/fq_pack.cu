// fq_pack: 2-bit codes (uint8, row-major) -> the tiled packed layout of framequant.h, with a
// check of the per-row scale and zero the descriptor will carry.
// Memory-bound: one thread writes one 16-byte group of 4 words (64 codes of one row).
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
