// C ABI of libframequant (declared in include/framequant.h): argument checks on the host, then
// dispatch to the bf16 tensor-core path (fq_tc.cu) or the fp32 debug path (fq_debug.cu).
#include <cuda_runtime.h>

#include <algorithm>

#include "fq_internal.h"

using namespace fq;

namespace {

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

fq_status cuda_status(cudaError_t e) { return e == cudaSuccess ? FQ_OK : FQ_ERR_CUDA; }

// mode = FQ_BF16 or FQ_FP32_DEBUG, optionally | FQ_ACT_BITS(N) with FQ_BF16 and 2 <= N <= 8
bool split_mode(int mode, int& base, int& act) {
  base = mode & 0xFF;
  act = (mode >> 8) & 0xFF;
  if ((mode & ~0xFFFF) != 0) return false;
  if (base != FQ_BF16 && base != FQ_FP32_DEBUG) return false;
  if (act != 0 && (base != FQ_BF16 || act < 2 || act > 8)) return false;
  return true;
}

// Compute capability of the current device, or -1.
int current_cc() {
  int dev = 0, major = 0, minor = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return -1;
  if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess)
    return -1;
  return major * 10 + minor;
}

}  // namespace

namespace fq {

fq_status check_packed(const fq_packed* C) {
  if (!C || !C->words || !C->scale_f16 || !C->zero_f16) return FQ_ERR_INVALID_ARG;
  if (C->n_in <= 0 || C->n_out <= 0) return FQ_ERR_INVALID_ARG;
  if (C->n_in % 16 || C->n_out % 16) return FQ_ERR_ALIGNMENT;
  if (C->ld_words != 4 * ceil_div(C->n_in, kColBlock)) return FQ_ERR_INVALID_ARG;
  if (C->bits != 2) return FQ_ERR_UNSUPPORTED;
  if (!aligned16(C->words) || !aligned16(C->scale_f16) || !aligned16(C->zero_f16))
    return FQ_ERR_ALIGNMENT;
  return FQ_OK;
}

}  // namespace fq

extern "C" {

size_t fq_packed_words(int n_out, int n_in) {
  if (n_out <= 0 || n_in <= 0) return 0;
  return static_cast<size_t>(round_up(n_out, kRowTile)) * round_up(n_in, kColBlock) / 16;
}

fq_status fq_pack(const uint8_t* codes, const uint16_t* scale_f16, const uint16_t* zero_f16,
                  int n_out, int n_in, fq_packed* out, int32_t* status, fq_stream_t stream) {
  if (!codes || !scale_f16 || !zero_f16 || !out || !out->words || n_out <= 0 || n_in <= 0)
    return FQ_ERR_INVALID_ARG;
  if (!aligned16(out->words) || !aligned16(scale_f16) || !aligned16(zero_f16))
    return FQ_ERR_ALIGNMENT;
  // the caller's buffer, writable by contract (the descriptor's view of it is const)
  uint32_t* words = const_cast<uint32_t*>(out->words);
  const cudaError_t e = launch_pack(codes, scale_f16, zero_f16, n_out, n_in, words, status,
                                    reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return FQ_ERR_CUDA;
  out->scale_f16 = scale_f16;
  out->zero_f16 = zero_f16;
  out->n_out = n_out;
  out->n_in = n_in;
  out->ld_words = static_cast<int32_t>(4 * ceil_div(n_in, kColBlock));
  out->bits = 2;
  return FQ_OK;
}

size_t fq_frame_tiles_bytes(int rows, int cols) {
  if (rows <= 0 || cols <= 0 || cols % 8 != 0) return 0;
  return frame_tiles_index_offset(rows, cols) +
         static_cast<size_t>(round_up(ceil_div(rows, kRowTile) * 12, 256));
}

fq_status fq_frame_tile(const void* T, int rows, int cols, void* out, size_t out_bytes,
                        fq_stream_t stream) {
  if (!T || !out || rows <= 0 || cols <= 0) return FQ_ERR_INVALID_ARG;
  if (cols % 8 != 0 || !aligned16(T) || !aligned16(out)) return FQ_ERR_ALIGNMENT;
  if (out_bytes < fq_frame_tiles_bytes(rows, cols)) return FQ_ERR_WORKSPACE;
  if (static_cast<const char*>(out) < static_cast<const char*>(T) +
          static_cast<size_t>(rows) * cols * 2 &&
      static_cast<const char*>(T) < static_cast<const char*>(out) + out_bytes)
    return FQ_ERR_INVALID_ARG;   // the copy may not overlap its source
  return launch_frame_tile(T, rows, cols, out, reinterpret_cast<cudaStream_t>(stream)) ==
                 cudaSuccess
             ? FQ_OK
             : FQ_ERR_CUDA;
}

size_t fq_workspace_bytes(int M, int d_in, int n_in, int n_out, int d_out, int mode) {
  if (M <= 0 || d_in <= 0 || n_in <= 0 || n_out <= 0 || d_out <= 0) return 0;
  int base = 0, act = 0;
  if (!split_mode(mode, base, act)) return 0;
  if (base == FQ_BF16) {
    if (act > 0) return tc_workspace_bytes(M, d_in, n_in, n_out, d_out, act);
    return M <= kDecodeMaxM ? decode_workspace_bytes(M, d_in, n_in, n_out, d_out)
                            : tc_workspace_bytes(M, d_in, n_in, n_out, d_out, 0);
  }
  return debug_workspace_bytes(M, n_in, n_out);
}

}  // extern "C"

namespace {

// The host-side checks of one layer forward, before anything is launched.
fq_status check_layer(const void* x, int M, int d_in, const void* T_in, const fq_packed* C,
                      const void* T_out_t, int d_out, const float* gamma, const void* y,
                      int mode) {
  if (!x || !T_in || !C || !T_out_t || !y) return FQ_ERR_INVALID_ARG;
  int base = 0, act = 0;
  if (!split_mode(mode, base, act)) return FQ_ERR_INVALID_ARG;
  if (M <= 0 || d_in <= 0 || d_out <= 0) return FQ_ERR_INVALID_ARG;
  if (const fq_status cs = check_packed(C)) return cs;
  if (d_in % 8 || d_out % 8) return FQ_ERR_ALIGNMENT;
  if (!aligned16(x) || !aligned16(T_in) || !aligned16(T_out_t) || !aligned16(y) ||
      (gamma && !aligned16(gamma)))
    return FQ_ERR_ALIGNMENT;
  return FQ_OK;
}

fq_status check_opts(const fq_forward_opts* opts, int& max_sms, const void*& pf,
                     size_t& pf_bytes, int64_t& inject) {
  max_sms = opts ? opts->max_sms : 0;
  pf = opts ? opts->l2_prefetch : nullptr;
  pf_bytes = opts ? (opts->l2_prefetch_bytes & ~static_cast<size_t>(15)) : 0;
  inject = opts ? opts->inject_timeout_cycles : 0;
  if (max_sms < 0 || (pf_bytes > 0 && !pf) || inject < 0) return FQ_ERR_INVALID_ARG;
  if (pf_bytes > 0 && !aligned16(pf)) return FQ_ERR_ALIGNMENT;
  return FQ_OK;
}

fq_status check_ws(const void* ws, size_t ws_bytes, size_t need) {
  if (!ws) return FQ_ERR_WORKSPACE;
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return FQ_ERR_ALIGNMENT;
  if (ws_bytes < need) return FQ_ERR_WORKSPACE;
  return FQ_OK;
}

// The group's layers as the decode kernel takes them.
bool group_layers(int n, const fq_layer* layers, DecGroupLayer* out) {
  for (int l = 0; l < n; ++l) {
    const fq_layer& L = layers[l];
    if (!L.C) return false;
    out[l] = DecGroupLayer{L.x, L.d_in, L.T_in, *L.C, L.T_out_t, L.d_out, L.gamma, L.y};
    // tiled copies of the frame operands (fq_frame_tile), read whole tiles at a time
    auto tiled = [](const void* p, int rows, int cols) {
      if (!p) return SparseOperand{};
      const auto* b = static_cast<const uint8_t*>(p);
      const int64_t RT = ceil_div(rows, kRowTile), KB = ceil_div(cols, kColBlock);
      return SparseOperand{b, reinterpret_cast<const int32_t*>(
                                  b + frame_tiles_index_offset(rows, cols)),
                           static_cast<int>(RT * KB)};
    };
    out[l].tin = tiled(L.T_in_tiles, L.C->n_in, L.d_in);
    out[l].tout = tiled(L.T_out_tiles, L.d_out, L.C->n_out);
  }
  return true;
}

}  // namespace

extern "C" {

fq_status fq_linear_forward_ex(const void* x, int M, int d_in, const void* T_in,
                               const fq_packed* C, const void* T_out_t, int d_out,
                               const float* gamma, void* y, void* ws, size_t ws_bytes, int mode,
                               const fq_forward_opts* opts, fq_stream_t stream) {
  int max_sms = 0;
  const void* pf = nullptr;
  size_t pf_bytes = 0;
  int64_t inject = 0;
  if (const fq_status os = check_opts(opts, max_sms, pf, pf_bytes, inject)) return os;
  if (inject > 0 && (mode != FQ_BF16 || M <= 0 || M > kDecodeMaxM || max_sms != 1))
    return FQ_ERR_INVALID_ARG;
  int base = 0, act = 0;
  if (!split_mode(mode, base, act)) return FQ_ERR_INVALID_ARG;
  if (const fq_status ls = check_layer(x, M, d_in, T_in, C, T_out_t, d_out, gamma, y, mode))
    return ls;
  const size_t need = fq_workspace_bytes(M, d_in, C->n_in, C->n_out, d_out, mode);
  if (const fq_status ws_st = check_ws(ws, ws_bytes, need)) return ws_st;
  auto s = reinterpret_cast<cudaStream_t>(stream);
  if (base == FQ_FP32_DEBUG) {
    if (cudaMemsetAsync(ws, 0, kWsHeader, s) != cudaSuccess) return FQ_ERR_CUDA;
    return cuda_status(launch_debug_forward(
        static_cast<const float*>(x), M, d_in, static_cast<const float*>(T_in), *C,
        static_cast<const float*>(T_out_t), d_out, gamma, static_cast<float*>(y),
        static_cast<char*>(ws), s));
  }
  if (current_cc() != 103) return FQ_ERR_UNSUPPORTED;
  // the status word is cleared by the forward's first kernel, in stream order; rounding the
  // activations needs the whole analysis before the code product, which the tensor-core
  // path's chain of three kernels has at any batch size
  if (M <= kDecodeMaxM && act == 0)
    return launch_decode_forward(x, M, d_in, T_in, *C, T_out_t, d_out, gamma, y,
                                 static_cast<char*>(ws), ws_bytes, max_sms, pf, pf_bytes, inject,
                                 s);
  return launch_tc_forward(x, M, d_in, T_in, *C, T_out_t, d_out, gamma, y,
                           static_cast<char*>(ws), ws_bytes, max_sms, act, s);
}

size_t fq_group_workspace_bytes(int M, int n_layers, const fq_layer* layers) {
  if (M <= 0 || n_layers < 1 || n_layers > FQ_MAX_GROUP || !layers) return 0;
  size_t need = 0;
  for (int l = 0; l < n_layers; ++l) {
    const fq_layer& L = layers[l];
    if (!L.C) return 0;
    const size_t one = fq_workspace_bytes(M, L.d_in, L.C->n_in, L.C->n_out, L.d_out, FQ_BF16);
    if (one == 0) return 0;
    need = std::max(need, one);
  }
  if (M <= kDecodeMaxM) {
    DecGroupLayer g[FQ_MAX_GROUP];
    if (!group_layers(n_layers, layers, g)) return 0;
    need = std::max(need, decode_group_workspace_bytes(M, n_layers, g));
  }
  return need;
}

fq_status fq_linear_forward_group(int M, int n_layers, const fq_layer* layers, void* ws,
                                  size_t ws_bytes, const fq_forward_opts* opts,
                                  fq_stream_t stream) {
  int max_sms = 0;
  const void* pf = nullptr;
  size_t pf_bytes = 0;
  int64_t inject = 0;
  if (const fq_status os = check_opts(opts, max_sms, pf, pf_bytes, inject)) return os;
  if (inject != 0 || !layers || n_layers < 1 || n_layers > FQ_MAX_GROUP)
    return FQ_ERR_INVALID_ARG;
  for (int l = 0; l < n_layers; ++l) {
    const fq_layer& L = layers[l];
    if (const fq_status ls = check_layer(L.x, M, L.d_in, L.T_in, L.C, L.T_out_t, L.d_out,
                                         L.gamma, L.y, FQ_BF16))
      return ls;
    // independent layers: no output is another layer's input or output
    for (int j = 0; j < n_layers; ++j)
      if (j != l && (layers[j].y == L.y || layers[j].x == L.y)) return FQ_ERR_INVALID_ARG;
    if (L.x == L.y) return FQ_ERR_INVALID_ARG;
    if (!aligned16(L.T_in_tiles) || !aligned16(L.T_out_tiles)) return FQ_ERR_ALIGNMENT;
  }
  const size_t need = fq_group_workspace_bytes(M, n_layers, layers);
  if (need == 0) return FQ_ERR_INVALID_ARG;
  if (const fq_status ws_st = check_ws(ws, ws_bytes, need)) return ws_st;
  if (current_cc() != 103) return FQ_ERR_UNSUPPORTED;
  auto s = reinterpret_cast<cudaStream_t>(stream);
  if (M <= kDecodeMaxM) {
    DecGroupLayer g[FQ_MAX_GROUP];
    group_layers(n_layers, layers, g);
    return launch_decode_group(M, n_layers, g, static_cast<char*>(ws), ws_bytes, max_sms, false,
                               pf, pf_bytes, 0, s);
  }
  // larger batches are tensor-bound: the layers run one after another on the tensor-core path
  for (int l = 0; l < n_layers; ++l) {
    const fq_layer& L = layers[l];
    if (const fq_status st = launch_tc_forward(L.x, M, L.d_in, L.T_in, *L.C, L.T_out_t, L.d_out,
                                               L.gamma, L.y, static_cast<char*>(ws), ws_bytes,
                                               max_sms, 0, s))
      return st;
  }
  return FQ_OK;
}

fq_status fq_linear_forward_sms(const void* x, int M, int d_in, const void* T_in,
                                const fq_packed* C, const void* T_out_t, int d_out,
                                const float* gamma, void* y, void* ws, size_t ws_bytes, int mode,
                                int max_sms, fq_stream_t stream) {
  const fq_forward_opts o{max_sms, nullptr, 0, 0};
  return fq_linear_forward_ex(x, M, d_in, T_in, C, T_out_t, d_out, gamma, y, ws, ws_bytes, mode,
                              &o, stream);
}

fq_status fq_linear_forward(const void* x, int M, int d_in, const void* T_in,
                            const fq_packed* C, const void* T_out_t, int d_out,
                            const float* gamma, void* y, void* ws, size_t ws_bytes, int mode,
                            fq_stream_t stream) {
  return fq_linear_forward_ex(x, M, d_in, T_in, C, T_out_t, d_out, gamma, y, ws, ws_bytes, mode,
                              nullptr, stream);
}

fq_status fq_check(const void* status_word, fq_stream_t stream) {
  if (!status_word) return FQ_ERR_INVALID_ARG;
  auto s = reinterpret_cast<cudaStream_t>(stream);
  int32_t v = 0;
  if (cudaStreamSynchronize(s) != cudaSuccess) return FQ_ERR_CUDA;
  if (cudaMemcpy(&v, status_word, sizeof(v), cudaMemcpyDeviceToHost) != cudaSuccess)
    return FQ_ERR_CUDA;
  if (v & (1 << FQ_ERR_TIMEOUT)) return FQ_ERR_TIMEOUT;
  if (v & (1 << FQ_ERR_DEVICE_CHECK)) return FQ_ERR_DEVICE_CHECK;
  return FQ_OK;
}

const char* fq_status_str(fq_status st) {
  switch (st) {
    case FQ_OK: return "FQ_OK";
    case FQ_ERR_INVALID_ARG: return "FQ_ERR_INVALID_ARG";
    case FQ_ERR_ALIGNMENT: return "FQ_ERR_ALIGNMENT";
    case FQ_ERR_UNSUPPORTED: return "FQ_ERR_UNSUPPORTED";
    case FQ_ERR_WORKSPACE: return "FQ_ERR_WORKSPACE";
    case FQ_ERR_CUDA: return "FQ_ERR_CUDA";
    case FQ_ERR_TIMEOUT: return "FQ_ERR_TIMEOUT";
    case FQ_ERR_DEVICE_CHECK: return "FQ_ERR_DEVICE_CHECK";
  }
  return "FQ_UNKNOWN";
}

}  // extern "C"
