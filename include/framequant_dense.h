/*
 * libframequant, weight-reconstruction path: the quantized layer rebuilt as one dense bf16
 * weight for batches large enough that a single dense product beats the three frame products.
 *
 * Appendix K writes the quantized layer back in the original space as P_l D_hat P_prev^T,
 * i.e. W_hat = T_out^T C_hat T_in (d_out x d_in) with C_hat_ij = s_i q_ij + zero_i (times
 * gamma_i with the de-noising gain).  Then y = W_hat x costs 2 M d_out d_in FLOPs instead of
 * 2 M (n_in d_in + n_out n_in + d_out n_out) (about 3.3 times fewer at r = 1.1), after a
 * one-off reconstruction that costs one forward of d_in tokens.  The reconstructed weight
 * occupies 2 d_out d_in bytes, as an unquantized bf16 layer would.
 *
 * Conventions are those of framequant.h (device pointers, 16-byte alignment, asynchronous on
 * `stream`, validation before any launch, no allocation by the library).
 */
#ifndef FRAMEQUANT_DENSE_H_
#define FRAMEQUANT_DENSE_H_

#include "framequant.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Workspace bytes of fq_reconstruct_weight; 0 for invalid sizes.  It holds the tensor-core
 * chain's workspace for M = d_in tokens (z and u of the d_in unit vectors) and the d_in x d_out
 * output before its transpose: about 108 MB for a 4096 x 4096 layer at r = 1.1, 227 MB for
 * 11008 x 4096, 460 MB for 4096 x 11008, 432 MB for 8192 x 8192, 1.14 GB for 28672 x 8192 and
 * 2.8 GB for 8192 x 28672. */
size_t fq_reconstruct_workspace_bytes(int d_in, int n_in, int n_out, int d_out);

/* W_hat = T_out^T diag(gamma) C_hat T_in, bf16 d_out x d_in row-major: the FQ_BF16 forward of
 * fq_linear_forward applied to the d_in unit vectors (so z and u are rounded to bf16 as in the
 * forward), then transposed.  The analysis of unit vector e_j is column j of T_in, exact in
 * bf16, so it is taken as a transpose rather than a product; the code product and the synthesis
 * run on the tensor cores.
 *   T_in, C, T_out_t, gamma  as in fq_linear_forward
 *   W_hat  device bf16 d_out x d_in output
 *   ws     device workspace of fq_reconstruct_workspace_bytes(...) bytes, 256-byte aligned,
 *          zero-filled before its first use (it holds a fq_linear_forward workspace)
 * Errors: those of fq_linear_forward for M = d_in. */
fq_status fq_reconstruct_weight(const void* T_in, const fq_packed* C, const void* T_out_t,
                                int d_in, int d_out, const float* gamma, void* W_hat, void* ws,
                                size_t ws_bytes, fq_stream_t stream);

/* Workspace bytes of fq_dense_forward; 0 for invalid sizes. */
size_t fq_dense_workspace_bytes(int M, int d_in, int d_out);

/* y = x W_hat^T for M tokens (bf16 in and out, fp32 accumulation on the tensor cores): one
 * product of the tensor-core path (128 x 128 or 128 x 256 tiles, split K when tiles are few).
 *   x  device bf16 M x d_in;  W_hat  device bf16 d_out x d_in;  y  device bf16 M x d_out
 *   ws device workspace of fq_dense_workspace_bytes(M, d_in, d_out) bytes, 256-byte aligned,
 *      zero-filled before its first use
 * Requirements: M, d_in, d_out >= 1; d_in and d_out multiples of 8.
 * Errors: FQ_ERR_INVALID_ARG, FQ_ERR_ALIGNMENT, FQ_ERR_WORKSPACE, FQ_ERR_UNSUPPORTED (device
 * not compute capability 10.3), FQ_ERR_CUDA. */
fq_status fq_dense_forward(const void* x, int M, int d_in, const void* W_hat, int d_out, void* y,
                           void* ws, size_t ws_bytes, fq_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* FRAMEQUANT_DENSE_H_ */
