/*
 * libframequant: forward pass of a frame-quantized linear layer (FrameQuant, Adepu et al.,
 * ICML 2024, arXiv 2403.06082) on one NVIDIA GB300 GPU (sm_103a).
 *
 * The layer (Sec. 3.2, the inference procedure; Sec. 3, D_l = P_l^T Theta_l P_prev):
 *
 *     z = T_in x                          analysis onto the input tight fusion frame
 *     u_i = gamma_i (s_i sum_j q_ij z_j + zero_i sum_j z_j)
 *                                         2-bit frame coefficients C_hat_ij = s_i q_ij + zero_i
 *     y = T_out^T u                       synthesis from the output frame
 *
 * for every token x (a row of X, M x d_in).  T_in (n_in x d_in) is the analysis operator of
 * the input frame, P_prev^T in the paper; T_out^T (d_out x n_out) is the synthesis operator of
 * the output frame, P_l in the paper.  n = k * rho is the number of frame coefficients; r = n/d
 * is the redundancy.  gamma is the optional diagonal de-noising gain (Sec. 3.1 (b),
 * Appendix I); pass NULL for none.
 *
 * Conventions for every entry point:
 *   - All tensor pointers are DEVICE pointers owned by the caller, row-major, 16-byte aligned.
 *     The library allocates no device memory; scratch space is the caller's workspace `ws`.
 *   - Work is enqueued on `stream` (a cudaStream_t; NULL is the legacy default stream) and is
 *     asynchronous: a return of FQ_OK means every check passed and every kernel launched.
 *   - Arguments are validated on the host before anything is launched; on any error the call
 *     returns a status and launches nothing.  No entry point aborts the process.
 *   - Device-side findings (code values out of range, a bounded wait that ran out) set bit
 *     (1 << status) of an int32 status word: fq_pack's `status` argument, or the head of
 *     fq_linear_forward's `ws`.  fq_check reads it back.
 *   - Outputs must not alias inputs; concurrent calls must not share a workspace.
 */
#ifndef FRAMEQUANT_H_
#define FRAMEQUANT_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* fq_stream_t; /* same type as cudaStream_t */

typedef enum {
  FQ_OK = 0,
  FQ_ERR_INVALID_ARG = 1,   /* null pointer, non-positive or inconsistent dimension, bad mode */
  FQ_ERR_ALIGNMENT = 2,     /* a pointer is not 16-byte aligned or a row pitch not 16 bytes */
  FQ_ERR_UNSUPPORTED = 3,   /* valid request this build cannot run (device not sm_103, sizes) */
  FQ_ERR_WORKSPACE = 4,     /* ws is NULL or smaller than fq_workspace_bytes() */
  FQ_ERR_CUDA = 5,          /* a CUDA runtime or launch error */
  FQ_ERR_TIMEOUT = 6,       /* device: a bounded wait inside a kernel ran out (fq_check) */
  FQ_ERR_DEVICE_CHECK = 7   /* device: fq_pack met a code above 3 or a non-finite scale or
                               zero (fq_check) */
} fq_status;

/* Arithmetic modes of fq_linear_forward. */
enum {
  FQ_BF16 = 0,        /* x, T_in, T_out^T, y are bf16; z and u are rounded to bf16 between the
                         three products; every product accumulates in fp32 (tensor cores) */
  FQ_FP32_DEBUG = 1   /* x, T_in, T_out^T, y, z, u are fp32 throughout (CUDA cores) */
};

/* FQ_BF16 | FQ_ACT_BITS(N), 2 <= N <= 8: round the frame representation of the activations to
 * N-bit integers before the code product (Appendix F: the INT8 form for N = 8).  With
 * Delta = max |z| / (2^(N-1) - 1) over every token and coefficient of the call (z = T_in x in
 * fp32) and zbar = nearest integer to z / Delta (ties to even), the layer computes
 *     u_i = Delta gamma_i (s_i sum_j q_ij zbar_j + zero_i sum_j zbar_j),   y = T_out^T u.
 * zbar is held exactly in bf16 and sum_j q_ij zbar_j is exact in the tensor cores' fp32
 * accumulator, so the product is the integer one.  The whole analysis must finish before any
 * rounding, so every batch size runs the tensor-core path's chain of kernels (an analysis that
 * writes fp32 z and the maximum, a rounding kernel, the code product, the synthesis). */
#define FQ_ACT_BITS(n) ((n) << 8)

/* Packed 2-bit frame coefficients with their per-row scale and zero (the paper keeps one scale
 * and one offset per row next to the 2-bit codes, Appendix K).  Code q_ij in {0,1,2,3}
 * dequantizes to s_i q_ij + zero_i.  fq_pack fills this descriptor; it is the one unit every
 * forward entry point takes.
 *
 * Layout of `words` (uint32; written by fq_pack): rows are grouped in tiles of 128 and
 * columns in blocks of 64; n_out and n_in are padded up to those multiples with code 0.  The
 * 64 codes of one (row, column block) are 4 consecutive words, and the 512 words of one
 * (row tile, column block) pair are contiguous:
 *     word index = ((row/128) * KB + col/64) * 512 + (row%128) * 4 + (col%64)/16,
 *     KB = ceil(n_in/64);
 * inside a word, column c = col%16 occupies bits [2*(c/2) + 16*(c%2), +2): even columns in the
 * low half-word, odd columns in the high half-word, so that one mask of 0x00030003 shifted by
 * 2*(c/2) isolates the adjacent pair (c, c+1).  ld_words = 4 * KB is the number of words that
 * hold one row (spread over its KB column blocks); a row tile spans 128 * ld_words contiguous
 * words, and the whole buffer ceil(n_out/128) * 128 * ld_words = fq_packed_words(n_out, n_in).
 */
typedef struct {
  const uint32_t* words;      /* device, fq_packed_words(n_out, n_in) words, 16-byte aligned */
  const uint16_t* scale_f16;  /* device, IEEE fp16 bit patterns, n_out entries, 16-byte aligned */
  const uint16_t* zero_f16;   /* device, IEEE fp16 bit patterns, n_out entries, 16-byte aligned */
  int32_t n_out;              /* rows of C_hat, = k_out * rho, a multiple of 16 */
  int32_t n_in;               /* columns of C_hat, = k_in * rho, a multiple of 16 */
  int32_t ld_words;           /* words per row of codes, 4 * ceil(n_in / 64) */
  int32_t bits;               /* bits per code; 2 is the only width this library runs */
} fq_packed;

/* Number of uint32 words of the packed layout above: ceil(n_out/128)*128 * ceil(n_in/64)*64 / 16.
 * Returns 0 when n_out or n_in is not positive. */
size_t fq_packed_words(int n_out, int n_in);

/* Pack 2-bit codes with their per-row scale and zero into one descriptor (Algorithm 1, step 5,
 * which stores the quantized D_hat; layout above).
 *   codes      device uint8, n_out x n_in row-major, values 0..3 (any alignment)
 *   scale_f16  device fp16 bit patterns [n_out], 16-byte aligned: the step s_i of row i
 *   zero_f16   device fp16 bit patterns [n_out], 16-byte aligned: the offset zero_i of row i
 *   out        host descriptor.  On input out->words must point to a writable device buffer of
 *              fq_packed_words(n_out, n_in) uint32 words, 16-byte aligned (caller-owned); fq_pack
 *              writes the packed codes there (padding positions with code 0) and sets every
 *              other field: scale_f16 and zero_f16 point at the caller's arrays (not copied, so
 *              they must outlive the descriptor's use), n_out, n_in, ld_words and bits = 2.
 *   status     device int32 or NULL: bit (1 << FQ_ERR_DEVICE_CHECK) is set there when a code
 *              above 3 is met (its low 2 bits are packed) or a scale or zero is not finite;
 *              fq_pack never clears it.  Read it with fq_check.
 * Any positive n_out and n_in can be packed; the forward entry points take multiples of 16.
 * Errors (nothing is launched and *out is left unchanged): FQ_ERR_INVALID_ARG (null codes,
 * scale, zero, out or out->words; n_out or n_in <= 0), FQ_ERR_ALIGNMENT, FQ_ERR_CUDA. */
fq_status fq_pack(const uint8_t* codes, const uint16_t* scale_f16, const uint16_t* zero_f16,
                  int n_out, int n_in, fq_packed* out, int32_t* status, fq_stream_t stream);

/* Bytes of workspace fq_linear_forward needs for these sizes and mode (independent of the
 * device).  Returns 0 for invalid sizes. */
size_t fq_workspace_bytes(int M, int d_in, int n_in, int n_out, int d_out, int mode);

/* Forward pass of the frame-quantized linear layer (Sec. 3.2; see the top of this file).
 *   x        device, M x d_in tokens (bf16 or fp32 by mode)
 *   T_in     device, n_in x d_in analysis operator of the input frame (P_prev^T)
 *   C        host pointer to a descriptor of device data (codes, scale, zero); C->n_in and
 *            C->n_out give the frame sizes
 *   T_out_t  device, d_out x n_out synthesis operator of the output frame (T_out^T = P_l),
 *            i.e. the output frame's analysis operator T_out (n_out x d_out) transposed, so that
 *            the synthesis contracts over the contiguous dimension of both of its operands, as
 *            the analysis and the code product do
 *   gamma    device fp32 [n_out] de-noising gain, or NULL for none
 *   y        device, M x d_out output (bf16 or fp32 by mode)
 *   ws       device workspace of at least fq_workspace_bytes(M, d_in, n_in, n_out, d_out,
 *            mode) bytes, 256-byte aligned, ZERO-FILLED BEFORE ITS FIRST USE.  Its first 64 KiB
 *            are a header at fixed offsets (status word, a call generation counter and
 *            ready flags per slice of a 128-row output tile) that every completed call leaves
 *            ready for the next, so a workspace can be reused across calls and layer shapes
 *            without being cleared again; zero it again after a call reported
 *            FQ_ERR_TIMEOUT.  Its first 4
 *            bytes are the device status word, which each call clears before reporting.
 *   mode     FQ_BF16 or FQ_FP32_DEBUG, or FQ_BF16 | FQ_ACT_BITS(N)
 * Requirements: M, d_in, d_out >= 1; d_in and d_out multiples of 8; C->n_in and C->n_out
 * positive multiples of 16, C->ld_words = 4 * ceil(C->n_in / 64) and C->bits = 2 (as fq_pack
 * sets them); all device pointers 16-byte aligned.
 * Errors: FQ_ERR_INVALID_ARG (also an ld_words that does not match n_in), FQ_ERR_ALIGNMENT,
 * FQ_ERR_WORKSPACE, FQ_ERR_UNSUPPORTED (C->bits other than 2; the current device is not
 * compute capability 10.3 in FQ_BF16 mode; M <= 64 in FQ_BF16 mode with n_in, n_out or d_out
 * above 81920 = 640 tiles of 128 rows), FQ_ERR_CUDA. */
fq_status fq_linear_forward(const void* x, int M, int d_in, const void* T_in,
                            const fq_packed* C, const void* T_out_t, int d_out,
                            const float* gamma, void* y, void* ws, size_t ws_bytes, int mode,
                            fq_stream_t stream);

/* fq_linear_forward on at most max_sms SMs (0: all of them), so that independent layers
 * (q, k and v of an attention block, or gate and up of an MLP, which read the same input) can
 * run side by side on different streams, each with its own workspace.  The grid and the plan
 * of the FQ_BF16 kernels are sized for the budget (one CTA per SM); FQ_FP32_DEBUG ignores it.
 * For M <= 64 the CTAs of one call wait on one another's partial results, so every CTA of the
 * call must be resident at once.  Such a call takes clusters of CTAs in proportion to its
 * budget's share of the SM count (a GPC holds a whole number of clusters), so that calls whose
 * budgets add up to no more than the device's SM count are resident together.  Calls whose
 * budgets overcommit the device, or that share it with other work holding SMs, can stall one
 * another until a bounded wait runs out (FQ_ERR_TIMEOUT through fq_check).
 * Errors: those of fq_linear_forward, and FQ_ERR_INVALID_ARG for max_sms < 0.  This entry
 * point has no counterpart in the paper. */
fq_status fq_linear_forward_sms(const void* x, int M, int d_in, const void* T_in,
                                const fq_packed* C, const void* T_out_t, int d_out,
                                const float* gamma, void* y, void* ws, size_t ws_bytes, int mode,
                                int max_sms, fq_stream_t stream);

/* Options of fq_linear_forward_ex. */
typedef struct {
  int32_t max_sms;             /* 0: the whole device; otherwise the SM budget of
                                  fq_linear_forward_sms */
  const void* l2_prefetch;     /* device range to bring into L2 while this call runs, or NULL */
  size_t l2_prefetch_bytes;    /* its length; rounded down to a multiple of 16 */
  int64_t inject_timeout_cycles; /* 0 in normal use.  A test hook for the device-error path:
                                  when > 0 (FQ_BF16, M <= 64 and max_sms = 1 only, i.e. one
                                  CTA with no cluster peers) the kernel's first wait for
                                  another phase's output expects a stamp that no call writes
                                  and gives up after this many SM clock cycles, so the call
                                  ends with FQ_ERR_TIMEOUT in the workspace status word (and
                                  the waiting role, task, stage and detail in the next four
                                  words) instead of a result, without a fault.  Zero the
                                  workspace again before its next use. */
} fq_forward_opts;

/* fq_linear_forward with options (opts NULL: none).  The L2 prefetch is a hint for chaining
 * layers, typically the next layer's T_in: the M <= 64 kernel issues it when this layer's own
 * T_out^T is small enough to be warmed in L2 during the code product, so that its synthesis
 * leaves HBM idle; each CTA then prefetches its share of the range when it reaches its first
 * synthesis task.  Other calls ignore it.  Results never depend on it.  This entry point has
 * no counterpart in the paper.
 * Errors: those of fq_linear_forward; FQ_ERR_INVALID_ARG for max_sms < 0, a NULL range of
 * nonzero length, or inject_timeout_cycles < 0 or set outside its one-CTA decode case;
 * FQ_ERR_ALIGNMENT for a range start that is not 16-byte aligned. */
fq_status fq_linear_forward_ex(const void* x, int M, int d_in, const void* T_in,
                               const fq_packed* C, const void* T_out_t, int d_out,
                               const float* gamma, void* y, void* ws, size_t ws_bytes, int mode,
                               const fq_forward_opts* opts, fq_stream_t stream);

/* One layer of fq_linear_forward_group: the arguments of fq_linear_forward for that layer. */
typedef struct {
  const void* x;           /* device bf16, M x d_in tokens */
  int32_t d_in;
  const void* T_in;        /* device bf16, n_in x d_in */
  const fq_packed* C;      /* host pointer to the layer's packed descriptor */
  const void* T_out_t;     /* device bf16, d_out x n_out */
  int32_t d_out;
  const float* gamma;      /* device fp32 [n_out] or NULL */
  void* y;                 /* device bf16, M x d_out output */
  /* Optional tiled copies of the frame operands, written by fq_frame_tile from this layer's
   * T_in (rows n_in, cols d_in) and T_out_t (rows d_out, cols n_out), or NULL.  For M <= 64
   * the fused launch reads a tiled operand instead of its row-major matrix, one contiguous
   * 16 KiB copy per 128 x 64 block (the same values, so the same result); batches above 64
   * read T_in and T_out_t, which stay required.  16-byte aligned. */
  const void* T_in_tiles;
  const void* T_out_tiles;
} fq_layer;

/* Most layers one fq_linear_forward_group call takes. */
#define FQ_MAX_GROUP 4

/* Bytes of workspace fq_linear_forward_group needs for these layers at M tokens (FQ_BF16);
 * 0 for invalid sizes or counts.  It is at least fq_workspace_bytes of each layer, so the
 * workspace also serves the layers' single calls. */
size_t fq_group_workspace_bytes(int M, int n_layers, const fq_layer* layers);

/* The FQ_BF16 forward of up to FQ_MAX_GROUP independent layers in one call: q, k and v of an
 * attention block, or gate and up of an MLP, which read the same input and whose outputs no
 * layer of the group reads.  Each layer's result is that of fq_linear_forward on its own
 * arguments.  For M <= 64 the layers run in one fused launch whose task lists interleave the
 * layers' phases (analysis, code product, synthesis), so that the point where one layer's
 * next phase waits for all of its previous phase falls while another layer streams its
 * weights; larger batches, which are tensor-bound, run the layers one after another.
 *   layers   host array of n_layers descriptors (1 <= n_layers <= FQ_MAX_GROUP); the layers may
 *            differ in every size; x may be shared; no y may equal another layer's x or y
 *   ws       device workspace of fq_group_workspace_bytes(M, n_layers, layers) bytes, with the
 *            rules of fq_linear_forward (256-byte aligned, zero-filled before its first use,
 *            reusable, zeroed again after FQ_ERR_TIMEOUT; status word at its head)
 *   opts     as in fq_linear_forward_ex (NULL: none); inject_timeout_cycles must be 0
 * Requirements and errors: those of fq_linear_forward for each layer; FQ_ERR_INVALID_ARG for a
 * bad count or an output that is another layer's input or output; FQ_ERR_UNSUPPORTED when the
 * layers' ready flags do not fit the workspace header (more than 2016 row tiles of 128 over
 * the layers' analyses and code products).  This entry point has no counterpart in the
 * paper. */
fq_status fq_linear_forward_group(int M, int n_layers, const fq_layer* layers, void* ws,
                                  size_t ws_bytes, const fq_forward_opts* opts,
                                  fq_stream_t stream);

/* Bytes of the tiled copy of a rows x cols frame operand (fq_frame_tile): ceil(rows/128) x
 * ceil(cols/64) tiles of 16 KiB, then a row-tile index of 12 bytes per row tile rounded up to
 * 256; 0 for non-positive sizes or cols not a multiple of 8. */
size_t fq_frame_tiles_bytes(int rows, int cols);

/* Tiled copy of a dense frame operand for fq_layer's T_in_tiles / T_out_tiles: the bf16
 * rows x cols row-major T (T_in, or T_out_t) as 128 x 64 blocks, row-block major then column
 * block, each block 128 rows of 128 bytes with the 16-byte groups of row r stored in the
 * order g ^ (r mod 8) (the 128-byte swizzle the tensor-core operand expects), zero padded
 * past rows and cols.  A layout of the same values, not a change of the operator (the frame
 * of Sec. 2.2 as T_in and T_out_t hold it).  Runs on the stream; T is read, out written.
 * Errors: FQ_ERR_INVALID_ARG for NULL pointers, non-positive sizes or out overlapping T;
 * FQ_ERR_ALIGNMENT for cols % 8 != 0 or a pointer not 16-byte aligned; FQ_ERR_WORKSPACE when
 * out_bytes < fq_frame_tiles_bytes(rows, cols); FQ_ERR_CUDA for a launch failure. */
fq_status fq_frame_tile(const void* T, int rows, int cols, void* out, size_t out_bytes,
                        fq_stream_t stream);

/* ------------------------------------------------------------------------------------------
 * Offline preparation of a layer (not on the inference path).  These produce the inputs of
 * fq_linear_forward on the device from a weight matrix W and the frame parameters.
 * ---------------------------------------------------------------------------------------- */

/* Random rotation R = Pi (Q_a kron Q_b) D of R^d, d = a * b (Sec. 2.2 remarks; Appendix K,
 * P_l = R_l T_l).  The raw random numbers are the caller's (HOST pointers): Q_a and Q_b are the
 * orthogonal factors of the QR decompositions of the a x a and b x b Gaussian matrices
 * gauss_a and gauss_b, with columns signed so that R has a positive diagonal; D = diag(signs);
 * (Pi v)[i] = v[perm[i]]. */
typedef struct {
  int32_t a;
  int32_t b;
  const double* gauss_a;   /* host, a x a row-major */
  const double* gauss_b;   /* host, b x b row-major */
  const int64_t* perm;     /* host, a permutation of 0 .. d-1 */
  const double* signs;     /* host, d entries, each +1 or -1 */
} fq_rotation;

/* Workspace bytes of fq_frame_build (a = b = 0 without rotation). */
size_t fq_frame_workspace_bytes(int k, int rho, int d, int a, int b);

/* Analysis operator of the real (k, rho, d) tight fusion frame (Sec. 2.2 Definition "Tight
 * Fusion Frames"; construction of Appendix J): spectral tetris gives F (rho/2 x d/2, unit
 * columns, orthogonal rows); row j of F modulated by (w^(k_i n))_n, w = exp(2 pi i / k), spans
 * subspace k_i of C^(d/2); each modulated vector is divided by sqrt(k) (Parseval, T^T T = I);
 * the entrywise map x + iy -> [[x, -y], [y, x]] makes it real.  Rows are ordered (row j of F,
 * k_i, real/imaginary part), columns (2c, 2c+1) are complex coordinate c.  With rot != NULL the
 * operator is T R^T.  (1, d, d) gives the identity (the trivial frame).
 *   T    device fp32 output, (k*rho) x d row-major
 *   ws   device workspace of fq_frame_workspace_bytes(k, rho, d, a, b) bytes
 * Synchronizes `stream` before returning (host staging buffers are released on return).
 * Errors: FQ_ERR_INVALID_ARG (invalid triple: rho and d even, d >= 2 rho, and k at least the
 * width of each row of F; bad rotation), FQ_ERR_WORKSPACE, FQ_ERR_CUDA. */
fq_status fq_frame_build(int k, int rho, int d, const fq_rotation* rot, float* T, void* ws,
                         size_t ws_bytes, fq_stream_t stream);

/* Workspace bytes of fq_coefficients. */
size_t fq_coefficients_workspace_bytes(int d_out, int n_in);

/* Frame coefficients C = T_out W T_in^T (Sec. 3: D_l = P_l^T Theta_l P_prev), fp32 on CUDA
 * cores.  W is d_out x d_in, T_in n_in x d_in, T_out n_out x d_out (analysis operators), C is
 * n_out x n_in; all device fp32 row-major. */
fq_status fq_coefficients(const float* W, int d_out, int d_in, const float* T_in, int n_in,
                          const float* T_out, int n_out, float* C, void* ws, size_t ws_bytes,
                          fq_stream_t stream);

/* Per-row 2-bit round-to-nearest of C (n_out x n_in, device fp32): zero_i = fp16(min_j C_ij),
 * scale_i = fp16((max_j C_ij - min_j C_ij) / 3) (1 when that is 0),
 * q_ij = clamp(rint((C_ij - zero_i) / scale_i), 0, 3) with the fp16 values (Algorithm 1 with
 * round-to-nearest in place of step 4).  gamma (nullable) receives the diagonal de-noising
 * gain P_i / (P_i + scale_i^2 / 12), P_i the mean square of row i (Sec. 3.1 (b), Appendix I).
 *   codes  device uint8 n_out x n_in;  scale, zero  device fp16 bits [n_out] */
fq_status fq_quantize_rtn(const float* C, int n_out, int n_in, uint8_t* codes, uint16_t* scale,
                          uint16_t* zero, float* gamma, fq_stream_t stream);

/* H = Z^T Z (n_in x n_in, fp64): the Hessian of Algorithm 1's proxy loss,
 * ||D C_prev - D_hat C_prev||_F^2 = tr((D - D_hat) H (D - D_hat)^T) with H = C_prev C_prev^T
 * (Sec. 3), from Z = C_prev^T, the frame representations T_in a of N calibration tokens a (one
 * token per row, N x n_in, fp64).  Device pointers, 8-byte aligned; fp64 CUDA-core product.
 * Errors: FQ_ERR_INVALID_ARG, FQ_ERR_ALIGNMENT, FQ_ERR_CUDA. */
fq_status fq_gptq_hessian(const double* Z, int N, int n_in, double* H, fq_stream_t stream);

/* Workspace bytes of fq_quantize_gptq: 8 (n_out n_in + 2 n_in^2 + 130 n_out) + n_out n_in
 * bytes and a few KB (about 0.83 GB for 12112 x 4512); 0 for invalid sizes. */
size_t fq_gptq_workspace_bytes(int n_out, int n_in);

/* 2-bit codes of C (n_out x n_in, fp64 frame coefficients) by the frame-domain quantizer of
 * Algorithm 1, steps 2-4, in fp64 on the GPU:
 *   - clip != 0: C is clipped to [mu - 2 sigma, mu + 2 sigma], mu and sigma over all of C;
 *   - every row's grid is fixed from the (clipped) row before the iteration, as in
 *     fq_quantize_rtn: zero = fp16(min), scale = fp16((max - min) / 3) (1 when 0); gamma
 *     (nullable) receives the de-noising gain P / (P + scale^2 / 12) of the clipped rows;
 *   - the Hessian H (n_in x n_in, e.g. from fq_gptq_hessian) is damped by damp mean(diag H)
 *     (0.01 is the usual value) and factored as H^-1 = U^T U, U upper triangular;
 *   - the columns are rounded in order, in blocks of 128; after column j each row's rounding
 *     error divided by U_jj is spread over its later columns in proportion to row j of U (the
 *     optimal-brain-surgeon update of the method GPTQ, which Algorithm 1 cites).
 *   codes  device uint8 n_out x n_in;  scale, zero  device fp16 bits [n_out];  gamma fp32 or NULL
 *   ws     device workspace of fq_gptq_workspace_bytes(n_out, n_in) bytes, 256-byte aligned
 * Synchronizes `stream` before returning.  n_in up to 25600 (the triangular inverse keeps one
 * column in shared memory).
 * Errors: FQ_ERR_INVALID_ARG, FQ_ERR_ALIGNMENT, FQ_ERR_WORKSPACE, FQ_ERR_UNSUPPORTED (n_in above
 * 25600), FQ_ERR_DEVICE_CHECK (the damped H is not positive definite), FQ_ERR_CUDA. */
fq_status fq_quantize_gptq(const double* C, int n_out, int n_in, const double* H, double damp,
                           int clip, uint8_t* codes, uint16_t* scale, uint16_t* zero,
                           float* gamma, void* ws, size_t ws_bytes, fq_stream_t stream);

/* ------------------------------------------------------------------------------------------
 * Frames in structured form (the paper's own deployment form: Sec. 2.2 and Appendix J build T
 * from rho/2 disjoint runs of a spectral-tetris frame, each modulated by k roots of unity;
 * Appendix K applies a random rotation).  With d a multiple of rho, run j of the un-rotated
 * frame covers complex coordinates c = j w .. (j+1) w - 1, w = d / rho (real coordinates 2c and
 * 2c + 1), and its k frame vectors are the realified rows of the k x w block
 * exp(2 pi i k_i c / k) / sqrt(k).  So T = T_u R^T with T_u block-diagonal, and
 *     z = T x = T_u (R^T x),        y = T^T u = R (T_u^T u),
 * which needs the rotation factors and k roots of unity instead of the n x d operator: a few
 * hundred KB per side instead of 2 n d bytes.
 * ---------------------------------------------------------------------------------------- */

/* A frame prepared by fq_frame_implicit: device arrays inside the caller's buffer.
 * The un-rotated operator T_u is block-diagonal; it is kept in both orientations as
 * block-sparse tile lists: for every 128-row tile of T_u (n x d, the analysis operand) or of
 * T_u^T (d x n, the synthesis operand), the 64-column blocks that meet the tile's runs, each a
 * contiguous 16 KiB bf16 tile laid out as the tensor cores read it from shared memory. */
typedef struct {
  int32_t k, rho, d;       /* (k, rho, d): rho even, d a multiple of rho, k >= d / rho */
  int32_t a, b;            /* rotation R = Pi (Q_a kron Q_b) D with a * b = d; 0, 0: R = I */
  const float* Qa;         /* device a x a row-major, and its transpose QaT */
  const float* QaT;
  const float* Qb;         /* device b x b row-major, and its transpose QbT */
  const float* QbT;
  const int32_t* perm;     /* device d: (Pi v)[i] = v[perm[i]] */
  const int32_t* iperm;    /* device d: the inverse permutation */
  const float* signs;      /* device d, the diagonal of D */
  const uint8_t* ana_tiles; /* device: the analysis operand's tiles (ana_count x 16 KiB) */
  const int32_t* ana_idx;  /* device [ceil(n/128)][3]: first K block, end K block, first tile */
  int32_t ana_count;
  const uint8_t* syn_tiles; /* device: the synthesis operand's tiles (syn_count x 16 KiB) */
  const int32_t* syn_idx;  /* device [ceil(d/128)][3], as ana_idx */
  int32_t syn_count;
} fq_frame;

/* Bytes of the device buffer fq_frame_implicit fills (a = b = 0 without rotation); 0 for an
 * invalid triple. */
size_t fq_frame_implicit_bytes(int k, int rho, int d, int a, int b);

/* Prepare the structured form of the (k, rho, d) frame with rotation `rot` (NULL: none), the
 * same frame fq_frame_build writes out densely.  Q_a and Q_b are computed on the host in double
 * precision (Householder QR, columns signed as in fq_rotation) and stored as fp32; the tiles of
 * T_u are computed on the host in double precision and stored as bf16 (rounded through fp32,
 * like the dense operator).
 *   buf    device buffer of fq_frame_implicit_bytes(k, rho, d, rot->a, rot->b) bytes, 256-byte
 *          aligned; it must outlive every use of *out (about 11 MB for (282, 16, 4096), 75 MB
 *          for (757, 16, 11008))
 *   out    host struct receiving the sizes and the device pointers into buf
 * Synchronizes `stream` before returning.
 * Errors: FQ_ERR_INVALID_ARG (rho odd, d not a multiple of rho, k < d / rho, a bad rotation),
 *         FQ_ERR_WORKSPACE (buf NULL or too small), FQ_ERR_ALIGNMENT, FQ_ERR_CUDA. */
fq_status fq_frame_implicit(int k, int rho, int d, const fq_rotation* rot, void* buf,
                            size_t bytes, fq_frame* out, fq_stream_t stream);

/* Bytes of workspace fq_linear_forward_implicit needs; 0 for invalid sizes. */
size_t fq_implicit_workspace_bytes(int M, int d_in, int n_in, int n_out, int d_out);

/* The layer forward of fq_linear_forward (Sec. 3.2) with T_in and T_out given in structured
 * form: v = R_in^T x, then the fused decode kernel of fq_linear_forward with block-sparse frame
 * operands (z = T_u,in v, the 2-bit code product, s = T_u,out^T u, all on the tensor cores; the
 * analysis and synthesis read only the tiles of each row tile's runs), then y = R_out s.  bf16
 * tokens in and out; the rotations are computed in fp32 on CUDA cores and v, z, u and s are
 * rounded to bf16.
 *   x      device bf16, M x F_in->d tokens;  y  device bf16, M x F_out->d
 *   F_in, F_out  host pointers to prepared frames; C->n_in = F_in->k * F_in->rho and
 *          C->n_out = F_out->k * F_out->rho
 *   gamma  device fp32 [C->n_out] or NULL
 *   ws     device workspace of fq_implicit_workspace_bytes(...) bytes, 256-byte aligned and
 *          zero-filled before its first use (the header rules of fq_linear_forward)
 *   max_sms  as in fq_linear_forward_sms (0: the whole device)
 * Requirements: 1 <= M <= 64; for each frame at most 640 row tiles of 128 per orientation and,
 * with a rotation, b <= 1024 and (d + 8 (a + b) + 8 g r + B) * 4 bytes of shared memory at
 * most 227 KiB, with d rounded up to a multiple of 4, r = b rounded up to a multiple of 32,
 * g = max(1, min(4, 1024 / r)), and B = b * b when b <= 128 and that total stays within
 * 110 KiB, else 64 b; sizes and alignment as in fq_linear_forward.
 * Errors: FQ_ERR_INVALID_ARG, FQ_ERR_ALIGNMENT, FQ_ERR_WORKSPACE, FQ_ERR_UNSUPPORTED (M > 64, a
 * frame above those limits, device not compute capability 10.3), FQ_ERR_CUDA. */
fq_status fq_linear_forward_implicit(const void* x, int M, const fq_frame* F_in,
                                     const fq_packed* C, const fq_frame* F_out,
                                     const float* gamma, void* y, void* ws, size_t ws_bytes,
                                     int max_sms, fq_stream_t stream);

/* One layer of fq_linear_forward_implicit_group: the arguments of fq_linear_forward_implicit
 * for that layer. */
typedef struct {
  const void* x;            /* device bf16, M x F_in->d */
  const fq_frame* F_in;     /* host pointers to prepared frames */
  const fq_packed* C;
  const fq_frame* F_out;
  const float* gamma;       /* device fp32 [C->n_out] or NULL */
  void* y;                  /* device bf16, M x F_out->d */
} fq_implicit_layer;

/* Workspace bytes of fq_linear_forward_implicit_group (0 for invalid sizes or counts). */
size_t fq_implicit_group_workspace_bytes(int M, int n_layers, const fq_implicit_layer* layers);

/* fq_linear_forward_implicit for up to FQ_MAX_GROUP independent layers: each layer's input
 * rotation, then one fused launch over all the layers (as fq_linear_forward_group does with
 * dense operators), then each layer's output rotation.  Requirements and errors: those of
 * fq_linear_forward_implicit for each layer, and those of fq_linear_forward_group for the
 * group (no y may be another layer's x or y).  This entry point has no counterpart in the
 * paper. */
fq_status fq_linear_forward_implicit_group(int M, int n_layers, const fq_implicit_layer* layers,
                                           void* ws, size_t ws_bytes, int max_sms,
                                           fq_stream_t stream);

/* ------------------------------------------------------------------------------------------
 * Forward pass without a caller-provided workspace.  The paper has no counterpart: this is a
 * convenience of the library for callers that cannot allocate device memory.
 * ---------------------------------------------------------------------------------------- */

/* Bytes of the library's own device scratch array used by fq_linear_forward_static. */
#define FQ_STATIC_SCRATCH_BYTES (16u << 20)

/* fq_linear_forward without `ws`: for callers that cannot allocate device memory (a host
 * framework that owns every allocation, a plugin interface that passes only inputs and
 * outputs, a C program without an allocator).  The scratch space is a __device__ array of
 * FQ_STATIC_SCRATCH_BYTES inside this library, reserved on every GPU that loads it until the
 * process exits; this call allocates nothing.
 *   - Requests whose fq_workspace_bytes(M, d_in, C->n_in, C->n_out, d_out, mode) exceeds
 *     FQ_STATIC_SCRATCH_BYTES return FQ_ERR_UNSUPPORTED and launch nothing.
 *   - Every call looks up the array's device address for the current device.  The first call
 *     on a device, and the first after a device reset, loads the library's device code there:
 *     make it before any stream capture.
 *   - All calls share the array and it keeps the last call's contents: calls whose work may
 *     overlap on the GPU (other streams, other host threads) race on it.
 *   - The device status word is the head of the array: read it with fq_static_check.
 * Other arguments, requirements and errors are those of fq_linear_forward. */
fq_status fq_linear_forward_static(const void* x, int M, int d_in, const void* T_in,
                                   const fq_packed* C, const void* T_out_t, int d_out,
                                   const float* gamma, void* y, int mode, fq_stream_t stream);

/* Synchronize `stream` and return the device status of the last fq_linear_forward_static call
 * on the current device (as fq_check does for a workspace).  When it is FQ_ERR_TIMEOUT, the
 * header of the library's scratch array is also cleared (on `stream`, synchronized before
 * returning), which a workspace's owner would do by zeroing it, so that later static calls run
 * again.  Allocates nothing.  Returns FQ_OK, FQ_ERR_TIMEOUT or FQ_ERR_CUDA. */
fq_status fq_static_check(fq_stream_t stream);

/* Synchronize `stream` and read the device status word at `status_word` (the head of a
 * forward workspace, or the `status` given to fq_pack).  Returns FQ_OK, FQ_ERR_TIMEOUT,
 * FQ_ERR_DEVICE_CHECK, or FQ_ERR_CUDA if the synchronization itself failed. */
fq_status fq_check(const void* status_word, fq_stream_t stream);

/* Static string naming a status. */
const char* fq_status_str(fq_status status);

#ifdef __cplusplus
}
#endif

#endif /* FRAMEQUANT_H_ */
