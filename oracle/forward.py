"""Oracle, part 4: the frame-quantized linear layer forward (plain fp64 CPU).

TEST INFRASTRUCTURE. Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline leg may
import this package; the product library never does, and shares no code with it.

Inference procedure (Sec. 3.2, Fig. "Inference for a FrameQuant quantized model"): the layer
input is taken to its fusion frame representation by the analysis operator (z = T_in x), the
quantized coefficients map it to the output's representation (u = C_hat z), and the synthesis
operator returns to the output space (y = T_out^T u).  The optional diagonal de-noising gain
scales u before synthesis (Appendix I, Z = F D_hat C_prev with F = P_l diag(gamma)).
"""
from __future__ import annotations

import numpy as np

from .quant import dequantize


def analysis(T_in: np.ndarray, X: np.ndarray) -> np.ndarray:
    """z = T_in x for every token: X (M x d_in) -> Z (M x n_in)  (Sec. 2.1, analysis operator)."""
    return X.astype(np.float64) @ T_in.T


def core(Z: np.ndarray, codes, scale, zero, gamma=None) -> np.ndarray:
    """u = gamma * (C_hat z) with C_hat = scale * q + zero row-wise: Z (M x n_in) -> U (M x n_out)
    (Sec. 3, the product D_hat C_prev)."""
    U = Z @ dequantize(codes, scale, zero).T
    if gamma is not None:
        U = U * gamma.astype(np.float64)[None, :]
    return U


def synthesis(T_out: np.ndarray, U: np.ndarray) -> np.ndarray:
    """y = T_out^T u for every token: U (M x n_out) -> Y (M x d_out)  (Sec. 2.1, synthesis
    operator, the adjoint of analysis)."""
    return U @ T_out


def layer_forward(X, T_in, codes, scale, zero, T_out, gamma=None) -> np.ndarray:
    """Y = T_out^T diag(gamma) C_hat T_in X^T, returned token-major (M x d_out)."""
    return synthesis(T_out, core(analysis(T_in, X), codes, scale, zero, gamma))


def round_bf16(A) -> np.ndarray:
    """Values of A (taken to fp32 first) rounded to the nearest bfloat16, ties to even, returned
    in fp64.  bfloat16 keeps the top 16 bits of an IEEE binary32: the 16 dropped bits decide
    the rounding, and a carry out of the mantissa moves the exponent (finite inputs)."""
    bits = np.asarray(A, dtype=np.float32).view(np.uint32).astype(np.uint64)
    keep_lsb = (bits >> 16) & 1
    rounded = ((bits + 0x7FFF + keep_lsb) >> 16) << 16
    return rounded.astype(np.uint32).view(np.float32).astype(np.float64)


def layer_forward_bf16_operands(X, T_in, codes, scale, zero, T_out, gamma=None) -> np.ndarray:
    """Diagnostic: layer_forward with T_in and T_out first rounded to bfloat16 (through fp32,
    as the bf16 path receives them), the rest of the arithmetic in fp64.  Its distance to
    layer_forward is the part of a bf16 result's error that the frame operands' precision
    alone causes."""
    return layer_forward(X, round_bf16(T_in), codes, scale, zero, round_bf16(T_out), gamma)
