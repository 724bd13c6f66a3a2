"""Oracle, part 2: frame coefficients and their 2-bit quantization (plain fp64 CPU).

TEST INFRASTRUCTURE. Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline leg may
import this package; the product library never does, and shares no code with it.

Sec. 3 (Eqs. for D_l) and Algorithm 1:
  * D_l = P_l^T Theta_l P_prev, i.e. C = T_out W T_in^T with T the analysis operators;
  * optional clipping of C to [mu - 2 sigma, mu + 2 sigma], sigma and mu over the whole matrix
    (Algorithm 1, steps 2-3);
  * per-row round-to-nearest quantization to 2 bits with a per-row fp16 scale and zero (the
    paper stores one scale and one offset per row, Appendix K).  The paper's own quantizer is
    GPTQ with calibration data (Algorithm 1, step 4); this oracle and the hot path it checks use
    round-to-nearest, as the workloads state.
  * optional diagonal de-noising gain (Sec. 3.1 (b), Appendix I: the paper reports that keeping
    only the diagonal of the Wiener filter already helps).
"""
from __future__ import annotations

import numpy as np


def coefficients(W: np.ndarray, T_in: np.ndarray, T_out: np.ndarray) -> np.ndarray:
    """C = T_out W T_in^T (n_out x n_in): the weight expressed between the two frames
    (Sec. 3, D_l = P_l^T Theta_l P_prev)."""
    return T_out @ W @ T_in.T


def clip_2sigma(C: np.ndarray) -> np.ndarray:
    """Clip to [mu - 2 sigma, mu + 2 sigma] with mu, sigma the mean and standard deviation of
    all entries (Algorithm 1, steps 2-3)."""
    mu, sigma = C.mean(), C.std()
    return np.clip(C, mu - 2.0 * sigma, mu + 2.0 * sigma)


def rtn(C: np.ndarray, bits: int = 2) -> tuple:
    """Per-row round-to-nearest.  For row i with minimum mn and maximum mx and L = 2^bits - 1:
    zero_i = fp16(mn), scale_i = fp16((mx - mn) / L) (1 when that is 0),
    q_ij = clamp(round_half_even((C_ij - zero_i) / scale_i), 0, L) with the fp16 values, and
    the dequantized coefficient is scale_i * q_ij + zero_i.
    Returns (codes uint8, scale float16, zero float16)."""
    L = (1 << bits) - 1
    mn = C.min(axis=1)
    mx = C.max(axis=1)
    zero = mn.astype(np.float16)
    scale = ((mx - mn) / L).astype(np.float16)
    if not np.all(np.isfinite(scale)) or not np.all(np.isfinite(zero)):
        raise OverflowError("row range exceeds float16")
    scale = np.where(scale == 0, np.float16(1.0), scale)
    s = scale.astype(np.float64)[:, None]
    z = zero.astype(np.float64)[:, None]
    q = np.clip(np.rint((C - z) / s), 0, L).astype(np.uint8)
    return q, scale, zero


def dequantize(codes: np.ndarray, scale: np.ndarray, zero: np.ndarray) -> np.ndarray:
    """C_hat = scale * q + zero, row-wise (fp64)."""
    return (scale.astype(np.float64)[:, None] * codes.astype(np.float64)
            + zero.astype(np.float64)[:, None])


def wiener_gain(C: np.ndarray, scale: np.ndarray) -> np.ndarray:
    """Diagonal de-noising gain per frame coefficient row: gamma_i = P_i / (P_i + scale_i^2/12),
    P_i the mean square of row i and scale_i^2/12 the variance of uniform rounding noise of step
    scale_i.  This is the scalar LMMSE (Wiener) shrinkage of each output coefficient under
    additive white quantization noise; the paper reports that the diagonal of the Wiener filter
    alone helps but prints no formula (Sec. 3.1 (b), Appendix I).  Pinned by brute force: the
    gain equals the Monte-Carlo minimiser of the mean squared error of gamma (c + n) against c
    for coefficients c of power P and uniform rounding noise n of step scale."""
    P = np.mean(C * C, axis=1)
    N = scale.astype(np.float64) ** 2 / 12.0
    return (P / (P + N)).astype(np.float32)
