"""Oracle, part 6: the frame-domain quantizer of Algorithm 1, step 4 (plain fp64 CPU).

TEST INFRASTRUCTURE. Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline leg may
import this package; the product library never does, and shares no code with it.

Algorithm 1 quantizes D_l = P_l^T Theta_l P_prev (quant.coefficients: C = T_out W T_in^T)
while keeping the proxy loss of Sec. 3 small:
    L(D_hat) = ||D C_prev - D_hat C_prev||_F^2 = tr((D - D_hat) H (D - D_hat)^T),
    H = C_prev C_prev^T,  C_prev = P_prev^T A_prev = T_in A_prev
(the frame representation of calibration tokens, one token per column).
Step 4 is the iterative Hessian-based method the paper cites (GPTQ), with the 2-sigma clip of
steps 2-3 applied first.  Restated:
  * each row's quantization grid is fixed before the iteration: the per-row fp16 scale and zero
    of quant.rtn, from the (clipped) row's range;
  * columns are quantized in order; after column j is rounded to its grid, the rounding error
    of each row is spread over that row's columns j+1.. so that the proxy loss is minimal given
    the columns already fixed (the optimal-brain-surgeon update, which needs the inverse of H
    restricted to the columns not yet fixed);
  * those restricted inverses come from one upper Cholesky factor U of H^-1 (H^-1 = U^T U):
    the update after column j is  w_k -= (w_j - q_j) / U_jj * U_jk  for k > j;
  * columns go in blocks of B; inside a block the update is applied column by column, to later
    blocks once per block.  In exact arithmetic the result does not depend on B;
  * H is damped by `damp` times its mean diagonal before inversion (the cited method's
    stabilisation; the paper does not state a value, 0.01 is the cited method's default).
"""
from __future__ import annotations

import numpy as np

from . import quant


def hessian(C_prev: np.ndarray) -> np.ndarray:
    """H = C_prev C_prev^T (n_in x n_in) from the frame representation of the calibration
    tokens (one token per column of C_prev)."""
    C_prev = np.asarray(C_prev, dtype=np.float64)
    return C_prev @ C_prev.T


def damped(H: np.ndarray, damp: float = 0.01) -> np.ndarray:
    """H + damp * mean(diag H) * I."""
    H = np.array(H, dtype=np.float64)
    H[np.diag_indices_from(H)] += damp * float(np.mean(np.diag(H)))
    return H


def proxy_loss(D: np.ndarray, D_hat: np.ndarray, H: np.ndarray) -> float:
    """tr((D - D_hat) H (D - D_hat)^T), the loss Algorithm 1 minimises (Sec. 3)."""
    E = np.asarray(D, dtype=np.float64) - np.asarray(D_hat, dtype=np.float64)
    return float(np.einsum("ij,jk,ik->", E, H, E))


def gptq(D: np.ndarray, H: np.ndarray, bits: int = 2, block: int = 128,
         damp: float = 0.01) -> tuple:
    """Quantize D (n_out x n_in) against the Hessian H (n_in x n_in) on the per-row RTN grid.
    Returns (codes uint8, scale float16, zero float16), the format of quant.rtn."""
    W = np.array(D, dtype=np.float64)
    n_out, n_in = W.shape
    levels = (1 << bits) - 1
    _, scale, zero = quant.rtn(W, bits)                  # the grid, fixed from the rows' ranges
    s = scale.astype(np.float64)
    z = zero.astype(np.float64)
    U = np.linalg.cholesky(np.linalg.inv(damped(H, damp))).T     # H^-1 = U^T U, U upper
    codes = np.zeros((n_out, n_in), dtype=np.uint8)
    for b0 in range(0, n_in, block):
        b1 = min(b0 + block, n_in)
        spread = np.zeros((n_out, b1 - b0))
        for j in range(b0, b1):
            q = np.clip(np.rint((W[:, j] - z) / s), 0, levels)
            codes[:, j] = q.astype(np.uint8)
            e = (W[:, j] - (s * q + z)) / U[j, j]
            W[:, j + 1:b1] -= np.outer(e, U[j, j + 1:b1])
            spread[:, j - b0] = e
        W[:, b1:] -= spread @ U[b0:b1, b1:]
    return codes, scale, zero


def quantize_layer(C: np.ndarray, C_prev: np.ndarray, clip: bool = True, bits: int = 2,
                   block: int = 128, damp: float = 0.01) -> tuple:
    """Algorithm 1, steps 2-4: the 2-sigma clip (quant.clip_2sigma) and the frame-domain GPTQ
    of C against H = C_prev C_prev^T.  Returns (codes, scale, zero)."""
    D = quant.clip_2sigma(C) if clip else np.asarray(C, dtype=np.float64)
    return gptq(D, hessian(C_prev), bits, block, damp)
