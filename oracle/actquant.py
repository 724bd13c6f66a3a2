"""Oracle, part 7: rounding the frame representation of the activations (plain fp64 CPU).

TEST INFRASTRUCTURE. Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline leg may
import this package; the product library never does, and shares no code with it.

Appendix F quantizes the activations in the fusion-frame domain: the layer's input is first
taken to its frame representation C_prev = P_prev^T A_prev (here z = T_in x for every token),
then rounded to N-bit integers with one step for the whole tensor,
    Delta = max |C_prev| / (2^(N-1) - 1),      C_bar = nearest integer to C_prev / Delta,
so that C_bar holds integers in [-(2^(N-1) - 1), 2^(N-1) - 1] (the INT8 form for N = 8) and
Delta * C_bar stands in for C_prev in the rest of the layer.  Readings where the appendix is
silent: the maximum and the step are taken over every token and coefficient of one call;
ties round to even; an all-zero tensor has Delta = 0 and C_bar = 0.
"""
from __future__ import annotations

import numpy as np

from .forward import analysis, core, synthesis


def levels(bits: int) -> int:
    """Largest integer magnitude of the N-bit symmetric grid, 2^(N-1) - 1."""
    if bits < 2:
        raise ValueError("at least 2 bits")
    return (1 << (bits - 1)) - 1


def quantize_ff(Z: np.ndarray, bits: int) -> tuple:
    """(C_bar as int64, Delta) for the frame representation Z (Appendix F, per tensor)."""
    Z = np.asarray(Z, dtype=np.float64)
    L = levels(bits)
    amax = float(np.max(np.abs(Z))) if Z.size else 0.0
    if amax == 0.0:
        return np.zeros(Z.shape, dtype=np.int64), 0.0
    delta = amax / L
    Zbar = np.clip(np.rint(Z / delta), -L, L).astype(np.int64)
    return Zbar, delta


def layer_forward_actquant(X, T_in, codes, scale, zero, T_out, gamma, bits: int) -> tuple:
    """The layer forward with the analysis output rounded as above: y = T_out^T diag(gamma)
    C_hat (Delta C_bar), C_bar from z = T_in x.  Returns (Y, C_bar, Delta, Z)."""
    Z = analysis(T_in, X)
    Zbar, delta = quantize_ff(Z, bits)
    U = core(delta * Zbar.astype(np.float64), codes, scale, zero, gamma)
    return synthesis(T_out, U), Zbar, delta, Z
