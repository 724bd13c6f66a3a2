"""Oracle, part 5: a whole quantized layer from a seeded workload (plain fp64 CPU).

TEST INFRASTRUCTURE. Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline leg may
import this package; the product library never does, and shares no code with it.

Algorithm 1 with round-to-nearest in place of GPTQ: build the input and output frames, compute
C = T_out W T_in^T, optionally clip at 2 sigma, quantize each row to 2 bits, optionally derive
the de-noising gain.  Everything stays fp64 except the fp16 scale/zero the format stores.
"""
from __future__ import annotations

from dataclasses import dataclass
from fractions import Fraction

import numpy as np

import workloads as wlmod

from . import frames, gptq, pack, quant


@dataclass
class QuantLayer:
    name: str
    d_in: int
    d_out: int
    k_in: int
    k_out: int
    rho: int
    T_in: np.ndarray        # n_in x d_in analysis operator (fp64)
    T_out: np.ndarray       # n_out x d_out analysis operator (fp64); synthesis is T_out^T
    W: np.ndarray
    C: np.ndarray           # unquantized frame coefficients
    codes: np.ndarray       # uint8 n_out x n_in
    scale: np.ndarray       # float16 n_out
    zero: np.ndarray        # float16 n_out
    gamma: np.ndarray       # float32 n_out de-noising gain

    @property
    def n_in(self) -> int:
        return self.T_in.shape[0]

    @property
    def n_out(self) -> int:
        return self.T_out.shape[0]

    def packed(self) -> np.ndarray:
        return pack.pack(self.codes)


def build(W: np.ndarray, k_in: int, k_out: int, rho: int = wlmod.RHO, *, rot_in=None,
          rot_out=None, clip: bool = False, name: str = "layer", A_calib=None) -> QuantLayer:
    """With A_calib (calibration tokens, one per row) the codes come from the frame-domain GPTQ
    of Algorithm 1, step 4, against H = (T_in A^T)(T_in A^T)^T; otherwise from per-row RTN."""
    d_out, d_in = W.shape
    T_in = frames.frame(k_in, rho if k_in > 1 else d_in, d_in, rot_in)
    T_out = frames.frame(k_out, rho if k_out > 1 else d_out, d_out, rot_out)
    C = quant.coefficients(W, T_in, T_out)
    if clip:
        C = quant.clip_2sigma(C)
    if A_calib is None:
        codes, scale, zero = quant.rtn(C)
    else:
        C_prev = T_in @ np.asarray(A_calib, dtype=np.float64).T
        codes, scale, zero = gptq.gptq(C, gptq.hessian(C_prev))
    gamma = quant.wiener_gain(C, scale)
    return QuantLayer(name, d_in, d_out, k_in, k_out, rho, T_in, T_out, W, C, codes, scale,
                      zero, gamma)


def from_workload(wl_key: str, layer_name: str, r: Fraction | None = None, *,
                  rotate: bool = True, clip: bool = False, calib_tokens: int = 0) -> QuantLayer:
    """Quantized layer for one layer of a workload, with the workload's seed and draws."""
    wl = wlmod.WORKLOADS[wl_key]
    layer = next(l for l in wl.layers if l.name == layer_name)
    r = wl.redundancy[0] if r is None else Fraction(r)
    if wl.fixed_k is not None:
        k_in = k_out = wl.fixed_k
    else:
        k_in, _ = frames.choose_k(r, layer.d_in, wlmod.RHO)
        k_out, _ = frames.choose_k(r, layer.d_out, wlmod.RHO)
    W = wlmod.weight(wl, layer)
    rot_in = rot_out = None
    if rotate:
        rot_in = wlmod.rotation_draws(wl.seed, wl.key, layer.name, "in", d=layer.d_in)
        rot_out = wlmod.rotation_draws(wl.seed, wl.key, layer.name, "out", d=layer.d_out)
    A = wlmod.calibration(wl, layer, calib_tokens) if calib_tokens else None
    return build(W, k_in, k_out, rot_in=rot_in, rot_out=rot_out, clip=clip,
                 name=f"{wl_key}/{layer_name}", A_calib=A)
