"""Helpers for the GPU tests: upload an oracle layer, run the library through its C ABI, and
compare with the fp64 oracle."""
from __future__ import annotations

import functools

import numpy as np
import torch

import paper_2403_06082_gb300 as fq
import workloads as wl
from oracle import forward, layer

DEV = torch.device("cuda:0")


@functools.lru_cache(maxsize=8)
def oracle_layer(wl_key: str, name: str, r=None, rotate: bool = True):
    return layer.from_workload(wl_key, name, r, rotate=rotate)


def activations(wl_key: str, name: str, M: int) -> np.ndarray:
    wk = wl.WORKLOADS[wl_key]
    return wl.activations(wk, next(l for l in wk.layers if l.name == name), M)


class DeviceLayer:
    """Device copies of one quantized layer (codes packed by fq_pack)."""

    def __init__(self, L, dtype=torch.bfloat16):
        self.L = L
        self.dtype = dtype
        self.T_in = torch.from_numpy(np.ascontiguousarray(L.T_in)).to(DEV, dtype)
        self.T_out_t = torch.from_numpy(np.ascontiguousarray(L.T_out.T)).to(DEV, dtype)
        codes = torch.from_numpy(L.codes).to(DEV)
        words = torch.zeros(fq.fq_packed_words(L.n_out, L.n_in), dtype=torch.int32, device=DEV)
        self.C = fq.fq_pack(codes, torch.from_numpy(L.scale.view(np.int16)).to(DEV),
                            torch.from_numpy(L.zero.view(np.int16)).to(DEV), L.n_out, L.n_in,
                            words)
        self.gamma = torch.from_numpy(L.gamma).to(DEV)

    def forward(self, X: np.ndarray, use_gamma: bool = False, ws=None):
        L = self.L
        M = X.shape[0]
        mode = fq.FQ_BF16 if self.dtype == torch.bfloat16 else fq.FQ_FP32_DEBUG
        x = torch.from_numpy(X).to(DEV, self.dtype)
        y = torch.full((M, L.d_out), float("nan"), dtype=self.dtype, device=DEV)
        nbytes = fq.fq_workspace_bytes(M, L.d_in, L.n_in, L.n_out, L.d_out, mode)
        if ws is None:
            ws = torch.zeros(nbytes, dtype=torch.uint8, device=DEV)
        fq.fq_linear_forward(x, M, L.d_in, self.T_in, self.C, self.T_out_t, L.d_out,
                             self.gamma if use_gamma else None, y, ws, nbytes, mode)
        st = fq.fq_check(ws)
        assert st == 0, fq.fq_status_str(st)
        return y.double().cpu().numpy()


def reference(L, X: np.ndarray, use_gamma: bool = False) -> np.ndarray:
    return forward.layer_forward(X, L.T_in, L.codes, L.scale, L.zero, L.T_out,
                                 L.gamma if use_gamma else None)


def rel_frobenius(got: np.ndarray, ref: np.ndarray) -> float:
    return float(np.linalg.norm(got - ref) / np.linalg.norm(ref))


# Elementwise companions of the whole-output bound, per tolerance: |got - ref| <= a * rms(ref)
# + r * |ref| for every element.  The whole-output relative Frobenius error is the stated
# tolerance; on its own it lets one wrong output column through on the widest layers (a zero
# column of an 11008-wide output adds only sqrt(1/11008) ~ 0.0095).  bf16: rounding z, u and y
# to bf16 gives an error of ~3e-3 of the rms per element, ~1.5e-2 at the tail of 1e5-1e6
# elements; a = 0.05 and r = 0.02 leave margin above that and fail any element that is off by
# more than ~5% of the output's rms (a dropped or misplaced column or row fails at almost every
# element).  fp32 (debug mode): a = r = 1e-4.
ELEMENTWISE = {1e-2: (0.05, 0.02), 1e-5: (1e-4, 1e-4)}


def assert_parity(got: np.ndarray, ref: np.ndarray, tol: float) -> float:
    """Relative Frobenius error <= tol, and every element within the companion bound above.
    Returns the relative Frobenius error."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, (got.shape, ref.shape)
    assert np.isfinite(got).all(), "non-finite output"
    err = rel_frobenius(got, ref)
    assert err <= tol, f"relative Frobenius error {err:.3e} > {tol:g}"
    a, r = ELEMENTWISE[tol]
    bound = a * np.sqrt(np.mean(ref * ref)) + r * np.abs(ref)
    ratio = np.abs(got - ref) / bound
    worst = np.unravel_index(int(np.argmax(ratio)), ratio.shape)
    assert ratio[worst] <= 1.0, (
        f"element {worst}: got {got[worst]:.6g}, oracle {ref[worst]:.6g}, "
        f"{ratio[worst]:.2f} x the elementwise bound (Frobenius {err:.3e})")
    return err
