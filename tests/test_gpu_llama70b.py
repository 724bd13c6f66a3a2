"""Llama-2-70B-shaped layers (8192x8192, 28672x8192, 8192x28672) through the C ABI against the
fp64 oracle: relative Frobenius error <= 1e-2 in FQ_BF16 and <= 1e-5 in FQ_FP32_DEBUG, each with
its elementwise companion bound.

The frames are built on the GPU by fq_frame_build from the workload's seeded rotation draws;
the oracle applies the same frames in structured form (oracle.frames.analysis_apply /
synthesis_apply, pinned against the dense construction), because the dense T of the 28672-wide
side takes 7 GB in fp64.  On the 8192 x 8192 layer the codes are the configuration's own: the
oracle computes C = T_out W T_in^T for W ~ N(0, 0.015^2) in structured form (the analysis of
the rows of W, then of the columns of the result; Sec. 3, D_l = P_l^T Theta_l P_prev) and
quantizes it per row (quant.rtn).  On the larger layers the codes, scales and zeros are seeded
uniform draws: the layer's arithmetic (analysis, code product, synthesis) is the same for any
codes, and the fp64 coefficients of a 28672-wide layer take minutes of host time per test.
"""
import functools
from fractions import Fraction

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2403_06082_gb300 as fq  # noqa: E402
import workloads as wl  # noqa: E402
from fqgpu import DEV, assert_parity, rel_frobenius  # noqa: E402
from oracle import forward, frames, quant  # noqa: E402

pytestmark = pytest.mark.gpu
WK = wl.WORKLOADS["llama2_70b"]
RHO = 16


def gpu_frame(k, d, draws, dtype=torch.bfloat16):
    nb = fq.fq_frame_workspace_bytes(k, RHO, d, draws.a, draws.b)
    ws = torch.empty(nb, dtype=torch.uint8, device=DEV)
    T = torch.empty(k * RHO, d, dtype=torch.float32, device=DEV)
    fq.fq_frame_build(k, RHO, d, (draws.a, draws.b, draws.ga, draws.gb, draws.perm, draws.signs),
                      T, ws, nb)
    del ws
    if dtype == torch.float32:
        return T
    out = T.to(dtype)
    del T
    return out


@functools.lru_cache(maxsize=1)
def real_codes(name, r):
    """Per-row RTN codes of the configuration's own frame coefficients C = T_out W T_in^T,
    computed by the oracle in fp64 without forming T (about half a minute on 16 cores)."""
    layer = next(l for l in WK.layers if l.name == name)
    k_in, _ = frames.choose_k(Fraction(r), layer.d_in, RHO)
    k_out, _ = frames.choose_k(Fraction(r), layer.d_out, RHO)
    draws_in = wl.rotation_draws(WK.seed, WK.key, layer.name, "in", d=layer.d_in)
    draws_out = wl.rotation_draws(WK.seed, WK.key, layer.name, "out", d=layer.d_out)
    W = wl.weight(WK, layer)
    WT = frames.analysis_apply(k_in, RHO, layer.d_in, draws_in, W)          # W T_in^T
    del W
    C = np.ascontiguousarray(
        frames.analysis_apply(k_out, RHO, layer.d_out, draws_out, WT.T).T)   # T_out W T_in^T
    del WT
    codes, scale, zero = quant.rtn(C)
    return np.ascontiguousarray(codes), scale, zero


def run_layer(name, r, M, dtype=torch.bfloat16, codes_from_w=False):
    """The layer through the C ABI on M tokens: (y on the host, X, the oracle as a function of
    the tokens it is given)."""
    layer = next(l for l in WK.layers if l.name == name)
    k_in, _ = frames.choose_k(Fraction(r), layer.d_in, RHO)
    k_out, _ = frames.choose_k(Fraction(r), layer.d_out, RHO)
    n_in, n_out = k_in * RHO, k_out * RHO
    draws_in = wl.rotation_draws(WK.seed, WK.key, layer.name, "in", d=layer.d_in)
    draws_out = wl.rotation_draws(WK.seed, WK.key, layer.name, "out", d=layer.d_out)
    if codes_from_w:
        codes, scale, zero = real_codes(name, r)
    else:
        codes = wl.random_codes(WK.seed, WK.key, layer.name, n_out=n_out, n_in=n_in)
        scale, zero = wl.random_scale_zero(WK.seed, WK.key, layer.name, n_out=n_out, mag=0.01)
    X = wl.activations(WK, layer, M)

    T_in = gpu_frame(k_in, layer.d_in, draws_in, dtype)
    T_out_t = gpu_frame(k_out, layer.d_out, draws_out, dtype).t().contiguous()
    torch.cuda.empty_cache()
    words = torch.zeros(fq.fq_packed_words(n_out, n_in), dtype=torch.int32, device=DEV)
    C = fq.fq_pack(torch.from_numpy(codes).to(DEV), torch.from_numpy(scale.view(np.int16)).to(DEV),
                   torch.from_numpy(zero.view(np.int16)).to(DEV), n_out, n_in, words)
    mode = fq.FQ_BF16 if dtype == torch.bfloat16 else fq.FQ_FP32_DEBUG
    x = torch.from_numpy(X).to(DEV, dtype)
    y = torch.empty(M, layer.d_out, dtype=dtype, device=DEV)
    nb = fq.fq_workspace_bytes(M, layer.d_in, n_in, n_out, layer.d_out, mode)
    ws = torch.zeros(nb, dtype=torch.uint8, device=DEV)
    fq.fq_linear_forward(x, M, layer.d_in, T_in, C, T_out_t, layer.d_out, None, y, ws, nb, mode)
    assert fq.fq_check(ws) == 0
    got = y.double().cpu().numpy()
    del T_in, T_out_t, words, x, y, ws
    torch.cuda.empty_cache()

    def ref(Xs):
        Z = frames.analysis_apply(k_in, RHO, layer.d_in, draws_in, Xs)
        U = forward.core(Z, codes, scale, zero)
        return frames.synthesis_apply(k_out, RHO, layer.d_out, draws_out, U)

    return got, X, ref


@pytest.mark.parametrize("name,r,M", [
    ("q", "1", 16), ("q", "11/10", 1), ("q", "11/10", 16), ("q", "6/5", 16),
    ("q", "11/10", 128), ("gate", "11/10", 16), ("down", "11/10", 1), ("down", "6/5", 16),
])
def test_llama70b_layer(name, r, M):
    got, X, ref = run_layer(name, r, M)
    err = assert_parity(got, ref(X), 1e-2)


@pytest.mark.parametrize("name,r,M", [
    ("q", "11/10", 1024), ("q", "1", 4096), ("gate", "11/10", 4096), ("down", "6/5", 1024),
])
def test_llama70b_large_batch_sampled(name, r, M):
    """The whole batch runs on the GPU (the tensor-core path, 256-token tiles); the oracle
    checks eight tokens: the first and last of the batch and of token tiles, and the middle."""
    got, X, ref = run_layer(name, r, M)
    rows = sorted({0, 1, 255, 256, M // 2, M // 2 + 1, M - 2, M - 1})
    err = assert_parity(got[rows], ref(X[rows]), 1e-2)
    assert np.isfinite(got).all()


@pytest.mark.parametrize("M,dtype,tol", [(16, torch.bfloat16, 1e-2), (1, torch.bfloat16, 1e-2),
                                         (16, torch.float32, 1e-5)],
                         ids=["bf16-m16", "bf16-m1", "fp32-m16"])
def test_llama70b_q_codes_of_its_own_weight(M, dtype, tol):
    """The 8192 x 8192 layer at r = 1.1 with the RTN codes of its own W ~ N(0, 0.015^2), in
    both modes."""
    got, X, ref = run_layer("q", "11/10", M, dtype, codes_from_w=True)
    assert_parity(got, ref(X), tol)


def test_llama70b_gate_fp32_debug():
    """The widest 70B layer (28672 x 8192 at r = 1.1, n_out = 31552) in FQ_FP32_DEBUG."""
    got, X, ref = run_layer("gate", "11/10", 4, torch.float32)
    assert_parity(got, ref(X), 1e-5)
