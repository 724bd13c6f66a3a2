"""Llama-2-70B-shaped layers (8192x8192, 28672x8192, 8192x28672) through the C ABI against the
fp64 oracle, relative Frobenius error <= 1e-2 in FQ_BF16.

The frames are built on the GPU by fq_frame_build from the workload's seeded rotation draws;
the oracle applies the same frames in structured form (oracle.frames.analysis_apply /
synthesis_apply, pinned against the dense construction), because the dense T of the 28672-wide
side takes 7 GB in fp64.  Codes, scales and zeros are seeded uniform draws: computing the real
frame coefficients C = T_out W T_in^T in fp64 at these sizes takes hours, and the layer's
arithmetic (analysis, code product, synthesis) is the same for any codes."""
from fractions import Fraction

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2403_06082_gb300 as fq  # noqa: E402
import workloads as wl  # noqa: E402
from fqgpu import DEV, rel_frobenius  # noqa: E402
from oracle import forward, frames  # noqa: E402

pytestmark = pytest.mark.gpu
WK = wl.WORKLOADS["llama2_70b"]
RHO = 16


def gpu_frame(k, d, draws):
    nb = fq.fq_frame_workspace_bytes(k, RHO, d, draws.a, draws.b)
    ws = torch.empty(nb, dtype=torch.uint8, device=DEV)
    T = torch.empty(k * RHO, d, dtype=torch.float32, device=DEV)
    fq.fq_frame_build(k, RHO, d, (draws.a, draws.b, draws.ga, draws.gb, draws.perm, draws.signs),
                      T, ws, nb)
    del ws
    out = T.to(torch.bfloat16)
    del T
    return out


def run_layer(name, r, M):
    """The layer through the C ABI on M tokens: (y on the host, X, the oracle as a function of
    the tokens it is given)."""
    layer = next(l for l in WK.layers if l.name == name)
    k_in, _ = frames.choose_k(Fraction(r), layer.d_in, RHO)
    k_out, _ = frames.choose_k(Fraction(r), layer.d_out, RHO)
    n_in, n_out = k_in * RHO, k_out * RHO
    draws_in = wl.rotation_draws(WK.seed, WK.key, layer.name, "in", d=layer.d_in)
    draws_out = wl.rotation_draws(WK.seed, WK.key, layer.name, "out", d=layer.d_out)
    codes = wl.random_codes(WK.seed, WK.key, layer.name, n_out=n_out, n_in=n_in)
    scale, zero = wl.random_scale_zero(WK.seed, WK.key, layer.name, n_out=n_out, mag=0.01)
    X = wl.activations(WK, layer, M)

    T_in = gpu_frame(k_in, layer.d_in, draws_in)
    T_out_t = gpu_frame(k_out, layer.d_out, draws_out).t().contiguous()
    torch.cuda.empty_cache()
    words = torch.zeros(fq.fq_packed_words(n_out, n_in), dtype=torch.int32, device=DEV)
    C = fq.fq_pack(torch.from_numpy(codes).to(DEV), torch.from_numpy(scale.view(np.int16)).to(DEV),
                   torch.from_numpy(zero.view(np.int16)).to(DEV), n_out, n_in, words)
    x = torch.from_numpy(X).to(DEV, torch.bfloat16)
    y = torch.empty(M, layer.d_out, dtype=torch.bfloat16, device=DEV)
    nb = fq.fq_workspace_bytes(M, layer.d_in, n_in, n_out, layer.d_out)
    ws = torch.zeros(nb, dtype=torch.uint8, device=DEV)
    fq.fq_linear_forward(x, M, layer.d_in, T_in, C, T_out_t, layer.d_out, None, y, ws, nb)
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
    err = rel_frobenius(got, ref(X))
    assert err <= 1e-2, err


@pytest.mark.parametrize("name,r,M", [
    ("q", "11/10", 1024), ("q", "1", 4096), ("gate", "11/10", 4096), ("down", "6/5", 1024),
])
def test_llama70b_large_batch_sampled(name, r, M):
    """The whole batch runs on the GPU (the tensor-core path, 256-token tiles); the oracle
    checks eight tokens: the first and last of the batch and of token tiles, and the middle."""
    got, X, ref = run_layer(name, r, M)
    rows = sorted({0, 1, 255, 256, M // 2, M // 2 + 1, M - 2, M - 1})
    err = rel_frobenius(got[rows], ref(X[rows]))
    assert err <= 1e-2, err
    assert np.isfinite(got).all()
