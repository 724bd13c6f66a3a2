"""fq_linear_forward through the C ABI against the fp64 oracle: relative Frobenius error
<= 1e-2 in FQ_BF16 (bf16 operands, fp32 accumulation, bf16 z and u) and <= 1e-5 in
FQ_FP32_DEBUG (fp32 everywhere).  At full workload sizes with many tokens the oracle computes
a seeded sample of tokens, which the GPU computes as part of the full batch."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2403_06082_gb300 as fq  # noqa: E402
import workloads as wl  # noqa: E402
from fqgpu import (DEV, DeviceLayer, activations, oracle_layer, reference,  # noqa: E402
                   rel_frobenius, assert_parity)

pytestmark = pytest.mark.gpu
BF16, FP32 = torch.bfloat16, torch.float32
TOL = {BF16: 1e-2, FP32: 1e-5}
DT = [pytest.param(FP32, id="fp32"), pytest.param(BF16, id="bf16")]


def _check(L, X, dtype, use_gamma, sample=None):
    got = DeviceLayer(L, dtype).forward(X, use_gamma)
    if sample is not None:
        got, X = got[sample], X[sample]
    err = assert_parity(got, reference(L, X, use_gamma), TOL[dtype])
    return err


@pytest.mark.parametrize("dtype", DT)
@pytest.mark.parametrize("use_gamma", [False, True])
def test_single256_m8(dtype, use_gamma):
    L = oracle_layer("single256", "single")
    _check(L, activations("single256", "single", 8), dtype, use_gamma)


@pytest.mark.parametrize("M", [1, 3, 16, 17, 33, 64, 100, 129, 300, 1000])
@pytest.mark.parametrize("dtype", DT)
def test_ragged_token_counts(M, dtype):
    L = oracle_layer("single256", "single")
    _check(L, activations("single256", "single", M), dtype, True)


@pytest.mark.parametrize("name", ["q", "gate", "down"])
@pytest.mark.parametrize("M", [1, 4, 16])
def test_llama7b_decode_full(name, M):
    L = oracle_layer("llama2_7b_decode", name)
    _check(L, activations("llama2_7b_decode", name, M), BF16, False)


@pytest.mark.parametrize("name", ["q", "gate", "down"])
@pytest.mark.parametrize("M", [1, 16])
def test_llama7b_decode_fp32_debug(name, M):
    L = oracle_layer("llama2_7b_decode", name)
    _check(L, activations("llama2_7b_decode", name, M), FP32, name == "gate")


@pytest.mark.parametrize("name,use_gamma", [("q", True), ("gate", False), ("down", True)])
def test_llama7b_prefill_fp32_debug_sampled(name, use_gamma):
    """The prefill configuration (2048 tokens, filter on and off) in FQ_FP32_DEBUG: the whole
    batch runs on the GPU, the oracle checks a seeded sample of tokens."""
    L = oracle_layer("llama2_7b_prefill", name)
    X = activations("llama2_7b_prefill", name, 2048)
    sample = np.sort(wl.rng(3, "sample-fp32", name).choice(2048, 32, replace=False))
    _check(L, X, FP32, use_gamma, sample)


@pytest.mark.parametrize("name", ["fc1", "fc2"])
def test_vit_mlp_fp32_debug_sampled(name):
    """The ViT-B/16 MLP pair at its full 12608-token batch in FQ_FP32_DEBUG, sampled tokens."""
    L = oracle_layer("vit_b16_mlp", name)
    X = activations("vit_b16_mlp", name, 12608)
    sample = np.sort(wl.rng(1, "sample-fp32", name).choice(12608, 48, replace=False))
    _check(L, X, FP32, name == "fc2", sample)


@pytest.mark.parametrize("name,use_gamma", [("q", False), ("q", True), ("up", True)])
def test_llama7b_prefill_sampled(name, use_gamma):
    L = oracle_layer("llama2_7b_prefill", name)
    X = activations("llama2_7b_prefill", name, 2048)
    sample = np.sort(wl.rng(3, "sample", name).choice(2048, 48, replace=False))
    _check(L, X, BF16, use_gamma, sample)


def test_llama7b_prefill_m4096_sampled():
    # the largest prefill batch of the workload: 4096 tokens, filter off, 32 tokens checked
    L = oracle_layer("llama2_7b_prefill", "gate")
    X = activations("llama2_7b_prefill", "gate", 4096)
    sample = np.sort(wl.rng(3, "sample-4096", "gate").choice(4096, 32, replace=False))
    _check(L, X, BF16, False, sample)


@pytest.mark.parametrize("name", ["fc1", "fc2"])
def test_vit_mlp_full_sampled(name):
    L = oracle_layer("vit_b16_mlp", name)
    X = activations("vit_b16_mlp", name, 12608)
    sample = np.sort(wl.rng(1, "sample", name).choice(12608, 64, replace=False))
    _check(L, X, BF16, False, sample)


def test_rotation_off_block_sparse_frames():
    L = oracle_layer("single256", "single", rotate=False)
    assert (L.T_in == 0).mean() > 0.8            # block-diagonal structure kept
    for dtype in (FP32, BF16):
        _check(L, activations("single256", "single", 40), dtype, True)


def test_degenerate_rows():
    import copy
    L = copy.copy(oracle_layer("single256", "single"))
    L.codes = L.codes.copy()
    L.scale = L.scale.copy()
    L.zero = L.zero.copy()
    L.codes[:20] = 0                              # constant rows: scale 1, value = zero
    L.scale[:20] = np.float16(1.0)
    L.zero[:20] = np.float16(-0.25)
    L.codes[20:40] = 3                            # all codes at the top level
    for dtype in (FP32, BF16):
        _check(L, activations("single256", "single", 24), dtype, False)


def test_workspace_reuse_across_shapes_and_determinism():
    La = oracle_layer("single256", "single")
    Lb = oracle_layer("vit_b16_mlp", "fc2")
    nbytes = max(fq.fq_workspace_bytes(M, L.d_in, L.n_in, L.n_out, L.d_out, 0)
                 for L, M in ((La, 8), (Lb, 300)))
    ws = torch.zeros(nbytes, dtype=torch.uint8, device=DEV)
    Da, Db = DeviceLayer(La, BF16), DeviceLayer(Lb, BF16)
    Xa = activations("single256", "single", 8)
    Xb = activations("vit_b16_mlp", "fc2", 300)
    ya1 = Da.forward(Xa, True, ws=ws)
    yb1 = Db.forward(Xb, False, ws=ws)
    ya2 = Da.forward(Xa, True, ws=ws)
    yb2 = Db.forward(Xb, False, ws=ws)
    np.testing.assert_array_equal(ya1, ya2)       # fixed-order reductions: bitwise repeatable
    np.testing.assert_array_equal(yb1, yb2)
    assert_parity(ya1, reference(La, Xa, True), 1e-2)
    assert_parity(yb1, reference(Lb, Xb, False), 1e-2)


def test_argument_errors_launch_nothing():
    L = oracle_layer("single256", "single")
    D = DeviceLayer(L, BF16)
    M = 8
    x = torch.from_numpy(activations("single256", "single", M)).to(DEV, BF16)
    y = torch.full((M + 1, L.d_out), 7.0, dtype=BF16, device=DEV)
    nb = fq.fq_workspace_bytes(M, L.d_in, L.n_in, L.n_out, L.d_out, 0)
    ws = torch.zeros(nb + 512, dtype=torch.uint8, device=DEV)

    def call(**kw):
        a = dict(x=x, M=M, d_in=L.d_in, T_in=D.T_in, C=D.C, T_out_t=D.T_out_t, d_out=L.d_out,
                 gamma=None, y=y[:M], ws=ws[:nb], ws_bytes=nb, mode=0)
        a.update(kw)
        with pytest.raises(fq.FrameQuantError) as e:
            fq.fq_linear_forward(**a)
        return e.value.status

    assert call(ws_bytes=nb - 1) == 4
    assert call(ws=ws[16:16 + nb]) == 2                     # workspace not 256-byte aligned
    assert call(y=y.view(-1)[1:1 + M * L.d_out]) == 2       # output misaligned by 2 bytes
    assert call(M=0) == 1
    assert call(mode=3) == 1
    assert call(d_in=L.d_in + 4) == 2
    bad = fq.Packed(D.C.words, D.C.scale, D.C.zero, L.n_out, L.n_in + 8, D.C.ld_words)
    assert call(C=bad) == 2
    torch.cuda.synchronize()
    assert (y == 7.0).all()                                 # nothing was written
    # and a good call on the same buffers still works and reports FQ_OK
    fq.fq_linear_forward(x, M, L.d_in, D.T_in, D.C, D.T_out_t, L.d_out, None, y[:M], ws[:nb],
                         nb, 0)
    assert fq.fq_check(ws) == 0


def test_stream_argument():
    L = oracle_layer("single256", "single")
    D = DeviceLayer(L, BF16)
    X = activations("single256", "single", 16)
    s = torch.cuda.Stream()
    x = torch.from_numpy(X).to(DEV, BF16)
    y = torch.empty(16, L.d_out, dtype=BF16, device=DEV)
    nb = fq.fq_workspace_bytes(16, L.d_in, L.n_in, L.n_out, L.d_out, 0)
    ws = torch.zeros(nb, dtype=torch.uint8, device=DEV)
    torch.cuda.synchronize()
    with torch.cuda.stream(s):
        fq.fq_linear_forward(x, 16, L.d_in, D.T_in, D.C, D.T_out_t, L.d_out, D.gamma, y, ws, nb,
                             0, stream=s)
    assert fq.fq_check(ws, stream=s) == 0
    assert_parity(y.double().cpu().numpy(), reference(L, X, True), 1e-2)


@pytest.mark.parametrize("name,M,use_gamma", [
    ("q", 65, False), ("q", 128, True), ("gate", 100, False), ("down", 128, False),
    ("q", 200, False), ("down", 256, True),
])
def test_split_k_tensor_core_path(name, M, use_gamma):
    """Batches just above the decode kernel's range on the 7B shapes: phases with fewer tiles
    than SMs split each tile's K range and the last split to arrive adds the partials in
    split order, so the result is also bitwise repeatable and independent of arrival order."""
    L = oracle_layer("llama2_7b_decode", name)
    X = activations("llama2_7b_decode", name, M)
    D = DeviceLayer(L, BF16)
    got = D.forward(X, use_gamma)
    assert_parity(got, reference(L, X, use_gamma), TOL[BF16])
    np.testing.assert_array_equal(got, D.forward(X, use_gamma))


def test_split_k_under_sm_budget():
    """A smaller SM budget changes the split count; the result stays within tolerance."""
    L = oracle_layer("llama2_7b_decode", "gate")
    X = activations("llama2_7b_decode", "gate", 128)
    D = DeviceLayer(L, BF16)
    x = torch.from_numpy(X).to(DEV, BF16)
    ref = reference(L, X, False)
    for budget in (40, 100, 0):
        y = torch.full((128, L.d_out), float("nan"), dtype=BF16, device=DEV)
        nb = fq.fq_workspace_bytes(128, L.d_in, L.n_in, L.n_out, L.d_out, 0)
        ws = torch.zeros(nb, dtype=torch.uint8, device=DEV)
        fq.fq_linear_forward_sms(x, 128, L.d_in, D.T_in, D.C, D.T_out_t, L.d_out, None, y, ws,
                                 nb, budget)
        assert fq.fq_check(ws) == 0
        assert_parity(y.double().cpu().numpy(), ref, TOL[BF16])
