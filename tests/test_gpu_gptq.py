"""The frame-domain GPTQ of Algorithm 1 on the GPU (fq_gptq_hessian, fq_quantize_gptq) against
the fp64 oracle (oracle.gptq).  Both sides work in fp64 and round each coefficient with the same
arithmetic inside a block of columns; they differ only in how the inverse Hessian's factor and
the block-to-block update are summed (rounding at 1e-15), so the codes must agree except where a
coefficient sits that close to the middle of two levels: every code is compared, and the per-row
scale and zero bit for bit."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2403_06082_gb300 as fq  # noqa: E402
import workloads as wl  # noqa: E402
from fqgpu import DEV, oracle_layer  # noqa: E402
from oracle import gptq, quant  # noqa: E402

pytestmark = pytest.mark.gpu


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float64)).to(DEV)


def _gpu_hessian(Z):
    N, n = Z.shape
    H = torch.empty(n, n, dtype=torch.float64, device=DEV)
    fq.fq_gptq_hessian(_dev(Z), N, n, H)
    return H


def _gpu_gptq(D, H, clip=False, damp=0.01):
    n_out, n_in = D.shape
    codes = torch.full((n_out, n_in), 255, dtype=torch.uint8, device=DEV)
    scale = torch.empty(n_out, dtype=torch.int16, device=DEV)
    zero = torch.empty(n_out, dtype=torch.int16, device=DEV)
    gamma = torch.empty(n_out, dtype=torch.float32, device=DEV)
    nb = fq.fq_gptq_workspace_bytes(n_out, n_in)
    ws = torch.zeros(nb, dtype=torch.uint8, device=DEV)
    Ht = H if torch.is_tensor(H) else _dev(H)
    fq.fq_quantize_gptq(_dev(D), n_out, n_in, Ht, codes, scale, zero, gamma, ws, nb, damp, clip)
    return (codes.cpu().numpy(), scale.cpu().numpy().view(np.float16),
            zero.cpu().numpy().view(np.float16), gamma.cpu().numpy())


def _compare(got, ref, D, H, max_mismatch=0):
    codes, scale, zero, gamma = got
    rc, rs, rz = ref
    np.testing.assert_array_equal(scale.view(np.uint16), rs.view(np.uint16))
    np.testing.assert_array_equal(zero.view(np.uint16), rz.view(np.uint16))
    assert codes.max() <= 3
    mism = int((codes != rc).sum())
    assert mism <= max_mismatch, (mism, codes.size)
    np.testing.assert_allclose(gamma, quant.wiener_gain(D, rs), rtol=2e-7)
    # the loss the method minimises, against the oracle's codes
    lg = gptq.proxy_loss(D, quant.dequantize(codes, scale, zero), H)
    lr = gptq.proxy_loss(D, quant.dequantize(rc, rs, rz), H)
    assert lg == pytest.approx(lr, rel=1e-9 if mism == 0 else 1e-3)


def test_hessian_matches_the_product():
    Z = wl.rng(0, "gptq-gpu-h").standard_normal((300, 288))
    H = _gpu_hessian(Z).cpu().numpy()
    np.testing.assert_allclose(H, gptq.hessian(Z.T), rtol=1e-12, atol=1e-10)
    np.testing.assert_array_equal(H, H.T)


@pytest.mark.parametrize("seed,n_out,n_in", [(0, 64, 200), (1, 130, 257), (2, 16, 129)])
def test_random_problems(seed, n_out, n_in):
    g = np.random.default_rng(seed)
    D = g.standard_normal((n_out, n_in))
    mix = g.standard_normal((n_in, n_in)) / np.sqrt(n_in) + np.eye(n_in)
    C_prev = mix @ g.standard_normal((n_in, 3 * n_in))            # correlated coordinates
    H = gptq.hessian(C_prev)
    _compare(_gpu_gptq(D, H), gptq.gptq(D, H), D, H)


@pytest.mark.parametrize("clip", [False, True])
def test_single256_with_calibration_tokens(clip):
    """The 256 x 256 layer's frame coefficients (n = 288) against the Hessian of 512
    calibration tokens (Algorithm 1, steps 2-4 with and without the 2-sigma clip)."""
    L = oracle_layer("single256", "single")
    wk = wl.WORKLOADS["single256"]
    A = wl.calibration(wk, wk.layers[0], 512)
    Z = A.astype(np.float64) @ L.T_in.T                         # C_prev^T
    H = _gpu_hessian(Z)
    D = quant.clip_2sigma(L.C) if clip else L.C
    ref = gptq.quantize_layer(L.C, Z.T, clip=clip)
    _compare(_gpu_gptq(L.C, H, clip=clip), ref, D, gptq.hessian(Z.T))


def test_vit_fc1_with_calibration_tokens():
    """ViT-B/16 fc1 (3392 x 848 frame coefficients) with the clip, 1024 calibration tokens;
    below round-to-nearest's loss as the method intends."""
    L = oracle_layer("vit_b16_mlp", "fc1")
    wk = wl.WORKLOADS["vit_b16_mlp"]
    layer = next(l for l in wk.layers if l.name == "fc1")
    A = wl.calibration(wk, layer, 1024)
    Z = A.astype(np.float64) @ L.T_in.T
    H64 = gptq.hessian(Z.T)
    got = _gpu_gptq(L.C, _gpu_hessian(Z), clip=True)
    D = quant.clip_2sigma(L.C)
    ref = gptq.gptq(D, H64)
    _compare(got, ref, D, H64, max_mismatch=int(1e-5 * D.size))
    rtn = quant.rtn(D)
    assert gptq.proxy_loss(D, quant.dequantize(got[0], got[1], got[2]), H64) < \
        0.9 * gptq.proxy_loss(D, quant.dequantize(*rtn), H64)


def test_diagonal_hessian_is_round_to_nearest():
    D = wl.rng(3, "gptq-gpu-diag").standard_normal((40, 96))
    H = np.diag(np.linspace(0.5, 3.0, 96))
    codes, scale, zero, _ = _gpu_gptq(D, H)
    rc, rs, rz = quant.rtn(D)
    np.testing.assert_array_equal(codes, rc)


def test_refusals_and_a_singular_hessian():
    D = wl.rng(4, "gptq-gpu-bad").standard_normal((16, 32))
    with pytest.raises(fq.FrameQuantError) as e:
        _gpu_gptq(D, np.eye(32), damp=-1.0)
    assert e.value.status == 1
    # H = 0 with no damping is not positive definite: reported, no fault, the context usable
    with pytest.raises(fq.FrameQuantError) as e:
        _gpu_gptq(D, np.zeros((32, 32)), damp=0.0)
    assert e.value.status == 7
    codes, _, _, _ = _gpu_gptq(D, np.eye(32))
    np.testing.assert_array_equal(codes, quant.rtn(D)[0])
