"""Weight-reconstruction path (include/framequant_dense.h) against the fp64 oracle: the rebuilt
weight W_hat = T_out^T diag(gamma) C_hat T_in and the dense forward x W_hat^T, relative
Frobenius error <= 1e-2 (bf16 z, u and W_hat)."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2403_06082_gb300 as fq  # noqa: E402
from fqgpu import DEV, DeviceLayer, activations, oracle_layer, reference, assert_parity, rel_frobenius  # noqa: E402
from oracle import quant  # noqa: E402

pytestmark = pytest.mark.gpu
BF16 = torch.bfloat16


def _w_hat(L, D, use_gamma):
    W = torch.full((L.d_out, L.d_in), float("nan"), dtype=BF16, device=DEV)
    nb = fq.fq_reconstruct_workspace_bytes(L.d_in, L.n_in, L.n_out, L.d_out)
    ws = torch.zeros(nb, dtype=torch.uint8, device=DEV)
    fq.fq_reconstruct_weight(D.T_in, D.C, D.T_out_t, L.d_in, L.d_out,
                             D.gamma if use_gamma else None, W, ws, nb)
    assert fq.fq_check(ws) == 0
    return W


def _oracle_w_hat(L, use_gamma):
    C_hat = quant.dequantize(L.codes, L.scale, L.zero)
    if use_gamma:
        C_hat = C_hat * L.gamma.astype(np.float64)[:, None]
    return L.T_out.T @ C_hat @ L.T_in


@pytest.mark.parametrize("wl_key,name,use_gamma", [
    ("single256", "single", False), ("single256", "single", True), ("vit_b16_mlp", "fc1", False),
    ("vit_b16_mlp", "fc2", True),
])
def test_reconstructed_weight(wl_key, name, use_gamma):
    L = oracle_layer(wl_key, name)
    W = _w_hat(L, DeviceLayer(L, BF16), use_gamma)
    err = assert_parity(W.double().cpu().numpy(), _oracle_w_hat(L, use_gamma), 1e-2)


@pytest.mark.parametrize("name,use_gamma", [("q", False), ("gate", True)])
def test_reconstructed_weight_llama7b_sampled_rows(name, use_gamma):
    """The 7B shapes (4096 x 4096 and 11008 x 4096 at r = 1.1): the whole W_hat is rebuilt on
    the GPU; the oracle computes 64 seeded rows of T_out^T diag(gamma) C_hat T_in."""
    import workloads as wl
    L = oracle_layer("llama2_7b_prefill", name)
    W = _w_hat(L, DeviceLayer(L, BF16), use_gamma).double().cpu().numpy()
    rows = np.sort(wl.rng(3, "w-hat-rows", name).choice(L.d_out, 64, replace=False))
    C_hat = quant.dequantize(L.codes, L.scale, L.zero)
    if use_gamma:
        C_hat = C_hat * L.gamma.astype(np.float64)[:, None]
    ref = (L.T_out.T[rows] @ C_hat) @ L.T_in
    assert_parity(W[rows], ref, 1e-2)


@pytest.mark.parametrize("M", [1, 8, 100, 300])
def test_dense_forward_matches_the_layer(M):
    L = oracle_layer("single256", "single")
    D = DeviceLayer(L, BF16)
    W = _w_hat(L, D, True)
    X = activations("single256", "single", M)
    x = torch.from_numpy(X).to(DEV, BF16)
    y = torch.full((M, L.d_out), float("nan"), dtype=BF16, device=DEV)
    nb = fq.fq_dense_workspace_bytes(M, L.d_in, L.d_out)
    ws = torch.zeros(nb, dtype=torch.uint8, device=DEV)
    fq.fq_dense_forward(x, M, L.d_in, W, L.d_out, y, ws, nb)
    assert fq.fq_check(ws) == 0
    err = assert_parity(y.double().cpu().numpy(), reference(L, X, True), 1e-2)


def test_dense_forward_vit_batch():
    L = oracle_layer("vit_b16_mlp", "fc1")
    D = DeviceLayer(L, BF16)
    W = _w_hat(L, D, False)
    M = 1000
    X = activations("vit_b16_mlp", "fc1", M)
    x = torch.from_numpy(X).to(DEV, BF16)
    y = torch.empty(M, L.d_out, dtype=BF16, device=DEV)
    nb = fq.fq_dense_workspace_bytes(M, L.d_in, L.d_out)
    ws = torch.zeros(nb, dtype=torch.uint8, device=DEV)
    fq.fq_dense_forward(x, M, L.d_in, W, L.d_out, y, ws, nb)
    assert fq.fq_check(ws) == 0
    rows = [0, 1, 127, 128, 499, 998, 999]
    err = assert_parity(y.double().cpu().numpy()[rows], reference(L, X[rows], False), 1e-2)


def test_errors_launch_nothing():
    L = oracle_layer("single256", "single")
    D = DeviceLayer(L, BF16)
    W = torch.full((L.d_out, L.d_in), 7.0, dtype=BF16, device=DEV)
    nb = fq.fq_reconstruct_workspace_bytes(L.d_in, L.n_in, L.n_out, L.d_out)
    ws = torch.zeros(nb, dtype=torch.uint8, device=DEV)
    with pytest.raises(fq.FrameQuantError) as e:
        fq.fq_reconstruct_weight(D.T_in, D.C, D.T_out_t, L.d_in, L.d_out, None, W, ws, nb - 256)
    assert e.value.status == 4
    with pytest.raises(fq.FrameQuantError) as e:
        fq.fq_reconstruct_weight(D.T_in, D.C, D.T_out_t, L.d_in, L.d_out, None,
                                 W.view(-1)[1:1 + L.d_out * L.d_in], ws, nb)
    assert e.value.status == 2
    torch.cuda.synchronize()
    assert (W == 7.0).all()
