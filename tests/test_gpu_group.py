"""fq_linear_forward_group: independent layers (q | k | v, gate | up) in one fused launch
through the C ABI, each layer's output against the fp64 oracle (relative Frobenius error
<= 1e-2 with the elementwise companion bound, FQ_BF16).  The launch interleaves the layers'
phases, so these cases cover the per-layer tensor maps, ready flags, code blocks and epilogue
constants, mixed shapes in one launch, every token tile width (16, 32, 64), SM budgets, the
sequential path of larger batches, workspace reuse with single-layer calls, and the host-side
refusals."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2403_06082_gb300 as fq  # noqa: E402
from fqgpu import (DEV, DeviceLayer, activations, assert_parity, oracle_layer,  # noqa: E402
                   reference)

pytestmark = pytest.mark.gpu
BF16 = torch.bfloat16


def _group(specs, M, shared_x=True, max_sms=0, ws=None):
    """specs: [(workload, layer name, use_gamma)]; returns the per-layer outputs and the
    oracle's."""
    Ds, Xs, ys, layers = [], [], [], []
    X0 = None
    for wl_key, name, use_gamma in specs:
        L = oracle_layer(wl_key, name)
        D = DeviceLayer(L, BF16)
        if shared_x and X0 is not None and X0.shape[1] == L.d_in:
            X = X0
        else:
            X = activations(wl_key, name, M)
            X0 = X if X0 is None else X0
        x = torch.from_numpy(X).to(DEV, BF16)
        y = torch.full((M, L.d_out), float("nan"), dtype=BF16, device=DEV)
        Ds.append((D, use_gamma))
        Xs.append((X, x))
        ys.append(y)
        layers.append(fq.Layer(x, L.d_in, D.T_in, D.C, D.T_out_t, L.d_out,
                               D.gamma if use_gamma else None, y))
    nb = fq.fq_group_workspace_bytes(M, layers)
    assert nb > 0
    if ws is None:
        ws = torch.zeros(nb, dtype=torch.uint8, device=DEV)
    fq.fq_linear_forward_group(M, layers, ws, nb, max_sms=max_sms)
    assert fq.fq_check(ws) == 0, fq.fq_status_str(fq.fq_check(ws))
    out = []
    for (D, g), (X, _), y in zip(Ds, Xs, ys):
        out.append((y.double().cpu().numpy(), reference(D.L, X, g)))
    return out, layers, ws


@pytest.mark.parametrize("M", [1, 16])
def test_qkv_one_launch(M):
    out, _, _ = _group([("llama2_7b_decode", n, False) for n in ("q", "k", "v")], M)
    for got, ref in out:
        assert_parity(got, ref, 1e-2)


@pytest.mark.parametrize("M", [1, 4])
def test_gate_up_one_launch(M):
    out, _, _ = _group([("llama2_7b_decode", "gate", True), ("llama2_7b_decode", "up", False)], M)
    for got, ref in out:
        assert_parity(got, ref, 1e-2)


@pytest.mark.parametrize("M", [17, 33, 64])
def test_mixed_shapes_every_tile_width(M):
    """q (4096 -> 4096) with gate (4096 -> 11008) and the 256 x 256 layer on its own input:
    different row-tile counts per phase in one launch, 32- and 64-token tiles."""
    out, _, _ = _group([("llama2_7b_decode", "q", True), ("llama2_7b_decode", "gate", False),
                        ("single256", "single", True)], M)
    for got, ref in out:
        assert_parity(got, ref, 1e-2)


def test_four_layers():
    out, _, _ = _group([("llama2_7b_decode", n, n == "o") for n in ("q", "k", "v", "o")], 16)
    for got, ref in out:
        assert_parity(got, ref, 1e-2)


@pytest.mark.parametrize("budget", [1, 7, 76])
def test_group_under_an_sm_budget(budget):
    out, _, _ = _group([("single256", "single", True), ("vit_b16_mlp", "fc2", False)], 16,
                       max_sms=budget)
    for got, ref in out:
        assert_parity(got, ref, 1e-2)


def test_larger_batches_run_the_layers_in_turn():
    out, _, _ = _group([("llama2_7b_decode", n, n == "k") for n in ("q", "k", "v")], 200)
    for got, ref in out:
        assert_parity(got, ref, 1e-2)


def test_workspace_shared_with_single_calls_and_repeatable():
    specs = [("llama2_7b_decode", "q", False), ("llama2_7b_decode", "down", True)]
    out1, layers, ws = _group(specs, 16)
    # a single-layer call on the same workspace, then the group again
    D = DeviceLayer(oracle_layer("single256", "single"), BF16)
    X = activations("single256", "single", 8)
    got = D.forward(X, True, ws=ws)
    assert_parity(got, reference(D.L, X, True), 1e-2)
    out2, _, _ = _group(specs, 16, ws=ws)
    for (a, ref), (b, _) in zip(out1, out2):
        np.testing.assert_array_equal(a, b)        # fixed-order reductions: bitwise repeatable
        assert_parity(a, ref, 1e-2)


def test_group_refusals_launch_nothing():
    L = oracle_layer("single256", "single")
    D = DeviceLayer(L, BF16)
    x = torch.from_numpy(activations("single256", "single", 8)).to(DEV, BF16)
    y = torch.full((8, L.d_out), 5.0, dtype=BF16, device=DEV)
    y2 = torch.full((8, L.d_out), 5.0, dtype=BF16, device=DEV)
    one = fq.Layer(x, L.d_in, D.T_in, D.C, D.T_out_t, L.d_out, None, y)
    nb = fq.fq_group_workspace_bytes(8, [one, one])
    ws = torch.zeros(nb, dtype=torch.uint8, device=DEV)

    def status(layers, **kw):
        with pytest.raises(fq.FrameQuantError) as e:
            fq.fq_linear_forward_group(8, layers, ws, kw.get("nb", nb))
        return e.value.status

    assert status([one, one]) == 1                                  # two layers, one output
    assert status([one, fq.Layer(y, L.d_in, D.T_in, D.C, D.T_out_t, L.d_out, None, y2)]) == 1
    assert status([one] * 5) == 1                                   # above FQ_MAX_GROUP
    two = fq.Layer(x, L.d_in, D.T_in, D.C, D.T_out_t, L.d_out, None, y2)
    assert status([one, two], nb=nb - 256) == 4
    torch.cuda.synchronize()
    assert (y == 5.0).all() and (y2 == 5.0).all()
