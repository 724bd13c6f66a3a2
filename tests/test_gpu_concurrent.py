"""fq_linear_forward_sms: independent layers on parallel streams, each on its own SM budget,
against the fp64 oracle (relative Frobenius error <= 1e-2 in FQ_BF16).

q, k and v of the Llama-2-7B block read the same input and are independent, as are gate and
up; with budgets that add up to no more than the device's SMs they run side by side.  Small
budgets (down to one SM) and budgets above the SM count exercise the planner's edges."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2403_06082_gb300 as fq  # noqa: E402
from fqgpu import DEV, DeviceLayer, activations, oracle_layer, reference, assert_parity, rel_frobenius  # noqa: E402

pytestmark = pytest.mark.gpu
BF16 = torch.bfloat16


def _group(wl_key, names, M, budget, use_gamma=False, sample=None):
    """Run `names` concurrently on one stream each, `budget` SMs per call."""
    layers = [oracle_layer(wl_key, n) for n in names]
    devs = [DeviceLayer(L, BF16) for L in layers]
    X = activations(wl_key, names[0], M)
    x = torch.from_numpy(X).to(DEV, BF16)
    ys, wss, streams = [], [], []
    for L in layers:
        ys.append(torch.full((M, L.d_out), float("nan"), dtype=BF16, device=DEV))
        nb = fq.fq_workspace_bytes(M, L.d_in, L.n_in, L.n_out, L.d_out, 0)
        wss.append((torch.zeros(nb, dtype=torch.uint8, device=DEV), nb))
        streams.append(torch.cuda.Stream())
    torch.cuda.synchronize()
    for L, D, y, (ws, nb), s in zip(layers, devs, ys, wss, streams):
        with torch.cuda.stream(s):
            fq.fq_linear_forward_sms(x, M, L.d_in, D.T_in, D.C, D.T_out_t, L.d_out,
                                     D.gamma if use_gamma else None, y, ws, nb, budget,
                                     stream=s)
    torch.cuda.synchronize()
    for L, y, (ws, _) in zip(layers, ys, wss):
        assert fq.fq_check(ws) == 0
        got = y.double().cpu().numpy()
        Xs = X
        if sample is not None:
            got, Xs = got[sample], X[sample]
        err = assert_parity(got, reference(L, Xs, use_gamma), 1e-2)


def test_qkv_decode_side_by_side():
    _group("llama2_7b_decode", ["q", "k", "v"], 16, 48)


def test_gate_up_decode_side_by_side():
    _group("llama2_7b_decode", ["gate", "up"], 4, 72, use_gamma=True)


def test_qkv_prefill_side_by_side():
    rows = sorted({0, 1, 127, 128, 255, 256, 511})
    _group("llama2_7b_decode", ["q", "k", "v"], 512, 48, sample=rows)


@pytest.mark.parametrize("M", [16, 64, 300])
@pytest.mark.parametrize("budget", [1, 3, 5, 8, 100000])
def test_budget_edges(M, budget):
    L = oracle_layer("single256", "single")
    D = DeviceLayer(L, BF16)
    X = activations("single256", "single", M)
    x = torch.from_numpy(X).to(DEV, BF16)
    y = torch.full((M, L.d_out), float("nan"), dtype=BF16, device=DEV)
    nb = fq.fq_workspace_bytes(M, L.d_in, L.n_in, L.n_out, L.d_out, 0)
    ws = torch.zeros(nb, dtype=torch.uint8, device=DEV)
    fq.fq_linear_forward_sms(x, M, L.d_in, D.T_in, D.C, D.T_out_t, L.d_out, D.gamma, y, ws, nb,
                             budget)
    assert fq.fq_check(ws) == 0
    assert_parity(y.double().cpu().numpy(), reference(L, X, True), 1e-2)


def test_budget_fp32_debug_and_negative():
    L = oracle_layer("single256", "single")
    D = DeviceLayer(L, torch.float32)
    M = 8
    X = activations("single256", "single", M)
    x = torch.from_numpy(X).to(DEV, torch.float32)
    y = torch.full((M, L.d_out), 7.0, dtype=torch.float32, device=DEV)
    nb = fq.fq_workspace_bytes(M, L.d_in, L.n_in, L.n_out, L.d_out, fq.FQ_FP32_DEBUG)
    ws = torch.zeros(nb, dtype=torch.uint8, device=DEV)
    with pytest.raises(fq.FrameQuantError) as e:
        fq.fq_linear_forward_sms(x, M, L.d_in, D.T_in, D.C, D.T_out_t, L.d_out, None, y, ws, nb,
                                 -1, mode=fq.FQ_FP32_DEBUG)
    assert e.value.status == 1
    torch.cuda.synchronize()
    assert (y == 7.0).all()
    fq.fq_linear_forward_sms(x, M, L.d_in, D.T_in, D.C, D.T_out_t, L.d_out, None, y, ws, nb, 2,
                             mode=fq.FQ_FP32_DEBUG)
    assert fq.fq_check(ws) == 0
    assert_parity(y.double().cpu().numpy(), reference(L, X, False), 1e-5)
    assert np.isfinite(y.cpu().numpy()).all()


def test_l2_prefetch_hint_changes_nothing():
    """The chaining hint (the next layer's T_in) only warms L2: outputs are bitwise equal."""
    Lq, Lk = oracle_layer("llama2_7b_decode", "q"), oracle_layer("llama2_7b_decode", "k")
    Dq, Dk = DeviceLayer(Lq, BF16), DeviceLayer(Lk, BF16)
    X = activations("llama2_7b_decode", "q", 16)
    x = torch.from_numpy(X).to(DEV, BF16)
    nb = fq.fq_workspace_bytes(16, Lq.d_in, Lq.n_in, Lq.n_out, Lq.d_out, 0)
    ws = torch.zeros(nb, dtype=torch.uint8, device=DEV)
    outs = []
    for hint in (None, Dk.T_in, Dk.T_in[:1000]):
        y = torch.full((16, Lq.d_out), float("nan"), dtype=BF16, device=DEV)
        fq.fq_linear_forward_ex(x, 16, Lq.d_in, Dq.T_in, Dq.C, Dq.T_out_t, Lq.d_out, None, y, ws,
                                nb, prefetch=hint)
        assert fq.fq_check(ws) == 0
        outs.append(y.cpu())
    assert torch.equal(outs[0], outs[1]) and torch.equal(outs[0], outs[2])
    assert_parity(outs[0].double().numpy(), reference(Lq, X, False), 1e-2)
