"""Activation rounding in the frame domain (Appendix F; mode FQ_BF16 | FQ_ACT_BITS(N)) through
the C ABI against the oracle (oracle.actquant).

The integer decision z -> zbar is taken from z = T_in x, which the GPU accumulates in fp32 from
bf16 x and bf16 T_in; the oracle takes it in the same precision up to rounding order (fp64 sums
of the same bf16 products), so the two can only differ where z / Delta lies within ~1e-5 of a
half-integer.  One test reads zbar back exactly (identity codes and an identity output frame
make y = bf16(Delta zbar)); the others check whole layers at the workloads' sizes, and that the
rounding really happened (at 4 bits the result is far from the unrounded layer)."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2403_06082_gb300 as fq  # noqa: E402
import workloads as wl  # noqa: E402
from fqgpu import DEV, DeviceLayer, activations, assert_parity, oracle_layer, rel_frobenius  # noqa: E402
from oracle import actquant, forward  # noqa: E402

pytestmark = pytest.mark.gpu
BF16 = torch.bfloat16


def _bf16(a):
    return wl.round_bf16(np.asarray(a, dtype=np.float32)).astype(np.float64)


def _run(D, X, bits, use_gamma=False, ws=None):
    L = D.L
    M = X.shape[0]
    mode = fq.FQ_BF16 | fq.FQ_ACT_BITS(bits)
    x = torch.from_numpy(X).to(DEV, BF16)
    y = torch.full((M, L.d_out), float("nan"), dtype=BF16, device=DEV)
    nb = fq.fq_workspace_bytes(M, L.d_in, L.n_in, L.n_out, L.d_out, mode)
    if ws is None:
        ws = torch.zeros(nb, dtype=torch.uint8, device=DEV)
    fq.fq_linear_forward(x, M, L.d_in, D.T_in, D.C, D.T_out_t, L.d_out,
                         D.gamma if use_gamma else None, y, ws, nb, mode)
    assert fq.fq_check(ws) == 0
    return y.double().cpu().numpy(), ws


def _oracle(L, X, bits, use_gamma=False):
    """The rounded layer with the decision taken from bf16 T_in (the kernel's operand)."""
    return actquant.layer_forward_actquant(X, _bf16(L.T_in), L.codes, L.scale, L.zero, L.T_out,
                                           L.gamma if use_gamma else None, bits)


class _IdentityLayer:
    """n_in = 288 frame coefficients of the 256-wide input frame, codes q_ii = 1 (else 0),
    scale 1, zero 0, and the trivial output frame T_out = I (d_out = n_out = 288): then
    u = Delta zbar and y = bf16(Delta zbar)."""

    def __init__(self):
        base = oracle_layer("single256", "single")
        n = base.n_in
        self.T_in = base.T_in
        self.T_out = np.eye(n)
        self.codes = np.eye(n, dtype=np.uint8)
        self.scale = np.ones(n, np.float16)
        self.zero = np.zeros(n, np.float16)
        self.gamma = np.ones(n, np.float32)
        self.d_in, self.d_out, self.n_in, self.n_out = base.d_in, n, n, n


@pytest.mark.parametrize("bits", [2, 4, 8])
@pytest.mark.parametrize("M", [8, 200, 300])
def test_rounded_integers_read_back_exactly(bits, M):
    L = _IdentityLayer()
    D = DeviceLayer(L, BF16)
    X = activations("single256", "single", M)
    got, _ = _run(D, X, bits)
    Z = X.astype(np.float64) @ _bf16(L.T_in).T
    Zbar, delta = actquant.quantize_ff(Z, bits)
    back = np.rint(got / delta)
    frac = np.abs(Z / delta - np.floor(Z / delta) - 0.5)      # distance of z / Delta to a tie
    mismatch = back != Zbar
    assert not (mismatch & (frac > 1e-4)).any(), np.argwhere(mismatch & (frac > 1e-4))[:5]
    assert mismatch.mean() < 1e-3
    assert np.abs(back).max() == (1 << (bits - 1)) - 1


@pytest.mark.parametrize("name", ["fc1", "fc2"])
def test_vit_mlp_int8_full_batch_sampled(name):
    """The paper's setting for activation rounding (ViT-B/16, Appendix F), 12608 tokens: the
    step is the maximum over the whole batch, so the oracle computes every token's z."""
    L = oracle_layer("vit_b16_mlp", name)
    D = DeviceLayer(L, BF16)
    X = activations("vit_b16_mlp", name, 12608)
    got, _ = _run(D, X, 8)
    Z = X.astype(np.float64) @ _bf16(L.T_in).T
    Zbar, delta = actquant.quantize_ff(Z, 8)
    rows = np.sort(wl.rng(1, "aq-sample", name).choice(12608, 48, replace=False))
    U = forward.core(delta * Zbar[rows].astype(np.float64), L.codes, L.scale, L.zero)
    assert_parity(got[rows], forward.synthesis(L.T_out, U), 1e-2)


@pytest.mark.parametrize("M,use_gamma", [(16, True), (1, False), (300, True)])
def test_llama7b_q_int8(M, use_gamma):
    L = oracle_layer("llama2_7b_decode", "q")
    D = DeviceLayer(L, BF16)
    X = activations("llama2_7b_decode", "q", M)
    got, _ = _run(D, X, 8, use_gamma)
    Y, _, _, _ = _oracle(L, X, 8, use_gamma)
    assert_parity(got, Y, 1e-2)


def test_four_bits_is_the_rounded_layer_not_the_plain_one():
    L = oracle_layer("llama2_7b_prefill", "q")
    D = DeviceLayer(L, BF16)
    X = activations("llama2_7b_prefill", "q", 256)
    got, _ = _run(D, X, 4)
    Y, _, _, _ = _oracle(L, X, 4)
    plain = forward.layer_forward(X, L.T_in, L.codes, L.scale, L.zero, L.T_out)
    assert_parity(got, Y, 1e-2)
    assert rel_frobenius(got, plain) > 5e-2          # 4-bit rounding moves the output


def test_workspace_alternating_with_plain_calls_is_repeatable():
    L = oracle_layer("single256", "single")
    D = DeviceLayer(L, BF16)
    X = activations("single256", "single", 100)
    a, ws = _run(D, X, 8, True)
    D.forward(activations("single256", "single", 16), True, ws=ws)     # decode kernel
    b, _ = _run(D, X, 8, True, ws=ws)
    np.testing.assert_array_equal(a, b)              # the maximum was reset for the next call
    Y, _, _, _ = _oracle(L, X, 8, True)
    assert_parity(a, Y, 1e-2)
