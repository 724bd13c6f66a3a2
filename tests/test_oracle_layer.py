"""Pins for the oracle's layer forward: exact recovery, brute force on a d = 16 layer, the
trivial frame, and the noise-robustness law of the paper (Sec. 2.1 Example 1 noise remark,
Sec. 3.1 (a), Sec. 3.2)."""
import math

import numpy as np
import pytest

import workloads as wl
from oracle import forward, frames, layer, quant


def test_exact_recovery_single256():
    L = layer.from_workload("single256", "single")
    X = wl.activations(wl.WORKLOADS["single256"], wl.WORKLOADS["single256"].layers[0], 8)
    Y = forward.synthesis(L.T_out, forward.analysis(L.T_in, X) @ L.C.T)
    ref = X.astype(np.float64) @ L.W.T
    assert np.abs(Y - ref).max() <= 1e-10 * np.abs(ref).max()


@pytest.mark.parametrize("name", ["fc1", "fc2"])
def test_exact_recovery_vit(name):
    L = layer.from_workload("vit_b16_mlp", name)
    wk = wl.WORKLOADS["vit_b16_mlp"]
    X = wl.activations(wk, next(l for l in wk.layers if l.name == name), 64)
    Y = forward.synthesis(L.T_out, forward.analysis(L.T_in, X) @ L.C.T)
    ref = X.astype(np.float64) @ L.W.T
    assert np.linalg.norm(Y - ref) <= 1e-10 * np.linalg.norm(ref)


def test_bruteforce_d16_layer():
    """Scalar sums over subspaces, basis vectors and codes against the matrix form."""
    d_in = d_out = 16
    k, rho = 5, 4                                  # w = 4 <= k: valid, r = 1.25
    W = wl.rng(11, "bf16").standard_normal((d_out, d_in))
    dr_in = wl.rotation_draws(11, "in", d=d_in)
    dr_out = wl.rotation_draws(11, "out", d=d_out)
    L = layer.build(W, k, k, rho, rot_in=dr_in, rot_out=dr_out)
    x = wl.round_bf16(wl.rng(11, "x").standard_normal(d_in)).astype(np.float64)
    Pin, Pout = L.T_in.T, L.T_out.T                # synthesis operators d x n (columns = basis)
    # subspace i, basis index b -> column i * rho + b of P (rows of T are ordered (j, k_i, re/im))
    def col(i, b):
        j, e = divmod(b, 2)
        return 2 * (j * k + i) + e
    y = [0.0] * d_out
    for jo in range(d_out):
        acc = 0.0
        for i_o in range(k):
            for b_o in range(rho):
                ro = col(i_o, b_o)
                u = 0.0
                for i_i in range(k):
                    for b_i in range(rho):
                        ci = col(i_i, b_i)
                        zc = sum(Pin[l, ci] * x[l] for l in range(d_in))
                        chat = float(L.scale[ro]) * int(L.codes[ro, ci]) + float(L.zero[ro])
                        u += chat * zc
                acc += Pout[jo, ro] * float(L.gamma[ro]) * u
        y[jo] = acc
    Ym = forward.layer_forward(x[None, :], L.T_in, L.codes, L.scale, L.zero, L.T_out, L.gamma)
    np.testing.assert_allclose(Ym[0], y, rtol=1e-12, atol=1e-12)


def test_trivial_frame_is_plain_rtn_gemm():
    """k = 1, rho = d, no rotation: T = I, so the layer is an RTN-quantized GEMM of W itself."""
    W = wl.rng(12, "triv").standard_normal((24, 40))
    L = layer.build(W, 1, 1)
    np.testing.assert_array_equal(L.T_in, np.eye(40))
    np.testing.assert_array_equal(L.C, W)
    X = wl.round_bf16(wl.rng(12, "tx").standard_normal((3, 40)))
    What = L.scale.astype(np.float64)[:, None] * L.codes + L.zero.astype(np.float64)[:, None]
    Y = forward.layer_forward(X, L.T_in, L.codes, L.scale, L.zero, L.T_out)
    np.testing.assert_allclose(Y, X.astype(np.float64) @ What.T, rtol=1e-13, atol=1e-13)


@pytest.mark.parametrize("k,reduction", [(3, 0.33), (4, 0.50)])
def test_noise_example_one_over_r(golden, k, reduction):
    """Example 1's noise remark: with white noise at 10 dB SNR on the coefficients, the MSE of
    the reconstruction falls by 33% at r = 1.5 and 50% at r = 2 relative to r = 1 (an
    orthonormal basis); for a Parseval frame the ratio is exactly 1/r (Sec. 3.1 (a))."""
    g = golden("example1.json")["noise_example"]
    assert [k * 2 / 4, reduction] in g["mse_reduction"]
    rng = wl.rng(13, "noise", str(k))
    trials = 20000

    def mse(kk):
        T = frames.tff_analysis(kk, 2, 4)
        X = rng.standard_normal((trials, 4))
        Z = X @ T.T
        sig = (Z ** 2).mean()
        noise = rng.standard_normal(Z.shape) * math.sqrt(sig / 10 ** (g["snr_db"] / 10))
        return (((Z + noise) @ T - X) ** 2).mean()
    ratio = mse(k) / mse(2)
    assert ratio == pytest.approx(2 / k, rel=0.03)
    assert 1 - ratio == pytest.approx(reduction, abs=0.02)


def test_filter_identity_and_shrinkage():
    L = layer.from_workload("single256", "single")
    X = wl.activations(wl.WORKLOADS["single256"], wl.WORKLOADS["single256"].layers[0], 8)
    one = np.ones(L.n_out, np.float32)
    np.testing.assert_array_equal(
        forward.layer_forward(X, L.T_in, L.codes, L.scale, L.zero, L.T_out, one),
        forward.layer_forward(X, L.T_in, L.codes, L.scale, L.zero, L.T_out))
    # on Gaussian weights the shrinkage lowers the error against W x (expected, not guaranteed)
    ref = X.astype(np.float64) @ L.W.T
    e0 = np.linalg.norm(forward.layer_forward(X, L.T_in, L.codes, L.scale, L.zero, L.T_out) - ref)
    e1 = np.linalg.norm(forward.layer_forward(X, L.T_in, L.codes, L.scale, L.zero, L.T_out,
                                              L.gamma) - ref)
    assert e1 < e0


def test_redundancy_lowers_quantization_error():
    """More redundancy, less error after 2-bit quantization (the paper's Table 8 trend, on
    synthetic Gaussian weights)."""
    W = wl.rng(14, "red").standard_normal((256, 256)) / 16
    X = wl.round_bf16(wl.rng(14, "redx").standard_normal((32, 256)))
    ref = X.astype(np.float64) @ W.T
    errs = []
    for k in (16, 24, 32):                          # r = 1, 1.5, 2
        L = layer.build(W, k, k, rot_in=wl.rotation_draws(14, "i", d=256),
                        rot_out=wl.rotation_draws(14, "o", d=256))
        Y = forward.layer_forward(X, L.T_in, L.codes, L.scale, L.zero, L.T_out)
        errs.append(np.linalg.norm(Y - ref) / np.linalg.norm(ref))
    assert errs[0] > errs[1] > errs[2]


def test_round_bf16_matches_the_format():
    """The oracle's bfloat16 rounding against torch's conversion (a library routine) on values
    that exercise ties, carries into the exponent, subnormals and signs."""
    torch = pytest.importorskip("torch")
    from oracle.forward import round_bf16
    vals = np.array([1.0, 1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8, 1.0 + 2.0 ** -9, -3.14159,
                     2.0 - 2.0 ** -9, 255.9, 1e-40, -1e-38, 65504.0, 0.0, -0.0], dtype=np.float64)
    g = np.random.default_rng(3)
    vals = np.concatenate([vals, g.standard_normal(2000) * 10.0 ** g.integers(-6, 6, 2000)])
    want = torch.from_numpy(vals.astype(np.float32)).to(torch.bfloat16).double().numpy()
    got = round_bf16(vals)
    assert np.array_equal(got.view(np.uint64), want.view(np.uint64))
    assert round_bf16(np.array([1.0 + 2.0 ** -8]))[0] == 1.0          # a tie goes to even
    assert round_bf16(np.array([1.0 + 3 * 2.0 ** -8]))[0] == 1.0 + 2.0 ** -6


def test_bf16_operand_diagnostic():
    """The diagnostic forward equals the exact one when the frames are exact in bfloat16 (the
    trivial frame without rotation is the identity), and otherwise differs by about the
    operands' rounding (bf16 keeps 8 significant bits)."""
    from oracle import forward, frames
    g = np.random.default_rng(11)
    d, M = 64, 5
    W = g.standard_normal((d, d)) / 8.0
    X = g.standard_normal((M, d))
    T = frames.frame(1, d, d, None)
    C = T @ W @ T.T
    codes, scale, zero = quant.rtn(C)
    exact = forward.layer_forward(X, T, codes, scale, zero, T)
    diag = forward.layer_forward_bf16_operands(X, T, codes, scale, zero, T)
    assert np.array_equal(exact, diag)
    L = layer.from_workload("single256", "single")
    Xs = g.standard_normal((M, L.d_in))
    exact = forward.layer_forward(Xs, L.T_in, L.codes, L.scale, L.zero, L.T_out)
    diag = forward.layer_forward_bf16_operands(Xs, L.T_in, L.codes, L.scale, L.zero, L.T_out)
    rel = np.linalg.norm(diag - exact) / np.linalg.norm(exact)
    assert 1e-5 < rel < 1e-2
