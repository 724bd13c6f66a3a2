"""fq_linear_forward_implicit (frames in structured form) through the C ABI against the fp64
oracle: relative Frobenius error <= 1e-2, the FQ_BF16 bound (z and u are rounded to bf16).

The oracle layers are the dense ones of the other parity tests (oracle.layer, T built densely
from the same rotation draws); the structured form has to reproduce the same layer.  For the
Llama-2-70B shapes the oracle applies the frames in structured form (oracle.frames, pinned
against the dense construction) with seeded uniform codes, as in test_gpu_llama70b."""
from fractions import Fraction

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2403_06082_gb300 as fq  # noqa: E402
import workloads as wl  # noqa: E402
from fqgpu import DEV, DeviceLayer, activations, oracle_layer, reference, assert_parity, rel_frobenius  # noqa: E402
from oracle import forward, frames  # noqa: E402

pytestmark = pytest.mark.gpu
BF16 = torch.bfloat16
RHO = 16


def _draws(wl_key, name, side, d):
    wk = wl.WORKLOADS[wl_key]
    dr = wl.rotation_draws(wk.seed, wk.key, name, side, d=d)
    return (dr.a, dr.b, dr.ga, dr.gb, dr.perm, dr.signs)


def _frames(wl_key, name, L, rotate=True):
    """The oracle layer's frames (same seeded rotation draws) in structured form."""
    Fi = fq.fq_frame_implicit(L.k_in, RHO, L.d_in,
                              _draws(wl_key, name, "in", L.d_in) if rotate else None, DEV)
    Fo = fq.fq_frame_implicit(L.k_out, RHO, L.d_out,
                              _draws(wl_key, name, "out", L.d_out) if rotate else None, DEV)
    return Fi, Fo


def _run(X, Fi, C, Fo, gamma, d_out, ws=None, max_sms=0):
    M = X.shape[0]
    x = torch.from_numpy(X).to(DEV, BF16)
    y = torch.full((M, d_out), float("nan"), dtype=BF16, device=DEV)
    nb = fq.fq_implicit_workspace_bytes(M, Fi.d, Fi.n, Fo.n, Fo.d)
    if ws is None:
        ws = torch.zeros(nb, dtype=torch.uint8, device=DEV)
    fq.fq_linear_forward_implicit(x, M, Fi, C, Fo, gamma, y, ws, nb, max_sms)
    st = fq.fq_check(ws)
    assert st == 0, fq.fq_status_str(st)
    return y.double().cpu().numpy()


def _check(wl_key, name, M, use_gamma, rotate=True, tol=1e-2):
    L = oracle_layer(wl_key, name, rotate=rotate)
    D = DeviceLayer(L, BF16)
    Fi, Fo = _frames(wl_key, name, L, rotate)
    X = activations(wl_key, name, M)
    got = _run(X, Fi, D.C, Fo, D.gamma if use_gamma else None, L.d_out)
    err = assert_parity(got, reference(L, X, use_gamma), tol)
    return got


@pytest.mark.parametrize("M", [1, 8, 17, 64])
@pytest.mark.parametrize("use_gamma", [False, True])
def test_single256(M, use_gamma):
    _check("single256", "single", M, use_gamma)


def test_single256_without_rotation():
    _check("single256", "single", 8, True, rotate=False)


@pytest.mark.parametrize("name", ["fc1", "fc2"])
def test_vit_shapes(name):
    _check("vit_b16_mlp", name, 40, False)


@pytest.mark.parametrize("name", ["q", "gate", "down"])
@pytest.mark.parametrize("M", [1, 16])
def test_llama7b_decode(name, M):
    _check("llama2_7b_decode", name, M, name == "gate")


def test_matches_dense_path():
    """Both forms of the same layer on the GPU agree to within bf16 rounding of z and u."""
    L = oracle_layer("llama2_7b_decode", "q")
    D = DeviceLayer(L, BF16)
    Fi, Fo = _frames("llama2_7b_decode", "q", L)
    X = activations("llama2_7b_decode", "q", 16)
    dense = D.forward(X)
    got = _run(X, Fi, D.C, Fo, None, L.d_out)
    assert_parity(got, dense, 1e-2)


def test_workspace_reuse_and_budget():
    """One workspace across shapes and calls, the dense path sharing it, and an SM budget."""
    La = oracle_layer("single256", "single")
    Lb = oracle_layer("llama2_7b_decode", "down")
    Da, Db = DeviceLayer(La, BF16), DeviceLayer(Lb, BF16)
    Fa, Fb = _frames("single256", "single", La), _frames("llama2_7b_decode", "down", Lb)
    nb = max(fq.fq_implicit_workspace_bytes(16, Lb.d_in, Lb.n_in, Lb.n_out, Lb.d_out),
             fq.fq_workspace_bytes(16, Lb.d_in, Lb.n_in, Lb.n_out, Lb.d_out, 0))
    ws = torch.zeros(nb, dtype=torch.uint8, device=DEV)
    Xa = activations("single256", "single", 16)
    Xb = activations("llama2_7b_decode", "down", 16)
    ya1 = _run(Xa, Fa[0], Da.C, Fa[1], Da.gamma, La.d_out, ws)
    yb1 = _run(Xb, Fb[0], Db.C, Fb[1], None, Lb.d_out, ws, max_sms=60)
    Db.forward(Xb, ws=ws)
    ya2 = _run(Xa, Fa[0], Da.C, Fa[1], Da.gamma, La.d_out, ws)
    np.testing.assert_array_equal(ya1, ya2)
    assert_parity(ya1, reference(La, Xa, True), 1e-2)
    assert_parity(yb1, reference(Lb, Xb, False), 1e-2)


@pytest.mark.parametrize("name,M", [("q", 16), ("gate", 1), ("down", 16)])
def test_llama70b_shapes(name, M):
    wk = wl.WORKLOADS["llama2_70b"]
    layer = next(l for l in wk.layers if l.name == name)
    r = Fraction(11, 10)
    k_in, _ = frames.choose_k(r, layer.d_in, RHO)
    k_out, _ = frames.choose_k(r, layer.d_out, RHO)
    n_in, n_out = k_in * RHO, k_out * RHO
    dr_in = wl.rotation_draws(wk.seed, wk.key, name, "in", d=layer.d_in)
    dr_out = wl.rotation_draws(wk.seed, wk.key, name, "out", d=layer.d_out)
    codes = wl.random_codes(wk.seed, wk.key, name, n_out=n_out, n_in=n_in)
    scale, zero = wl.random_scale_zero(wk.seed, wk.key, name, n_out=n_out, mag=0.01)
    X = wl.activations(wk, layer, M)
    Fi = fq.fq_frame_implicit(k_in, RHO, layer.d_in,
                              (dr_in.a, dr_in.b, dr_in.ga, dr_in.gb, dr_in.perm, dr_in.signs), DEV)
    Fo = fq.fq_frame_implicit(k_out, RHO, layer.d_out,
                              (dr_out.a, dr_out.b, dr_out.ga, dr_out.gb, dr_out.perm,
                               dr_out.signs), DEV)
    words = torch.zeros(fq.fq_packed_words(n_out, n_in), dtype=torch.int32, device=DEV)
    C = fq.fq_pack(torch.from_numpy(codes).to(DEV), torch.from_numpy(scale.view(np.int16)).to(DEV),
                   torch.from_numpy(zero.view(np.int16)).to(DEV), n_out, n_in, words)
    got = _run(X, Fi, C, Fo, None, layer.d_out)
    Z = frames.analysis_apply(k_in, RHO, layer.d_in, dr_in, X)
    U = forward.core(Z, codes, scale, zero)
    ref = frames.synthesis_apply(k_out, RHO, layer.d_out, dr_out, U)
    err = assert_parity(got, ref, 1e-2)


def test_errors_launch_nothing():
    L = oracle_layer("single256", "single")
    D = DeviceLayer(L, BF16)
    Fi, Fo = _frames("single256", "single", L)
    M = 65
    x = torch.zeros(M, L.d_in, dtype=BF16, device=DEV)
    y = torch.full((M, L.d_out), 7.0, dtype=BF16, device=DEV)
    nb = fq.fq_implicit_workspace_bytes(64, L.d_in, L.n_in, L.n_out, L.d_out)
    ws = torch.zeros(nb, dtype=torch.uint8, device=DEV)
    with pytest.raises(fq.FrameQuantError) as e:
        fq.fq_linear_forward_implicit(x, M, Fi, D.C, Fo, None, y, ws, nb)
    assert e.value.status == 3                      # M > 64: decode batches only
    nb8 = fq.fq_implicit_workspace_bytes(8, L.d_in, L.n_in, L.n_out, L.d_out)
    with pytest.raises(fq.FrameQuantError) as e:
        fq.fq_linear_forward_implicit(x, 8, Fo, D.C, Fi, None, y, ws, nb8 - 1)
    assert e.value.status == 4
    with pytest.raises(fq.FrameQuantError):
        fq.fq_frame_implicit(15, RHO, 256, None, DEV)   # k < d / rho: not tight
    torch.cuda.synchronize()
    assert (y == 7.0).all()


def _run_group(specs, M, max_sms=0):
    """specs: [(workload, layer name, use_gamma, rotate)] in one fq_linear_forward_implicit_group
    call; returns [(got, oracle)] per layer."""
    keep, layers, out = [], [], []
    for wl_key, name, use_gamma, rotate in specs:
        L = oracle_layer(wl_key, name, rotate=rotate)
        D = DeviceLayer(L, BF16)
        Fi, Fo = _frames(wl_key, name, L, rotate)
        X = activations(wl_key, name, M)
        x = torch.from_numpy(X).to(DEV, BF16)
        y = torch.full((M, L.d_out), float("nan"), dtype=BF16, device=DEV)
        keep.append((D, Fi, Fo, x))
        layers.append(fq.ImplicitLayer(x, Fi, D.C, Fo, D.gamma if use_gamma else None, y))
        out.append((L, X, use_gamma, y))
    nb = fq.fq_implicit_group_workspace_bytes(M, layers)
    assert nb > 0
    ws = torch.zeros(nb, dtype=torch.uint8, device=DEV)
    fq.fq_linear_forward_implicit_group(M, layers, ws, nb, max_sms)
    assert fq.fq_check(ws) == 0
    return [(y.double().cpu().numpy(), reference(L, X, g)) for L, X, g, y in out]


@pytest.mark.parametrize("M", [1, 16])
def test_group_qkv(M):
    for got, ref in _run_group([("llama2_7b_decode", n, False, True) for n in ("q", "k", "v")], M):
        assert_parity(got, ref, 1e-2)


def test_group_gate_up_and_mixed():
    for got, ref in _run_group([("llama2_7b_decode", "gate", True, True),
                                ("llama2_7b_decode", "up", False, True)], 4):
        assert_parity(got, ref, 1e-2)
    # different widths, one layer without rotation, and a budget
    for got, ref in _run_group([("single256", "single", True, False),
                                ("llama2_7b_decode", "down", False, True),
                                ("vit_b16_mlp", "fc1", True, True)], 33, max_sms=100):
        assert_parity(got, ref, 1e-2)


def test_group_refusals():
    L = oracle_layer("single256", "single")
    D = DeviceLayer(L, BF16)
    Fi, Fo = _frames("single256", "single", L)
    x = torch.zeros(8, L.d_in, dtype=BF16, device=DEV)
    y = torch.zeros(8, L.d_out, dtype=BF16, device=DEV)
    one = fq.ImplicitLayer(x, Fi, D.C, Fo, None, y)
    nb = fq.fq_implicit_group_workspace_bytes(8, [one, one])
    ws = torch.zeros(nb, dtype=torch.uint8, device=DEV)
    with pytest.raises(fq.FrameQuantError) as e:
        fq.fq_linear_forward_implicit_group(8, [one, one], ws, nb)      # one output twice
    assert e.value.status == 1
    assert fq.fq_implicit_group_workspace_bytes(65, [one]) == 0         # decode batches only


@pytest.mark.parametrize("d,a,b", [
    (512, 16, 32),     # B staged whole with asynchronous copies (b <= 128, b % 4 == 0)
    (160, 16, 10),     # B staged whole with plain loads (b % 4 != 0)
    (2176, 16, 136),   # B streamed in chunks with asynchronous copies (b > 128)
    (2080, 16, 130),   # B streamed in chunks with plain loads, a partial last chunk
])
def test_rotation_kernel_paths(d, a, b):
    """Each way the rotation kernel stages its second factor, on square layers whose rotation
    factor pairs select it, against the structured oracle (seeded uniform codes)."""
    k = d // RHO + 1
    n = k * RHO
    key = ("rotation-paths", str(d), str(a))
    dr_in = wl.rotation_draws_ab(7, *key, "in", d=d, a=a, b=b)
    dr_out = wl.rotation_draws_ab(7, *key, "out", d=d, a=a, b=b)
    codes = wl.random_codes(7, *key, n_out=n, n_in=n)
    scale, zero = wl.random_scale_zero(7, *key, n_out=n, mag=0.01)
    M = 17
    X = torch.from_numpy(wl.rng(7, *key, "x").standard_normal((M, d))).to(BF16).double().numpy()
    Fi = fq.fq_frame_implicit(k, RHO, d, (a, b, dr_in.ga, dr_in.gb, dr_in.perm, dr_in.signs), DEV)
    Fo = fq.fq_frame_implicit(k, RHO, d, (a, b, dr_out.ga, dr_out.gb, dr_out.perm, dr_out.signs),
                              DEV)
    words = torch.zeros(fq.fq_packed_words(n, n), dtype=torch.int32, device=DEV)
    C = fq.fq_pack(torch.from_numpy(codes).to(DEV), torch.from_numpy(scale.view(np.int16)).to(DEV),
                   torch.from_numpy(zero.view(np.int16)).to(DEV), n, n, words)
    got = _run(X, Fi, C, Fo, None, d)
    Z = frames.analysis_apply(k, RHO, d, dr_in, X)
    U = forward.core(Z, codes, scale, zero)
    ref = frames.synthesis_apply(k, RHO, d, dr_out, U)
    assert_parity(got, ref, 1e-2)
