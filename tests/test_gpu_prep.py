"""Offline preparation on the GPU (fq_frame_build, fq_coefficients, fq_quantize_rtn) against
the fp64 oracle on the same seeded draws."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2403_06082_gb300 as fq  # noqa: E402
import workloads as wl  # noqa: E402
from oracle import frames, quant  # noqa: E402

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def build_frame(k, rho, d, draws=None):
    a, b = (draws.a, draws.b) if draws is not None else (0, 0)
    nb = fq.fq_frame_workspace_bytes(k, rho, d, a, b)
    ws = torch.empty(nb, dtype=torch.uint8, device=DEV)
    T = torch.empty(k * rho, d, dtype=torch.float32, device=DEV)
    rot = None if draws is None else (a, b, draws.ga, draws.gb, draws.perm, draws.signs)
    fq.fq_frame_build(k, rho, d, rot, T, ws, nb)
    return T


@pytest.mark.parametrize("k,rho,d", [(18, 16, 256), (53, 16, 768), (282, 16, 4096), (5, 8, 22),
                                     (7, 8, 48), (1, 48, 48)])
@pytest.mark.parametrize("rotate", [False, True])
def test_frame_build_matches_oracle(k, rho, d, rotate):
    draws = wl.rotation_draws(21, "prep", str(k), d=d) if rotate else None
    got = build_frame(k, rho, d, draws).double().cpu().numpy()
    ref = frames.frame(k, rho, d, draws)
    assert np.abs(got - ref).max() <= 2e-6
    # tight: T^T T = I in fp32
    G = got.T @ got
    assert np.abs(G - np.eye(d)).max() <= 1e-5


def test_frame_build_rejects_invalid_triple():
    nb = fq.fq_frame_workspace_bytes(10, 16, 256)
    ws = torch.empty(nb, dtype=torch.uint8, device=DEV)
    T = torch.empty(160, 256, device=DEV)
    with pytest.raises(fq.FrameQuantError) as e:
        fq.fq_frame_build(10, 16, 256, None, T, ws, nb)
    assert e.value.status == 1


@pytest.mark.parametrize("wl_key,name", [("single256", "single"), ("vit_b16_mlp", "fc1")])
def test_coefficients_and_rtn_match_oracle(wl_key, name):
    wk = wl.WORKLOADS[wl_key]
    layer = next(l for l in wk.layers if l.name == name)
    from oracle import layer as olayer
    L = olayer.from_workload(wl_key, name)
    W = torch.from_numpy(L.W).to(DEV, torch.float32)
    T_in = torch.from_numpy(L.T_in).to(DEV, torch.float32)
    T_out = torch.from_numpy(L.T_out).to(DEV, torch.float32)
    C = torch.empty(L.n_out, L.n_in, dtype=torch.float32, device=DEV)
    nb = fq.fq_coefficients_workspace_bytes(layer.d_out, L.n_in)
    ws = torch.empty(nb, dtype=torch.uint8, device=DEV)
    fq.fq_coefficients(W, layer.d_out, layer.d_in, T_in, L.n_in, T_out, L.n_out, C, ws, nb)
    Cg = C.double().cpu().numpy()
    assert np.linalg.norm(Cg - L.C) <= 1e-5 * np.linalg.norm(L.C)

    # RTN on the GPU's C against the oracle's RTN of the same (fp32) values
    codes = torch.empty(L.n_out, L.n_in, dtype=torch.uint8, device=DEV)
    scale = torch.empty(L.n_out, dtype=torch.int16, device=DEV)
    zero = torch.empty(L.n_out, dtype=torch.int16, device=DEV)
    gamma = torch.empty(L.n_out, dtype=torch.float32, device=DEV)
    fq.fq_quantize_rtn(C, L.n_out, L.n_in, codes, scale, zero, gamma)
    q_ref, s_ref, z_ref = quant.rtn(Cg)
    np.testing.assert_array_equal(scale.cpu().numpy().view(np.float16), s_ref)
    np.testing.assert_array_equal(zero.cpu().numpy().view(np.float16), z_ref)
    # codes are unique except within rounding distance of a tie
    t = (Cg - z_ref.astype(np.float64)[:, None]) / s_ref.astype(np.float64)[:, None]
    clear = np.abs(t - np.floor(t) - 0.5) > 1e-5
    q = codes.cpu().numpy()
    np.testing.assert_array_equal(q[clear], q_ref[clear])
    assert np.abs(q.astype(int) - q_ref).max() <= 1
    np.testing.assert_allclose(gamma.cpu().numpy(), quant.wiener_gain(Cg, s_ref), rtol=1e-5)
