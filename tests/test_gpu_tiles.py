"""Tiled frame operands (fq_frame_tile, fq_layer's T_in_tiles / T_out_tiles) through the C ABI.

The layout is checked byte for byte against a numpy statement of it (128 x 64 blocks, row-block
major, 16-byte groups of row r stored in the order g ^ (r mod 8), zero padding) on ragged
shapes.  The forward on tiled frames reads the same values as on row-major frames and runs the
same products in the same order, so its output is compared bit for bit with the row-major
launch, and against the fp64 oracle (relative Frobenius error <= 1e-2 with the elementwise
companion bound)."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2403_06082_gb300 as fq  # noqa: E402
from fqgpu import (DEV, DeviceLayer, activations, assert_parity, oracle_layer,  # noqa: E402
                   reference)

pytestmark = pytest.mark.gpu
BF16 = torch.bfloat16


def _tiles_numpy(T):
    """The tiled layout of a rows x cols uint16 matrix, as uint16, plus the row-tile index."""
    rows, cols = T.shape
    RT, KB = -(-rows // 128), -(-cols // 64)
    P = np.zeros((RT * 128, KB * 64), dtype=np.uint16)
    P[:rows, :cols] = T
    out = np.zeros((RT, KB, 128, 8, 8), dtype=np.uint16)   # [tile][kb][row][stored group][8]
    for r in range(128):
        for g in range(8):
            out[:, :, r, g ^ (r & 7), :] = P.reshape(RT, 128, KB, 8, 8)[:, r, :, g, :]
    idx = np.array([[0, KB, t * KB] for t in range(RT)], dtype=np.int32)
    return out.reshape(-1), idx


def _tile(T):
    rows, cols = T.shape
    nb = fq.fq_frame_tiles_bytes(rows, cols)
    out = torch.full((nb,), 0xA5, dtype=torch.uint8, device=DEV)
    fq.fq_frame_tile(T, rows, cols, out, nb)
    torch.cuda.synchronize()
    return out


@pytest.mark.parametrize("rows,cols", [(1, 8), (130, 72), (300, 200), (4512, 4096)])
def test_layout_byte_for_byte(rows, cols):
    g = np.random.default_rng(rows * 7 + cols)
    T = torch.from_numpy(g.standard_normal((rows, cols)).astype(np.float32)).to(DEV, BF16)
    got = _tile(T).cpu().numpy()
    want, idx = _tiles_numpy(T.view(torch.int16).cpu().numpy().view(np.uint16))
    nt = want.size * 2
    np.testing.assert_array_equal(got[:nt].view(np.uint16), want)
    np.testing.assert_array_equal(got[nt:nt + idx.size * 4].view(np.int32), idx.reshape(-1))


def test_refusals():
    T = torch.zeros(64, 64, dtype=BF16, device=DEV)
    nb = fq.fq_frame_tiles_bytes(64, 64)
    out = torch.empty(nb, dtype=torch.uint8, device=DEV)
    for args, status in [((T, 64, 60, out, nb), 2),          # cols not a multiple of 8
                         ((T, 64, 64, out, nb - 1), 4),      # buffer too small
                         ((T, 0, 64, out, nb), 1),
                         ((T, 64, 64, T, nb), 1)]:           # overlaps its source
        with pytest.raises(fq.FrameQuantError) as e:
            fq.fq_frame_tile(*args)
        assert e.value.status == status


def _run(specs, M, tiled):
    """specs: [(workload, layer, use_gamma)] -> [(y, oracle)] for one group launch."""
    layers, keep, refs = [], [], []
    for wl_key, name, use_gamma in specs:
        L = oracle_layer(wl_key, name)
        D = DeviceLayer(L, BF16)
        X = activations(wl_key, name, M)
        x = torch.from_numpy(X).to(DEV, BF16)
        y = torch.full((M, L.d_out), float("nan"), dtype=BF16, device=DEV)
        ti = _tile(D.T_in) if tiled else None
        to = _tile(D.T_out_t) if tiled else None
        keep += [D, x, ti, to]
        layers.append(fq.Layer(x, L.d_in, D.T_in, D.C, D.T_out_t, L.d_out,
                               D.gamma if use_gamma else None, y, ti, to))
        refs.append((L, X, use_gamma))
    nb = fq.fq_group_workspace_bytes(M, layers)
    ws = torch.zeros(nb, dtype=torch.uint8, device=DEV)
    fq.fq_linear_forward_group(M, layers, ws, nb)
    assert fq.fq_check(ws) == 0, fq.fq_status_str(fq.fq_check(ws))
    return [(Ly.y.double().cpu().numpy(), (L, X, g)) for Ly, (L, X, g) in zip(layers, refs)]


CASES = [
    ([("single256", "single", True)], 8),
    ([("llama2_7b_decode", "o", False)], 16),
    ([("llama2_7b_decode", "down", True)], 1),
    ([("llama2_7b_decode", n, False) for n in ("q", "k", "v")], 16),
    ([("llama2_7b_decode", "gate", True), ("llama2_7b_decode", "up", False)], 16),
    ([("vit_b16_mlp", "fc1", False), ("single256", "single", False)], 40),
    ([("vit_b16_mlp", "fc2", True)], 64),
]


@pytest.mark.parametrize("specs,M", CASES)
def test_forward_tiled_equals_row_major_and_oracle(specs, M):
    tiled = _run(specs, M, True)
    plain = _run(specs, M, False)
    for (yt, (L, X, g)), (yp, _) in zip(tiled, plain):
        np.testing.assert_array_equal(yt, yp)
        assert_parity(yt, reference(L, X, g), 1e-2)


def test_mixed_tiled_and_row_major_operands():
    """One layer tiled on the analysis side only, another on the synthesis side only."""
    M = 16
    outs = []
    for mode in ("in", "out"):
        L = oracle_layer("llama2_7b_decode", "q")
        D = DeviceLayer(L, BF16)
        X = activations("llama2_7b_decode", "q", M)
        x = torch.from_numpy(X).to(DEV, BF16)
        y = torch.full((M, L.d_out), float("nan"), dtype=BF16, device=DEV)
        ti = _tile(D.T_in) if mode == "in" else None
        to = _tile(D.T_out_t) if mode == "out" else None
        lay = [fq.Layer(x, L.d_in, D.T_in, D.C, D.T_out_t, L.d_out, None, y, ti, to)]
        nb = fq.fq_group_workspace_bytes(M, lay)
        ws = torch.zeros(nb, dtype=torch.uint8, device=DEV)
        fq.fq_linear_forward_group(M, lay, ws, nb)
        assert fq.fq_check(ws) == 0
        outs.append(y.double().cpu().numpy())
        assert_parity(outs[-1], reference(L, X, False), 1e-2)
    np.testing.assert_array_equal(outs[0], outs[1])


def test_tiles_are_ignored_above_64_tokens():
    (y, (L, X, g)), = _run([("single256", "single", True)], 100, True)
    assert_parity(y, reference(L, X, g), 1e-2)
