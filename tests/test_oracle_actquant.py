"""Pins for the oracle's frame-domain activation rounding (Appendix F): a hand-worked case, the
grid's end points, brute force over the grid, the half-step error bound, symmetry,
idempotence, the vanishing of the error as the bit count grows, the uniform-noise variance, and
the reduction of the whole layer to the unrounded forward."""
import numpy as np
import pytest

import workloads as wl
from oracle import actquant, forward, layer


def test_hand_worked_ternary_case():
    # N = 2: grid {-1, 0, 1} times Delta = max |z| / 1
    Z = np.array([[0.5, -2.0, 1.2, 0.1], [0.0, 1.0, -0.99, 1.01]])
    Zbar, delta = actquant.quantize_ff(Z, 2)
    assert delta == 2.0
    # z / Delta: [.25 -1 .6 .05] and [0 .5 -.495 .505]; .5 is a tie and rounds to even (0)
    np.testing.assert_array_equal(Zbar, [[0, -1, 1, 0], [0, 0, 0, 1]])


def test_hand_worked_int8_case():
    # binary fractions, so every quotient below is exact: max |z| = 127/32, Delta = 1/32
    Z = np.array([[127 / 32, -1.25, 1 / 64, 3 / 64, -0.3]])
    Zbar, delta = actquant.quantize_ff(Z, 8)
    assert delta == 1 / 32
    # z / Delta = 127, -40, 0.5, 1.5, -9.6: ties (0.5, 1.5) round to even
    np.testing.assert_array_equal(Zbar, [[127, -40, 0, 2, -10]])


@pytest.mark.parametrize("bits", [2, 3, 4, 6, 8])
def test_grid_ends_and_range(bits):
    Z = wl.rng(1, "aq-range", str(bits)).standard_normal((37, 301))
    Zbar, delta = actquant.quantize_ff(Z, bits)
    L = (1 << (bits - 1)) - 1
    assert np.abs(Zbar).max() == L                    # the largest |z| lands on the grid's end
    i = np.unravel_index(np.argmax(np.abs(Z)), Z.shape)
    assert Zbar[i] == np.sign(Z[i]) * L
    assert delta == pytest.approx(np.abs(Z).max() / L, rel=1e-15)


@pytest.mark.parametrize("bits", [2, 4, 8])
def test_nearest_grid_point_by_brute_force(bits):
    Z = wl.rng(2, "aq-brute", str(bits)).standard_normal((20, 50)) * 3.0
    Zbar, delta = actquant.quantize_ff(Z, bits)
    L = (1 << (bits - 1)) - 1
    grid = delta * np.arange(-L, L + 1)
    dist = np.abs(Z[..., None] - grid)                 # every element against every level
    best = np.argmin(dist, axis=-1) - L
    srt = np.sort(dist, axis=-1)
    clear = srt[..., 1] - srt[..., 0] > 1e-12          # ties excepted
    np.testing.assert_array_equal(Zbar[clear], best[clear])


@pytest.mark.parametrize("bits", [3, 8])
def test_half_step_bound_symmetry_idempotence(bits):
    Z = wl.rng(3, "aq-props", str(bits)).standard_normal((64, 128))
    Zbar, delta = actquant.quantize_ff(Z, bits)
    assert np.all(np.abs(delta * Zbar - Z) <= delta / 2 * (1 + 1e-12))
    Zn, dn = actquant.quantize_ff(-Z, bits)
    assert dn == delta
    np.testing.assert_array_equal(Zn, -Zbar)
    Z2, d2 = actquant.quantize_ff(delta * Zbar, bits)  # values on the grid stay put
    assert d2 == pytest.approx(delta, rel=1e-15)
    np.testing.assert_array_equal(Z2, Zbar)


def test_zero_tensor():
    Zbar, delta = actquant.quantize_ff(np.zeros((3, 16)), 8)
    assert delta == 0.0 and not Zbar.any()


def test_rounding_noise_is_uniform_over_a_step():
    """Away from the grid's ends, the rounding error of a smooth input is uniform over one
    step: mean 0 and variance Delta^2 / 12 (the model behind the de-noising gain too)."""
    Z = wl.rng(4, "aq-noise").uniform(-1.0, 1.0, (400, 1000))
    Zbar, delta = actquant.quantize_ff(Z, 6)
    e = delta * Zbar - Z
    assert abs(e.mean()) < 1e-3 * delta
    assert e.var() == pytest.approx(delta * delta / 12, rel=0.01)


def test_layer_reduces_to_the_unrounded_forward_as_bits_grow():
    L = layer.from_workload("single256", "single")
    X = wl.activations(wl.WORKLOADS["single256"], wl.WORKLOADS["single256"].layers[0], 8)
    ref = forward.layer_forward(X, L.T_in, L.codes, L.scale, L.zero, L.T_out, L.gamma)
    errs = []
    for bits in (4, 8, 12, 16, 20):
        Y, _, _, _ = actquant.layer_forward_actquant(X, L.T_in, L.codes, L.scale, L.zero,
                                                      L.T_out, L.gamma, bits)
        errs.append(np.linalg.norm(Y - ref) / np.linalg.norm(ref))
    # each 4 more bits shrink the step, and so the error, about 16-fold
    for a, b in zip(errs, errs[1:]):
        assert b < a / 8
    assert errs[-1] < 1e-5
