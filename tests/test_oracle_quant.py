"""Pins for the oracle's quantizer, de-noising gain and packed layout (Algorithm 1, Appendix I,
Appendix K), checked against brute force, closed forms and hand-worked bit positions."""
import numpy as np
import pytest

import workloads as wl
from oracle import pack, quant


def _gauss(m, n, seed=0, scale=1.0):
    return wl.rng(seed, "quant-test").standard_normal((m, n)) * scale


def test_rtn_codes_in_range_and_fp16_exact():
    C = _gauss(64, 300, scale=0.02)
    q, s, z = quant.rtn(C)
    assert q.dtype == np.uint8 and q.min() >= 0 and q.max() <= 3
    assert s.dtype == np.float16 and z.dtype == np.float16
    # zero is the fp16 value nearest to the row minimum, scale the nearest to range/3
    for i in range(C.shape[0]):
        mn, mx = C[i].min(), C[i].max()
        cands = np.array([np.nextafter(z[i], np.float16(-np.inf)), z[i],
                          np.nextafter(z[i], np.float16(np.inf))], dtype=np.float16)
        assert np.argmin(np.abs(cands.astype(np.float64) - mn)) == 1
        cs = np.array([np.nextafter(s[i], np.float16(0)), s[i],
                       np.nextafter(s[i], np.float16(np.inf))], dtype=np.float16)
        assert np.argmin(np.abs(cs.astype(np.float64) - (mx - mn) / 3)) == 1
    # every code value is used on Gaussian rows
    assert set(np.unique(q)) == {0, 1, 2, 3}


def test_rtn_picks_the_nearest_level_bruteforce():
    C = _gauss(40, 257, seed=1)
    q, s, z = quant.rtn(C)
    levels = s.astype(np.float64)[:, None, None] * np.arange(4)[None, None, :] \
        + z.astype(np.float64)[:, None, None]                         # (rows, 1, 4)
    dist = np.abs(C[:, :, None] - levels)
    best = dist.argmin(axis=2)
    srt = np.sort(dist, axis=2)
    clear = (srt[:, :, 1] - srt[:, :, 0]) > 1e-12                     # ties excepted
    assert clear.mean() > 0.99
    np.testing.assert_array_equal(q[clear], best[clear])


def test_rtn_equally_spaced_row_is_exact():
    C = np.array([[0.5, 1.0, 1.5, 2.0, 1.0, 0.5],
                  [-3.0, -1.0, 1.0, 3.0, 3.0, -3.0]])
    q, s, z = quant.rtn(C)
    np.testing.assert_array_equal(quant.dequantize(q, s, z), C)
    np.testing.assert_array_equal(q, [[0, 1, 2, 3, 1, 0], [0, 1, 2, 3, 3, 0]])


def test_rtn_degenerate_rows():
    C = np.array([[0.25] * 8, [-7.0] * 8])
    q, s, z = quant.rtn(C)
    np.testing.assert_array_equal(q, 0)
    np.testing.assert_array_equal(s, [1.0, 1.0])
    np.testing.assert_array_equal(quant.dequantize(q, s, z), C)


def test_rtn_error_bounded_by_half_step():
    C = _gauss(32, 1000, seed=2, scale=0.05)
    q, s, z = quant.rtn(C)
    err = np.abs(quant.dequantize(q, s, z) - C)
    # half a step, plus the fp16 rounding of zero and of 3*scale at the row ends
    bound = s.astype(np.float64)[:, None] / 2 + 2e-3 * np.abs(C).max(axis=1, keepdims=True)
    assert (err <= bound).all()


def test_clip_2sigma_closed_form():
    C = 100.0 + _gauss(200, 500, seed=3)
    out = quant.clip_2sigma(C)
    mu, sd = C.mean(), C.std()
    assert out.min() == pytest.approx(mu - 2 * sd) and out.max() == pytest.approx(mu + 2 * sd)
    inside = np.abs(C - mu) <= 2 * sd
    np.testing.assert_array_equal(out[inside], C[inside])
    # the share clipped is the Gaussian tail beyond 2 sigma, 4.55%
    assert abs((~inside).mean() - 0.0455) < 0.003
    # bounds are global, not per row: a shifted row is clipped as a whole
    C2 = _gauss(20, 1000, seed=4)
    C2[0] += 10.0                    # global mu ~ 0.5, sigma ~ 2.4: row 0 lies above mu + 2 sigma
    assert (quant.clip_2sigma(C2)[0] < C2[0]).mean() > 0.9


def test_wiener_gain_range_and_identity():
    C = _gauss(16, 2000, seed=5)
    q, s, z = quant.rtn(C)
    g = quant.wiener_gain(C, s)
    assert g.dtype == np.float32 and (g > 0).all() and (g < 1).all()
    # a row without rounding noise (step 0) keeps gain 1
    assert quant.wiener_gain(np.ones((1, 4)), np.array([0.0], np.float16))[0] == 1.0


@pytest.mark.parametrize("snr", [0.02, 0.08, 0.3, 1.0, 4.0])
def test_wiener_gain_is_the_empirical_mse_minimiser(snr):
    """The gain is fixed by what it is for (Sec. 3.1 (b), Appendix I): among all scalings
    gamma of a noisy coefficient c + n, the one with the least mean squared error against c.
    Draw coefficients c ~ N(0, P) and independent rounding noise n ~ U(-s/2, s/2) (the error of
    rounding to a grid of step s), search gamma on a fine grid by brute force, and compare the
    minimiser with the oracle's gain for a row of power P and step s.  The ratios P / s^2 span
    the regime of 2-bit rows; a wrong noise constant (s^2/4 or s^2/6 instead of the variance of
    a uniform step, s^2/12) or a wrong power (mean |c| instead of mean c^2) moves the gain by
    far more than the Monte-Carlo error."""
    r = wl.rng(7, "wiener-mc", str(snr))
    n = 400_000
    s = 1.0
    P = snr * s * s
    c = r.standard_normal(n) * np.sqrt(P)
    noisy = c + r.uniform(-s / 2, s / 2, n)
    grid = np.linspace(0.0, 1.2, 2401)
    # mean((gamma * noisy - c)^2) for every gamma of the grid, from the three sums it needs
    a, b, d = np.mean(noisy * noisy), np.mean(noisy * c), np.mean(c * c)
    mse = grid * grid * a - 2.0 * grid * b + d
    best = grid[np.argmin(mse)]
    row = c[None, :]                                # the row's own power is P up to sampling
    g = float(quant.wiener_gain(row, np.array([s], np.float16))[0])
    # sampling error of the minimiser at n = 4e5 is below 3e-3; the grid step is 5e-4
    assert abs(g - best) < 5e-3, (snr, g, best)


# ------------------------------------------------------------------- packed layout
def test_pack_bit_positions_by_hand():
    n_out, n_in = 130, 70            # two row tiles, two column blocks, both ragged
    assert pack.padded(n_out, n_in) == (256, 128)
    assert pack.packed_words(n_out, n_in) == 256 * 128 // 16
    cases = [(0, 0, 0, 0), (0, 1, 0, 16), (0, 2, 0, 2), (0, 15, 0, 30), (0, 16, 1, 0),
             (0, 63, 3, 30), (1, 0, 4, 0), (0, 64, 512, 0),
             (129, 69, (1 * 2 + 1) * 512 + 1 * 4 + 0, 20)]
    for row, col, widx, bit in cases:
        assert pack.word_index(row, col, n_in) == widx
        assert pack.bit_offset(col) == bit
        codes = np.zeros((n_out, n_in), np.uint8)
        codes[row, col] = 3
        w = pack.pack(codes)
        nz = np.flatnonzero(w)
        assert list(nz) == [widx] and int(w[widx]) == 3 << bit


def test_pack_roundtrip_and_padding():
    codes = wl.random_codes(0, "pack", n_out=300, n_in=200)
    w = pack.pack(codes)
    assert w.dtype == np.uint32 and w.size == pack.packed_words(300, 200)
    np.testing.assert_array_equal(pack.unpack(w, 300, 200), codes)
    # padding rows/columns hold code 0
    po, pi = pack.padded(300, 200)
    mask = np.zeros((po, pi), bool)
    mask[:300, :200] = True
    allc = ((w.reshape(po // 128, pi // 64, 128, 4).transpose(0, 2, 1, 3)[..., None]
             >> np.array([pack.bit_offset(c) for c in range(16)], np.uint32)) & 3)
    assert not allc.reshape(po, pi)[~mask].any()


def test_pack_rejects_out_of_range():
    with pytest.raises(ValueError):
        pack.pack(np.array([[4]], np.uint8))
