"""Pins for the oracle's frame construction against what the paper prints and what the
mathematics fixes (Sec. 2.1 Example 1, Sec. 2.2, Appendix J, Appendix K)."""
import math
from fractions import Fraction

import numpy as np
import pytest

import workloads as wl
from oracle import frames


def _printed_F(g, corrected):
    F = np.zeros((g["rho"], g["d"]))
    for r, c, s, m in g["entries"]:
        F[r, c] = s * math.sqrt(m / 8)
    if corrected:
        for r, c, s, m in g["typos"]["corrected"]:
            F[r, c] = s * math.sqrt(m / 8)
    return F


def test_spectral_tetris_matches_printed_4x11(golden):
    g = golden("spectral_tetris_4x11.json")
    F = frames.spectral_tetris(g["rho"], g["d"])
    # equal to the printed matrix once the recorded typo is corrected
    np.testing.assert_allclose(F, _printed_F(g, corrected=True), atol=1e-15)
    # and the printed entries differ from it only at the recorded typo positions
    diff = np.argwhere(np.abs(F - _printed_F(g, corrected=False)) > 1e-12)
    assert sorted(map(tuple, diff)) == [(2, 8), (2, 9)]


@pytest.mark.parametrize("rho_c,d_c", [(4, 11), (3, 7), (5, 13), (8, 16), (8, 2048), (7, 100),
                                       (1, 2), (2, 5), (8, 5504)])
def test_spectral_tetris_is_unit_norm_tight(rho_c, d_c):
    F = frames.spectral_tetris(rho_c, d_c)
    np.testing.assert_allclose((F ** 2).sum(axis=0), 1.0, atol=1e-14)          # unit columns
    np.testing.assert_allclose(F @ F.T, np.eye(rho_c) * d_c / rho_c, atol=1e-12)  # tight rows


def test_spectral_tetris_rejects_low_ratio():
    with pytest.raises(ValueError):
        frames.spectral_tetris(4, 7)


def test_modulated_5_4_11_matches_table(golden):
    g = golden("tff_5_4_11.json")
    k, rho, d = g["k"], g["rho"], g["d"]
    F = frames.spectral_tetris(rho, d)
    V = frames.modulate(F, k) * math.sqrt(k)       # the table prints unnormalised vectors
    w = np.exp(2j * np.pi / k)
    fix = {(r, c): m for r, c, m in g["typos"]["magnitude_corrections"]}
    for row, entries in enumerate(g["rows"]):
        expect = np.zeros(d, dtype=complex)
        for c, s, m, p in entries:
            expect[c] = s * math.sqrt(fix.get((row, c), m) / 8) * w ** p
        np.testing.assert_allclose(V[row], expect, atol=1e-12, err_msg=f"row {row}")
    # tight fusion frame: projections onto the k subspaces sum to (k rho / d) I
    S = np.zeros((d, d), dtype=complex)
    for ki in range(k):
        B = V[[j * k + ki for j in range(rho)]]                 # rho x d basis of subspace ki
        G = B.conj() @ B.T
        np.testing.assert_allclose(G, np.eye(rho) * d / rho, atol=1e-12)   # orthogonal basis
        S += B.T @ np.linalg.inv(G) @ B.conj()
    np.testing.assert_allclose(S, np.eye(d) * k * rho / d, atol=1e-12)


def test_example1_frame_coefficients_projections(golden):
    g = golden("example1.json")
    T = frames.tff_analysis(g["k"], g["rho"], g["d"])
    # Printed subspaces are this construction's k_i = 0, 2, 1 (printed entries truncated)
    order = [0, 2, 1]
    x = np.array(g["x"])
    for b, ki in enumerate(order):
        P = T[2 * ki: 2 * ki + 2].T                              # 4 x 2 synthesis block
        np.testing.assert_allclose(P, g["synthesis_blocks"][b], atol=0.01)
        coef = P.T @ x
        np.testing.assert_allclose(coef, g["coefficients"][b], atol=0.01)
        np.testing.assert_allclose(P @ coef, g["projections"][b], atol=1e-4)
    # the weighted projections add up to x, and S = T^T T = I (Parseval)
    np.testing.assert_allclose(T.T @ (T @ x), x, atol=1e-15)
    np.testing.assert_allclose(T.T @ T, np.eye(4), atol=1e-15)
    # exact values behind the truncated entries: 1/sqrt3, 1/(2 sqrt3), 1/2
    assert abs(T[0, 0] - 1 / math.sqrt(3)) < 1e-15
    assert abs(abs(T[2, 2]) - 1 / (2 * math.sqrt(3))) < 1e-15
    assert abs(abs(T[2, 3]) - 0.5) < 1e-15


def _shapes():
    out = [(18, 16, 256)]
    for d in (768, 3072, 4096):
        for r in (Fraction(1), Fraction(11, 10), Fraction(6, 5)):
            out.append((wl.k_for(r, d), 16, d))
    out.append((wl.k_for(Fraction(11, 10), 11008), 16, 11008))
    out.append((wl.k_for(Fraction(6, 5), 8192), 16, 8192))
    return sorted(set(out))


@pytest.mark.parametrize("k,rho,d", _shapes())
def test_tff_is_parseval_at_workload_shapes(k, rho, d):
    T = frames.tff_analysis(k, rho, d)
    assert T.shape == (k * rho, d)
    if d <= 4096:
        err = np.abs(T.T @ T - np.eye(d)).max()
    else:   # T^T (T V) = V on random probes: the full Gram matrix costs minutes at this size
        V = wl.rng(0, "probe").standard_normal((d, 16))
        err = np.abs(T.T @ (T @ V) - V).max() / np.abs(V).max()
    assert err <= 1e-10, err
    # each row has squared norm 1/r (weights w_i = 1/sqrt(r) absorbed, Sec. 3)
    np.testing.assert_allclose((T ** 2).sum(axis=1), d / (k * rho), rtol=1e-12)


def test_largest_shape_is_valid():
    # d = 28672 (Llama-2-70B MLP) at r = 1, 1.1, 1.2: the validity certificate of the
    # modulation step (full T^T T would need tens of GB in fp64)
    F = frames.spectral_tetris(8, 14336)
    for r in (Fraction(1), Fraction(11, 10), Fraction(6, 5)):
        assert frames.modulation_is_tight(F, wl.k_for(r, 28672))


def test_subspace_bases_are_orthonormal():
    k, rho, d = 18, 16, 256
    T = frames.tff_analysis(k, rho, d)
    r = k * rho / d
    for ki in range(k):
        rows = [2 * (j * k + ki) + e for j in range(rho // 2) for e in (0, 1)]
        B = T[rows] * math.sqrt(r)
        np.testing.assert_allclose(B @ B.T, np.eye(rho), atol=1e-12)
    # different subspaces are not orthogonal to each other (they overlap: it is a frame)
    assert np.abs(T[0] @ T[2]) > 1e-3


@pytest.mark.parametrize("k,rho,d", [(18, 16, 256), (282, 16, 4096), (5, 8, 22)])
def test_unrotated_block_structure(k, rho, d):
    """Appendix K: the un-rotated operator is block diagonal, one block per row of F, each
    block k (complex) rows wide on at most ceil(d/rho) + 2 (complex) columns."""
    T = frames.tff_analysis(k, rho, d)
    rho_c = rho // 2
    limit = 2 * (math.ceil(d / rho) + 2)
    prev_hi = -1
    for j in range(rho_c):
        blk = T[2 * k * j: 2 * k * (j + 1)]
        cols = np.flatnonzero(np.abs(blk).sum(axis=0) > 1e-15)
        lo, hi = cols.min(), cols.max()
        assert hi - lo + 1 <= limit
        assert lo >= prev_hi - 3          # neighbours share at most one T(x) column pair
        prev_hi = hi


def test_rotation_is_orthogonal_and_matches_rows():
    d = 48
    draws = wl.rotation_draws(7, "test", d=d)
    R = frames.rotation_matrix(draws)
    np.testing.assert_allclose(R.T @ R, np.eye(d), atol=1e-13)
    T = frames.tff_analysis(7, 8, d)
    np.testing.assert_allclose(frames.rotate_rows(T, draws), T @ R.T, atol=1e-13)
    Tr = frames.frame(7, 8, d, draws)
    np.testing.assert_allclose(Tr.T @ Tr, np.eye(d), atol=1e-13)   # still a TFF
    # same draws, same rotation
    np.testing.assert_array_equal(frames.rotation_matrix(wl.rotation_draws(7, "test", d=d)), R)


def test_haar_factor_is_the_positive_qr():
    g = wl.rng(3, "haar").standard_normal((20, 20))
    Q = frames.haar_orthogonal(g)
    np.testing.assert_allclose(Q.T @ Q, np.eye(20), atol=1e-13)
    Rf = Q.T @ g                                   # must be upper triangular, positive diagonal
    assert np.abs(np.tril(Rf, -1)).max() < 1e-12
    assert (np.diag(Rf) > 0).all()


def test_choose_k_rule_and_fallbacks():
    assert frames.choose_k(Fraction(11, 10), 4096, 16) == (282, 16)
    assert frames.choose_k(Fraction(11, 10), 11008, 16) == (757, 16)
    assert frames.choose_k(Fraction(11, 10), 768, 16) == (53, 16)
    assert frames.choose_k(Fraction(6, 5), 28672, 16) == (2151, 16)
    assert frames.choose_k(Fraction(1), 8192, 16) == (512, 16)
    # d = 20, rho = 4: w = 5, so k = 4 (r = 0.8 < 1) is never reached; r = 1 gives k = 5
    assert frames.choose_k(Fraction(1), 20, 4) == (5, 4)
    # rho = 8 on d = 12: d/rho < 2, no construction: trivial frame
    assert frames.choose_k(Fraction(3, 2), 12, 8) == (1, 12)
    np.testing.assert_array_equal(frames.tff_analysis(1, 12, 12), np.eye(12))


def test_invalid_triple_rejected():
    # k smaller than the support width w = d/rho breaks tightness
    with pytest.raises(ValueError):
        frames.tff_analysis(10, 16, 256)


# ---- structured application (no dense T), for layers whose dense T does not fit in fp64
@pytest.mark.parametrize("k,rho,d", [(18, 16, 256), (53, 16, 768), (5, 8, 40), (7, 8, 48),
                                     (1, 48, 48), (20, 16, 256)])
@pytest.mark.parametrize("rotate", [False, True])
def test_structured_application_equals_the_dense_frame(k, rho, d, rotate):
    draws = wl.rotation_draws(5, "structured", str(k), d=d) if rotate else None
    T = frames.frame(k, rho, d, draws)
    g = wl.rng(5, "structured-x", str(k), str(d))
    X = g.standard_normal((6, d))
    U = g.standard_normal((6, T.shape[0]))
    np.testing.assert_allclose(frames.analysis_apply(k, rho, d, draws, X), X @ T.T, atol=1e-12)
    np.testing.assert_allclose(frames.synthesis_apply(k, rho, d, draws, U), U @ T, atol=1e-12)


def test_unrotate_is_the_transpose_rotation():
    d = 96
    draws = wl.rotation_draws(9, "unrotate", d=d)
    R = frames.rotation_matrix(draws)
    Y = wl.rng(9, "unrotate-y").standard_normal((4, d))
    np.testing.assert_allclose(frames.unrotate_rows(Y, draws), Y @ R, atol=1e-13)
    np.testing.assert_allclose(frames.unrotate_rows(frames.rotate_rows(Y, draws), draws), Y,
                               atol=1e-13)


@pytest.mark.parametrize("d", [8192, 28672])
def test_structured_frame_is_tight_at_llama70b_widths(d):
    # Parseval at full width, without the dense operator: synthesis(analysis(x)) = x
    k, rho = frames.choose_k(Fraction(11, 10), d, 16)
    draws = wl.rotation_draws(4, "tight", d=d)
    X = wl.rng(4, "tight-x", str(d)).standard_normal((2, d))
    Z = frames.analysis_apply(k, rho, d, draws, X)
    assert Z.shape == (2, k * rho)
    np.testing.assert_allclose(frames.synthesis_apply(k, rho, d, draws, Z), X, atol=1e-10)
    # and the energy is kept (T^T T = I means |T x| = |x|)
    np.testing.assert_allclose(np.linalg.norm(Z, axis=1), np.linalg.norm(X, axis=1), rtol=1e-12)


def test_structured_application_needs_integer_runs():
    # d / rho not an integer: spectral tetris places T(x) blocks, no runs of ones
    with pytest.raises(ValueError):
        frames.analysis_apply(5, 4, 22, None, np.zeros((1, 22)))
