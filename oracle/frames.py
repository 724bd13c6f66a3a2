"""Oracle, part 1: tight fusion frames (plain fp64 CPU).

TEST INFRASTRUCTURE. Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline leg may
import this package; the product library never does, and shares no code with it.

A (k, rho, d)-TFF (Sec. 2.2, Definition "Tight Fusion Frames") is built the way the paper's
Appendix J describes:
  1. spectral tetris: a rho' x d' real matrix F with unit columns and orthogonal rows of squared
     norm d'/rho' (App. J "Spectral Tetris"), using the 2x2 block T(x);
  2. modulation: row j of F times (w^(k_i n))_n, w = exp(2 pi i / k), for k_i = 0..k-1, spans the
     k subspaces of C^d' (App. J "Modulation");
  3. Parseval normalisation: each modulated vector divided by sqrt(k), so that the fusion frame
     operator is the identity (Sec. 2.1 "Operators in Fusion Frames", S = T* T = I);
  4. realification: the entrywise map x + iy -> [[x, -y], [y, x]] turns a complex (k, rho', d')
     TFF into a real (k, 2 rho', 2 d') one (Sec. 2.2, App. J);
  5. an optional random rotation R gives another TFF, analysis P^T = T R^T (Sec. 2.2 remarks,
     Appendix K: P_l = R_l T_l).

Matrices here are analysis operators: T is n x d with n = k * rho rows, T^T T = I_d.  Row order is
(row j of F, then k_i, then real/imaginary part); real coordinates of complex coordinate c are
(2c, 2c+1).
"""
from __future__ import annotations

import math
from fractions import Fraction

import numpy as np


def spectral_tetris(rho_c: int, d_c: int) -> np.ndarray:
    """Unit-norm tight frame of d_c vectors in C^rho_c as the columns of a real rho_c x d_c
    matrix F (App. J "Spectral Tetris").  Rows are filled left to right: whole ones while the
    row still lacks at least 1 of its squared norm d_c/rho_c, then the remainder x in (0, 1) is
    placed with T(x) = (1/sqrt 2) [[sqrt x, sqrt x], [sqrt(2-x), -sqrt(2-x)]], which also puts
    2 - x into the next row.  Requires d_c/rho_c >= 2."""
    target = Fraction(d_c, rho_c)
    if target < 2:
        raise ValueError(f"spectral tetris needs d/rho >= 2, got {d_c}/{rho_c}")
    F = np.zeros((rho_c, d_c))
    col = 0
    carried = Fraction(0)          # squared norm already in row j from the previous T(x)
    for j in range(rho_c):
        rem = target - carried
        while rem >= 1:
            F[j, col] = 1.0
            col += 1
            rem -= 1
        if rem > 0:
            x = rem
            if j + 1 >= rho_c:
                raise ValueError("spectral tetris ran past the last row")
            top = math.sqrt(float(x) / 2.0)
            bot = math.sqrt(float(2 - x) / 2.0)
            F[j, col], F[j, col + 1] = top, top
            F[j + 1, col], F[j + 1, col + 1] = bot, -bot
            col += 2
            carried = 2 - x
        else:
            carried = Fraction(0)
    if col != d_c:
        raise ValueError("spectral tetris did not use every column")
    return F


def modulation_is_tight(F: np.ndarray, k: int) -> bool:
    """The modulated family is a TFF exactly when every two distinct columns n, m of F with
    n = m (mod k) are orthogonal (the off-diagonal terms of the frame operator are
    sum_j F_jn F_jm * sum_ki w^(ki (n-m)), which vanishes unless n = m mod k)."""
    d_c = F.shape[1]
    for shift in range(k, d_c, k):
        dots = np.einsum("jn,jn->n", F[:, : d_c - shift], F[:, shift:])
        if np.abs(dots).max() > 1e-12:
            return False
    return True


def modulate(F: np.ndarray, k: int) -> np.ndarray:
    """Complex frame vectors (rows) F_j * (w^(k_i n))_n / sqrt(k), ordered (j, k_i).  They are
    the columns of a synthesis operator V (d_c x rho_c k) with V V^* = I (Parseval)."""
    rho_c, d_c = F.shape
    n = np.arange(d_c)
    out = np.empty((rho_c * k, d_c), dtype=np.complex128)
    for j in range(rho_c):
        for ki in range(k):
            ang = 2.0 * np.pi * ((ki * n) % k) / k      # exact reduction before the angle
            out[j * k + ki] = F[j] * np.exp(1j * ang)
    return out / math.sqrt(k)


def realify_analysis(vecs: np.ndarray) -> np.ndarray:
    """Real analysis operator of the realified synthesis operator.  With V = vecs^T (columns are
    the complex frame vectors) and each entry x + iy mapped to [[x, -y], [y, x]], the real
    synthesis operator is V_R (2 d_c x 2 n_c) and the analysis operator is T = V_R^T."""
    n_c, d_c = vecs.shape
    V = vecs.T                                  # d_c x n_c
    VR = np.zeros((2 * d_c, 2 * n_c))
    VR[0::2, 0::2] = V.real
    VR[0::2, 1::2] = -V.imag
    VR[1::2, 0::2] = V.imag
    VR[1::2, 1::2] = V.real
    return VR.T.copy()


def tff_analysis(k: int, rho: int, d: int) -> np.ndarray:
    """Un-rotated real (k, rho, d)-TFF analysis operator, n x d with n = k * rho.
    (1, d, d) is the trivial TFF (the identity), which the paper keeps as the fallback when no
    other triple is valid (Sec. 2.2 remarks)."""
    if k == 1 and rho == d:
        return np.eye(d)
    if rho % 2 or d % 2:
        raise ValueError("the real construction needs even rho and d")
    F = spectral_tetris(rho // 2, d // 2)
    if not modulation_is_tight(F, k):
        raise ValueError(f"(k={k}, rho={rho}, d={d}) is not a valid TFF for this construction")
    return realify_analysis(modulate(F, k))


def is_valid(k: int, rho: int, d: int) -> bool:
    if k == 1 and rho == d:
        return True
    if rho % 2 or d % 2 or (d // 2) < 2 * (rho // 2):
        return False
    return modulation_is_tight(spectral_tetris(rho // 2, d // 2), k)


def choose_k(r: Fraction, d: int, rho: int) -> tuple:
    """(k, rho) for a target redundancy r: k = ceil(r d / rho); when that triple is not valid,
    lower the redundancy one subspace at a time, ending at the trivial (1, d, d) frame
    (Sec. 2.2 remarks)."""
    k = math.ceil(Fraction(r) * d / rho)
    while k * rho >= d:
        if is_valid(k, rho, d):
            return k, rho
        k -= 1
    return 1, d


# --------------------------------------------------------------------------------------------
# random rotation
# --------------------------------------------------------------------------------------------
def haar_orthogonal(g: np.ndarray) -> np.ndarray:
    """Orthogonal factor of the QR decomposition of a square Gaussian matrix, with columns
    signed so that R has a positive diagonal (this makes Q Haar distributed and unique)."""
    q, r = np.linalg.qr(g)
    return q * np.sign(np.diag(r))[None, :]


def rotation_matrix(draws) -> np.ndarray:
    """R = Pi (Q_a kron Q_b) D as an explicit d x d matrix: D = diag(signs), Q_a and Q_b Haar
    from the Gaussian draws, and (Pi v)[i] = v[perm[i]]."""
    Qa, Qb = haar_orthogonal(draws.ga), haar_orthogonal(draws.gb)
    K = np.kron(Qa, Qb) * draws.signs[None, :]
    return K[draws.perm, :]


def rotate_rows(T: np.ndarray, draws) -> np.ndarray:
    """T R^T without forming R: each row t of T becomes R t, and (Q_a kron Q_b) v equals
    vec(Q_a X Q_b^T) for X the a x b row-major reshape of v."""
    Qa, Qb = haar_orthogonal(draws.ga), haar_orthogonal(draws.gb)
    n, d = T.shape
    X = (T * draws.signs[None, :]).reshape(n, draws.a, draws.b)
    Y = np.matmul(np.matmul(Qa[None, :, :], X), Qb.T[None, :, :]).reshape(n, d)
    return np.ascontiguousarray(Y[:, draws.perm])


def unrotate_rows(Y: np.ndarray, draws) -> np.ndarray:
    """Y R without forming R: each row y becomes R^T y = D (Q_a kron Q_b)^T Pi^T y, with
    (Q_a kron Q_b)^T v = vec(Q_a^T X Q_b) for X the a x b row-major reshape of v."""
    Qa, Qb = haar_orthogonal(draws.ga), haar_orthogonal(draws.gb)
    m, d = Y.shape
    Z = np.empty((m, d))
    Z[:, draws.perm] = Y
    X = Z.reshape(m, draws.a, draws.b)
    V = np.matmul(np.matmul(Qa.T[None, :, :], X), Qb[None, :, :]).reshape(m, d)
    return V * draws.signs[None, :]


def run_width(k: int, rho: int, d: int):
    """w = d / rho when spectral tetris gives rho/2 disjoint runs of w ones (F_j = 1 on
    complex coordinates j w .. (j+1) w - 1, App. J with an integer d/rho), else None."""
    if rho % 2 or d % 2 or d % rho:
        return None
    w = d // rho
    F = spectral_tetris(rho // 2, d // 2)
    if not np.array_equal(F, np.kron(np.eye(rho // 2), np.ones((1, w)))):
        return None
    if not modulation_is_tight(F, k):
        raise ValueError(f"(k={k}, rho={rho}, d={d}) is not a valid TFF for this construction")
    return w


def _run_dft(k: int, j: int, w: int) -> np.ndarray:
    """k x w matrix with entries w^(-ki n) / sqrt(k), n = j w .. (j+1) w - 1 the absolute complex
    coordinates of run j (the conjugated modulation of App. J)."""
    n = np.arange(j * w, (j + 1) * w)
    ki = np.arange(k)
    return np.exp(-2j * np.pi * ((ki[:, None] * n[None, :]) % k) / k) / math.sqrt(k)


def analysis_apply(k: int, rho: int, d: int, draws, X: np.ndarray) -> np.ndarray:
    """X T^T (M x n) for T = frame(k, rho, d, draws) without forming T, when d/rho is an
    integer.  T = T_u R^T, so each token is first taken to R^T x; then, with x_c[n] =
    x[2n] + i x[2n+1], the complex coefficient of frame vector (j, ki) is the inner product
    with F_j * w^(ki n) / sqrt(k), i.e. k^-1/2 sum over run j of w^(-ki n) x_c[n]; its real and
    imaginary parts are rows 2 (j k + ki) and 2 (j k + ki) + 1 of the realified operator."""
    X = np.asarray(X, dtype=np.float64)
    if k == 1 and rho == d:
        return X if draws is None else unrotate_rows(X, draws)
    w = run_width(k, rho, d)
    if w is None:
        raise ValueError("structured application needs d / rho to be an integer")
    Xr = X if draws is None else unrotate_rows(X, draws)
    xc = Xr[:, 0::2] + 1j * Xr[:, 1::2]
    Z = np.empty((X.shape[0], k * rho))
    for j in range(rho // 2):
        zc = xc[:, j * w:(j + 1) * w] @ _run_dft(k, j, w).T
        Z[:, 2 * j * k:2 * (j + 1) * k:2] = zc.real
        Z[:, 2 * j * k + 1:2 * (j + 1) * k:2] = zc.imag
    return Z


def synthesis_apply(k: int, rho: int, d: int, draws, U: np.ndarray) -> np.ndarray:
    """U T (M x d), the adjoint of analysis_apply: per run j the complex coordinates are
    sum over ki of u_(j,ki) w^(ki n) / sqrt(k) with u_c = u[2c] + i u[2c+1], written back as
    (Re, Im) pairs, then each token is taken to R y."""
    U = np.asarray(U, dtype=np.float64)
    if k == 1 and rho == d:
        return U if draws is None else rotate_rows(U, draws)
    w = run_width(k, rho, d)
    if w is None:
        raise ValueError("structured application needs d / rho to be an integer")
    uc = U[:, 0::2] + 1j * U[:, 1::2]
    Y = np.empty((U.shape[0], d))
    for j in range(rho // 2):
        yc = uc[:, j * k:(j + 1) * k] @ np.conj(_run_dft(k, j, w))
        Y[:, 2 * j * w:2 * (j + 1) * w:2] = yc.real
        Y[:, 2 * j * w + 1:2 * (j + 1) * w:2] = yc.imag
    return Y if draws is None else rotate_rows(Y, draws)


def frame(k: int, rho: int, d: int, draws=None) -> np.ndarray:
    """Analysis operator P^T (n x d) of the TFF, rotated when rotation draws are given."""
    T = tff_analysis(k, rho, d)
    return T if draws is None else rotate_rows(T, draws)
