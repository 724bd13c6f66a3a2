"""Seeded synthetic inputs for the frame-quantized linear layer.

The shapes and value distributions follow the paper's workloads: the ViT-B/16 MLP (Table 1),
Llama-2-7B and Llama-2-70B linear layers (Tables 5-7), and a small 256x256 layer.  The paper's
datasets and trained weights are not used; every tensor here is drawn from a numpy generator
keyed by (seed, layer name, role), so that the oracle, the tests and the benchmark see the same
values.

This module holds none of the method's arithmetic.  It draws weights, activations, outlier
positions, and the raw random numbers that a random rotation consumes (Gaussian matrices, a
permutation and signs).  Frame construction, frame coefficients, quantization and the layer
forward live elsewhere.
"""
from __future__ import annotations

import math
import zlib
from dataclasses import dataclass, field
from fractions import Fraction

import numpy as np

RHO = 16  # subspace dimension used by every workload


# --------------------------------------------------------------------------------------------
# random streams
# --------------------------------------------------------------------------------------------
def rng(seed: int, *key: str) -> np.random.Generator:
    """Independent stream for (seed, key...): SeedSequence spawn keys from crc32 of each part."""
    spawn = tuple(zlib.crc32(k.encode()) for k in key)
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence(seed, spawn_key=spawn)))


def round_bf16(a: np.ndarray) -> np.ndarray:
    """Round to the nearest bfloat16 (ties to even); returns float32 holding bf16 values."""
    f = np.ascontiguousarray(a, dtype=np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    lsb = (u >> 16) & 1
    u = (u + 0x7FFF + lsb) & 0xFFFF0000
    out = u.astype(np.uint32).view(np.float32)
    nan = np.isnan(f)
    if nan.any():
        out = out.copy()
        out[nan] = np.nan
    return out


def bf16_bits(a: np.ndarray) -> np.ndarray:
    """uint16 bit patterns of bf16-representable float32 values (as returned by round_bf16)."""
    f = np.ascontiguousarray(a, dtype=np.float32)
    return (f.view(np.uint32) >> 16).astype(np.uint16)


# --------------------------------------------------------------------------------------------
# workload table
# --------------------------------------------------------------------------------------------
@dataclass(frozen=True)
class Layer:
    name: str
    d_out: int
    d_in: int


@dataclass(frozen=True)
class Workload:
    key: str
    layers: tuple
    tokens: tuple                    # token counts M exercised by this workload
    redundancy: tuple                # r values (Fraction) swept
    seed: int
    weight: str                      # weight distribution recipe name
    act: str                         # activation distribution recipe name
    gamma: tuple = (False,)          # de-noising filter off / on
    fixed_k: int | None = None       # explicit k (both sides), overrides the r rule
    note: str = ""


_7B = (Layer("q", 4096, 4096), Layer("k", 4096, 4096), Layer("v", 4096, 4096),
       Layer("o", 4096, 4096), Layer("gate", 11008, 4096), Layer("up", 11008, 4096),
       Layer("down", 4096, 11008))
_70B = (Layer("q", 8192, 8192), Layer("o", 8192, 8192), Layer("gate", 28672, 8192),
        Layer("up", 28672, 8192), Layer("down", 8192, 28672))

WORKLOADS = {
    "single256": Workload(
        "single256", (Layer("single", 256, 256),), (8,), (Fraction(9, 8),), 0,
        weight="normal_1_over_din_cols20", act="normal_bf16", fixed_k=18,
        note="256x256, W~N(0,1/256) with 4 input columns x20, k=18 rho=16 (r=1.125), M=8"),
    "vit_b16_mlp": Workload(
        "vit_b16_mlp", (Layer("fc1", 3072, 768), Layer("fc2", 768, 3072)), (12608,),
        (Fraction(11, 10),), 1, weight="normal_1_over_din_t3", act="normal_bf16",
        note="ViT-B/16 MLP pair, 64 images x 197 tokens, 0.5% Student-t(3) weight entries"),
    "llama2_7b_decode": Workload(
        "llama2_7b_decode", _7B, (1, 4, 16), (Fraction(11, 10),), 2,
        weight="normal_0.02", act="normal_bf16_outlier30",
        note="Llama-2-7B block shapes, decode"),
    "llama2_7b_prefill": Workload(
        "llama2_7b_prefill", _7B, (2048, 4096), (Fraction(11, 10),), 3,
        weight="normal_0.02", act="normal_bf16_outlier30", gamma=(False, True),
        note="Llama-2-7B block shapes, prefill, de-noising filter off and on"),
    "llama2_70b": Workload(
        "llama2_70b", _70B, (1, 16, 128, 1024, 4096),
        (Fraction(1), Fraction(11, 10), Fraction(6, 5)), 4,
        weight="normal_0.015", act="normal_bf16_outlier30",
        note="Llama-2-70B-shaped layers, token and redundancy sweep"),
}


def k_for(r: Fraction, d: int, rho: int = RHO) -> int:
    """Number of subspaces for a target redundancy: k = ceil(r*d/rho)."""
    return math.ceil(Fraction(r) * d / rho)


def factor_pair(d: int) -> tuple:
    """(a, b) with a*b = d and a the largest divisor of d not above sqrt(d)."""
    a = int(math.isqrt(d))
    while d % a:
        a -= 1
    return a, d // a


# --------------------------------------------------------------------------------------------
# draws
# --------------------------------------------------------------------------------------------
def weight(wl: Workload, layer: Layer) -> np.ndarray:
    """W (d_out x d_in, float64) with the workload's distribution."""
    g = rng(wl.seed, wl.key, layer.name, "W")
    d_out, d_in = layer.d_out, layer.d_in
    if wl.weight == "normal_1_over_din_cols20":
        W = g.standard_normal((d_out, d_in)) / math.sqrt(d_in)
        cols = rng(wl.seed, wl.key, layer.name, "W-outlier-cols").choice(d_in, 4, replace=False)
        W[:, cols] *= 20.0
        return W
    if wl.weight == "normal_1_over_din_t3":
        W = g.standard_normal((d_out, d_in)) / math.sqrt(d_in)
        go = rng(wl.seed, wl.key, layer.name, "W-outliers")
        n = d_out * d_in
        pos = go.choice(n, int(round(0.005 * n)), replace=False)
        W.reshape(-1)[pos] = go.standard_t(3, size=pos.size) / math.sqrt(d_in)
        return W
    if wl.weight.startswith("normal_"):
        sd = float(wl.weight.split("_")[1])
        return g.standard_normal((d_out, d_in)) * sd
    raise ValueError(wl.weight)


def activations(wl: Workload, layer: Layer, M: int) -> np.ndarray:
    """X (M x d_in) as bf16-representable float32 values."""
    g = rng(wl.seed, wl.key, layer.name, "X", str(M))
    X = g.standard_normal((M, layer.d_in))
    if wl.act == "normal_bf16_outlier30":
        # 1% of channels carry outliers x30, at the same positions for every token
        go = rng(wl.seed, wl.key, layer.name, "X-outlier-channels")
        ch = go.choice(layer.d_in, max(1, layer.d_in // 100), replace=False)
        X[:, ch] *= 30.0
    elif wl.act != "normal_bf16":
        raise ValueError(wl.act)
    return round_bf16(X)


def calibration(wl: Workload, layer: Layer, N: int) -> np.ndarray:
    """N calibration tokens (N x d_in) with the distribution of `activations`, drawn from their
    own stream (the quantizer's A_prev of Algorithm 1)."""
    g = rng(wl.seed, wl.key, layer.name, "calibration", str(N))
    X = g.standard_normal((N, layer.d_in))
    if wl.act == "normal_bf16_outlier30":
        go = rng(wl.seed, wl.key, layer.name, "X-outlier-channels")
        ch = go.choice(layer.d_in, max(1, layer.d_in // 100), replace=False)
        X[:, ch] *= 30.0
    elif wl.act != "normal_bf16":
        raise ValueError(wl.act)
    return round_bf16(X)


@dataclass
class RotationDraws:
    """Raw random numbers for one d x d random rotation: two Gaussian matrices (a x a, b x b,
    a*b = d), a permutation of range(d) and d random signs."""
    d: int
    a: int
    b: int
    ga: np.ndarray
    gb: np.ndarray
    perm: np.ndarray
    signs: np.ndarray = field(repr=False)


def rotation_draws(seed: int, *key: str, d: int) -> RotationDraws:
    a, b = factor_pair(d)
    return rotation_draws_ab(seed, *key, d=d, a=a, b=b)


def rotation_draws_ab(seed: int, *key: str, d: int, a: int, b: int) -> RotationDraws:
    """The draws of rotation_draws for a given factor pair a * b = d (the same stream when
    (a, b) is factor_pair(d))."""
    assert a * b == d
    g = rng(seed, *key, "rotation", str(d))
    ga = g.standard_normal((a, a))
    gb = g.standard_normal((b, b))
    perm = g.permutation(d)
    signs = np.where(g.integers(0, 2, size=d) == 1, 1.0, -1.0)
    return RotationDraws(d, a, b, ga, gb, perm, signs)


def random_codes(seed: int, *key: str, n_out: int, n_in: int, levels: int = 4) -> np.ndarray:
    """Uniform integer codes in [0, levels) (uint8), for kernel-arithmetic checks at sizes
    where computing real frame coefficients in fp64 is too slow."""
    return rng(seed, *key, "codes").integers(0, levels, size=(n_out, n_in), dtype=np.uint8)


def random_scale_zero(seed: int, *key: str, n_out: int, mag: float) -> tuple:
    """fp16 per-row scale in [mag/2, mag] and zero in [-2 mag, -mag] (float16 arrays)."""
    g = rng(seed, *key, "scale-zero")
    s = (g.uniform(0.5, 1.0, n_out) * mag).astype(np.float16)
    z = (-g.uniform(1.0, 2.0, n_out) * mag).astype(np.float16)
    return s, z
