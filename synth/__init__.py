"""Seeded synthetic inputs shared by the oracle tests, the GPU parity tests and
the benchmark.

This module draws random numbers and lays them out; it holds none of the
method's arithmetic (no packing rule, no scale product, no contraction).
Distributions follow the workloads the paper evaluates on (LLaMA / Qwen /
Gemma linears): i.i.d. +-1 sign factors, FP16 scales |N(0, 0.02)| + 1e-3,
FP16 N(0, 1) activations, optionally with 1 % outlier channels scaled by 20.

Draw order for one layer is fixed: U signs, V signs, a, s, b, x.
"""
from __future__ import annotations

import numpy as np

# LLaMA-3-8B decoder linears as (name, d_out, d_in).
LLAMA3_8B_LINEARS = (
    ("q", 4096, 4096),
    ("k", 1024, 4096),
    ("v", 1024, 4096),
    ("o", 4096, 4096),
    ("gate", 14336, 4096),
    ("up", 14336, 4096),
    ("down", 4096, 14336),
)

# 70B-class shapes (d_out, d_in).
LLAMA_70B_SHAPES = ((8192, 8192), (1024, 8192), (28672, 8192), (8192, 28672))


def rng(seed: int) -> np.random.Generator:
    return np.random.default_rng(np.random.PCG64(seed))


def signs(g: np.random.Generator, rows: int, cols: int) -> np.ndarray:
    """rows x cols int8 matrix of i.i.d. +-1."""
    return np.where(g.integers(0, 2, size=(rows, cols), dtype=np.int8) == 1, 1, -1).astype(np.int8)


def random_words(g: np.random.Generator, rows: int, words: int, valid_cols: int) -> np.ndarray:
    """rows x words uint32 of i.i.d. uniform bits, with every bit at column
    >= valid_cols of each row cleared (the row padding of a packed factor).
    Uniform bits are i.i.d. +-1 signs in any bit-per-sign encoding."""
    w = g.integers(0, 2**32, size=(rows, words), dtype=np.uint32)
    full = valid_cols // 32
    rem = valid_cols % 32
    if full < words:
        if rem:
            w[:, full] &= np.uint32((1 << rem) - 1)
            w[:, full + 1:] = 0
        else:
            w[:, full:] = 0
    return w


def scales_f16(g: np.random.Generator, size: int) -> np.ndarray:
    """FP16 bit patterns of |N(0, 0.02)| + 1e-3."""
    v = np.abs(g.normal(0.0, 0.02, size=size)) + 1e-3
    return v.astype(np.float16).view(np.uint16)


def unit_gain_scales_f16(g: np.random.Generator, size: int, level: float) -> np.ndarray:
    """FP16 bit patterns of level * U(0.5, 1.5): scales for chains of layers
    whose activations should stay of order one (level ~ 1 / sqrt(n r) for the
    rank scale, 1 for the row and column scales)."""
    return (level * g.uniform(0.5, 1.5, size=size)).astype(np.float16).view(np.uint16)


def activations_f16(g: np.random.Generator, tokens: int, d_in: int, outlier_frac: float = 0.0,
                    outlier_gain: float = 20.0) -> np.ndarray:
    """FP16 bit patterns of N(0, 1) activations (tokens x d_in); a seeded
    `outlier_frac` of the channels (columns) is multiplied by `outlier_gain`."""
    x = g.normal(0.0, 1.0, size=(tokens, d_in))
    if outlier_frac > 0:
        k = max(1, int(round(outlier_frac * d_in)))
        cols = g.choice(d_in, size=k, replace=False)
        x[:, cols] *= outlier_gain
    return x.astype(np.float16).view(np.uint16)


def layer_signs(seed: int, d_out: int, d_in: int, r: int, tokens: int, outlier_frac: float = 0.0):
    """Layer with explicit sign matrices: U (d_out x r), V (d_in x r) int8,
    a, s, b FP16 bits, x FP16 bits (tokens x d_in)."""
    g = rng(seed)
    U = signs(g, d_out, r)
    V = signs(g, d_in, r)
    a = scales_f16(g, d_out)
    s = scales_f16(g, r)
    b = scales_f16(g, d_in)
    x = activations_f16(g, tokens, d_in, outlier_frac)
    return dict(U=U, V=V, a=a, s=s, b=b, x=x)


def layer_words(seed: int, d_out: int, d_in: int, r: int, tokens: int, outlier_frac: float = 0.0):
    """Layer drawn directly as packed words (same i.i.d. sign distribution,
    cheaper at full size). Word counts follow the 16-byte padded row layout
    of the packed format: U is d_out x 4*ceil(r/128), V is r x 4*ceil(d_in/128)."""
    g = rng(seed)
    wu = 4 * ((r + 127) // 128)
    wv = 4 * ((d_in + 127) // 128)
    Uw = random_words(g, d_out, wu, r)
    Vw = random_words(g, r, wv, d_in)
    a = scales_f16(g, d_out)
    s = scales_f16(g, r)
    b = scales_f16(g, d_in)
    x = activations_f16(g, tokens, d_in, outlier_frac)
    return dict(Uw=Uw, Vw=Vw, a=a, s=s, b=b, x=x)


def integer_layer(seed: int, d_out: int, d_in: int, r: int, tokens: int, xmax: int = 2):
    """Integer-exact case: unit scales, integer activations in [-xmax, xmax]."""
    g = rng(seed)
    U = signs(g, d_out, r)
    V = signs(g, d_in, r)
    one = np.float16(1.0).view(np.uint16)
    a = np.full(d_out, one, dtype=np.uint16)
    s = np.full(r, one, dtype=np.uint16)
    b = np.full(d_in, one, dtype=np.uint16)
    x = g.integers(-xmax, xmax + 1, size=(tokens, d_in)).astype(np.float16).view(np.uint16)
    return dict(U=U, V=V, a=a, s=s, b=b, x=x)


def hisa_rank_factors(seed: int, count: int) -> np.ndarray:
    """Per-matrix rank factors for a HiSA-like allocation over `count`
    matrices: i.i.d. uniform in [0.7, 1.3] (the +-30 % spread around the
    1.0-BPW rank), plus a seeded visiting order for the final +1 steps of the
    renormalisation. Random numbers only; the budget arithmetic is the
    caller's."""
    g = rng(seed)
    return g.uniform(0.7, 1.3, size=count), g.permutation(count)
