"""Seeded synthetic inputs for PIFA layers (shared by the tests, the bench and the oracle's callers).

This module draws random numbers and rounds them to storage precisions. It holds none of the
method's arithmetic: it never forms W' = U V^T, never selects pivots, never solves for C and never
runs a forward pass. Both the CUDA path and the fp64 oracle receive the arrays made here.

Recipe (one layer, one seed):
  * ``rng = numpy.random.default_rng(seed)`` (PCG64);
  * U = rng.standard_normal((m, r)) / sqrt(r), then V = rng.standard_normal((n, r)) / sqrt(r),
    both stored as float32 (their canonical values). The low-rank factors W' = U V^T of Sec. 3.2
    stand in for a pruned LLM weight; each entry of W' then has variance 1/r;
  * X = rng.standard_normal((T, n)) drawn after U and V from the same generator, rounded to the
    activation dtype (bf16 for the LLaMA shapes).

``round_bf16`` is round-to-nearest-even from float64 straight to bf16 (8 significant bits), returned
as float32 values that are exactly representable in bf16.
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np


@dataclasses.dataclass(frozen=True)
class LayerShape:
    """One linear layer W' (m x n) of rank r: m outputs, n inputs."""

    name: str
    m: int
    n: int
    r: int


# LLaMA-2 shaped layers (m outputs x n inputs) at the ranks used for the synthetic workloads.
TINY = LayerShape("tiny_256x256_r128", 256, 256, 128)
ATTN7B = LayerShape("llama2_7b_attn_4096x4096_r2048", 4096, 4096, 2048)
MLP7B_GATE = LayerShape("llama2_7b_mlp_gate_11008x4096_r2048", 11008, 4096, 2048)
MLP7B_UP = LayerShape("llama2_7b_mlp_up_11008x4096_r2048", 11008, 4096, 2048)
MLP7B_DOWN = LayerShape("llama2_7b_mlp_down_4096x11008_r2048", 4096, 11008, 2048)
ATTN70B = LayerShape("llama2_70b_qo_8192x8192_r4096", 8192, 8192, 4096)
MLP70B_GATE = LayerShape("llama2_70b_gate_up_28672x8192_r4096", 28672, 8192, 4096)


def rank_sweep_shapes(d: int = 4096, fractions=(0.25, 0.4, 0.5, 0.6, 0.75)) -> list[LayerShape]:
    """d x d layers with r = round(f * d): 1024, 1638, 2048, 2458, 3072 at d = 4096."""
    out = []
    for f in fractions:
        r = int(math.floor(f * d + 0.5))
        out.append(LayerShape(f"sweep_{d}x{d}_r{r}", d, d, r))
    return out


def round_bf16(a) -> np.ndarray:
    """Round float64 values to bf16 (round to nearest, ties to even); return them as float32.

    Works on the float64 bit pattern: bf16 keeps 1 sign, 8 exponent and 7 stored mantissa bits,
    so the low 45 of float64's 52 mantissa bits are rounded away. Values are assumed finite and
    inside bf16's normal range (true for every Gaussian input drawn here).
    """
    a64 = np.ascontiguousarray(np.asarray(a, dtype=np.float64))
    bits = a64.view(np.uint64)
    drop = np.uint64(45)
    keep_lsb = (bits >> drop) & np.uint64(1)
    bias = (np.uint64(1) << np.uint64(44)) - np.uint64(1) + keep_lsb
    rounded = (bits + bias) & ~((np.uint64(1) << drop) - np.uint64(1))
    return rounded.view(np.float64).astype(np.float32)


def round_fp16(a) -> np.ndarray:
    """Round float64 values to IEEE fp16 (round to nearest even, numpy's cast); return float32.

    Values beyond +-65504 become inf: callers keep C (|C| of order 1) well inside the range."""
    return np.asarray(a, dtype=np.float64).astype(np.float16).astype(np.float32)


def bf16_bits(a32: np.ndarray) -> np.ndarray:
    """The 16-bit bf16 encodings of float32 values that are already exactly bf16 (see round_bf16)."""
    a32 = np.ascontiguousarray(np.asarray(a32, dtype=np.float32))
    return (a32.view(np.uint32) >> np.uint32(16)).astype(np.uint16)


def make_factors(m: int, n: int, r: int, seed: int):
    """Low-rank factors U (m x r) and V (n x r), float32, i.i.d. N(0, std = r^-1/2); plus the rng.

    The returned generator continues the same stream, so activations drawn from it come after
    U and V, as the recipe in the module docstring states.
    """
    rng = np.random.default_rng(seed)
    s = 1.0 / math.sqrt(r)
    U = (rng.standard_normal((m, r)) * s).astype(np.float32)
    V = (rng.standard_normal((n, r)) * s).astype(np.float32)
    return U, V, rng


def make_activations(rng: np.random.Generator, T: int, n: int, dtype: str = "bf16") -> np.ndarray:
    """X (T x n) i.i.d. N(0, 1), rounded to ``dtype`` ('bf16' or 'fp32'); returned as float32."""
    x = rng.standard_normal((T, n))
    if dtype == "bf16":
        return round_bf16(x)
    if dtype == "fp32":
        return x.astype(np.float32)
    raise ValueError(f"unknown activation dtype {dtype!r}")


def make_case(shape: LayerShape, T: int, seed: int = 0, x_dtype: str = "bf16"):
    """U, V (float32) and X (T x n) for one layer and one token count, in the documented order."""
    U, V, rng = make_factors(shape.m, shape.n, shape.r, seed)
    X = make_activations(rng, T, shape.n, x_dtype)
    return U, V, X


def random_rows(T: int, k: int, seed: int) -> np.ndarray:
    """A seeded, sorted sample of k distinct token rows out of T (for checking large outputs)."""
    rng = np.random.default_rng(10_000 + seed)
    k = min(k, T)
    return np.sort(rng.choice(T, size=k, replace=False))


def synthetic_layer(m: int, n: int, r: int, seed: int, c_std: float = 0.18):
    """A PIFA layer drawn directly at random (no compression): I, I^c, W_p, C as float32 values.

    For forward-pass tests that only need *some* valid operands: I is a seeded random r-subset of
    [0, m) in ascending order, W_p ~ N(0, 1/r) and C ~ N(0, c_std^2). Both are bf16-rounded.
    """
    rng = np.random.default_rng(20_000 + seed)
    pivots = np.sort(rng.choice(m, size=r, replace=False)).astype(np.int32)
    mask = np.ones(m, dtype=bool)
    mask[pivots] = False
    nonpivots = np.flatnonzero(mask).astype(np.int32)
    Wp = round_bf16(rng.standard_normal((r, n)) / math.sqrt(r))
    C = round_bf16(rng.standard_normal((m - r, r)) * c_std)
    return pivots, nonpivots, Wp, C
