"""The seeded input generators hold to the recipe they state (and the design notes repeat): the
draw order, the distributions, the index sets of a synthetic layer, and round-to-nearest-even to
bf16 checked against an independent scalar reference, exact ties included."""
import math

import numpy as np
import pytest

from paper_2501_19090_gb300 import inputs


def _bf16_reference(x: float) -> float:
    """Nearest bf16 value (8 significant bits), ties to even, by scaling to an integer and Python's
    round() (which rounds half to even exactly for floats)."""
    if x == 0.0:
        return x
    _, e = math.frexp(x)                 # x = f 2^e, 0.5 <= |f| < 1
    scale = math.ldexp(1.0, e - 8)       # one unit in the 8th significant bit
    return round(x / scale) * scale      # x / scale is exact (a power-of-two scaling)


def test_round_bf16_matches_the_scalar_reference():
    rng = np.random.default_rng(3)
    x = np.concatenate([rng.standard_normal(20000) * 10.0 ** rng.integers(-6, 7, 20000),
                        [1.0, -1.0, 3.0e38 / 2, 1e-30, 0.0]])
    # exact ties: halfway between two bf16 neighbours, with even and odd lower neighbours
    base = inputs.round_bf16(rng.standard_normal(2000)).astype(np.float64)
    ulp = np.array([math.ldexp(1.0, math.frexp(b)[1] - 8) for b in base])
    x = np.concatenate([x, base + ulp / 2, base - ulp / 2])
    got = inputs.round_bf16(x).astype(np.float64)
    ref = np.array([_bf16_reference(float(v)) for v in x])
    assert np.array_equal(got, ref)
    # the results are bf16 values: their low 16 float32 bits are zero
    assert not np.any(inputs.round_bf16(x).view(np.uint32) & np.uint32(0xFFFF))


def test_make_case_draws_u_then_v_then_x_from_one_stream():
    U, V, X = inputs.make_case(inputs.TINY, 16, seed=5)
    rng = np.random.default_rng(5)
    s = 1.0 / math.sqrt(inputs.TINY.r)
    assert np.array_equal(U, (rng.standard_normal((256, 128)) * s).astype(np.float32))
    assert np.array_equal(V, (rng.standard_normal((256, 128)) * s).astype(np.float32))
    assert np.array_equal(X, inputs.round_bf16(rng.standard_normal((16, 256))))


def test_factor_and_activation_scales():
    U, V, rng = inputs.make_factors(2048, 1024, 512, 0)
    assert U.dtype == V.dtype == np.float32 and U.shape == (2048, 512) and V.shape == (1024, 512)
    assert U.std() == pytest.approx(512 ** -0.5, rel=0.01) and V.std() == pytest.approx(512 ** -0.5, rel=0.01)
    X = inputs.make_activations(rng, 256, 1024)
    assert X.std() == pytest.approx(1.0, rel=0.01) and abs(X.mean()) < 0.01


def test_synthetic_layer_index_sets_and_operands():
    m, n, r = 1000, 776, 301
    piv, nonp, Wp, C = inputs.synthetic_layer(m, n, r, 3)
    assert piv.dtype == nonp.dtype == np.int32
    assert np.all(np.diff(piv) > 0) and np.all(np.diff(nonp) > 0)
    assert np.array_equal(np.sort(np.concatenate([piv, nonp])), np.arange(m))
    assert Wp.shape == (r, n) and C.shape == (m - r, r)
    assert np.array_equal(inputs.round_bf16(Wp), Wp) and np.array_equal(inputs.round_bf16(C), C)
    assert Wp.std() == pytest.approx(r ** -0.5, rel=0.02) and C.std() == pytest.approx(0.18, rel=0.02)
    # seeded: the same call gives the same layer, another seed another one
    piv2, _, Wp2, _ = inputs.synthetic_layer(m, n, r, 3)
    assert np.array_equal(piv, piv2) and np.array_equal(Wp, Wp2)
    assert not np.array_equal(piv, inputs.synthetic_layer(m, n, r, 4)[0])


def test_random_rows_and_rank_sweep():
    rows = inputs.random_rows(8192, 512, 0)
    assert rows.size == 512 and np.all(np.diff(rows) > 0) and rows.min() >= 0 and rows.max() < 8192
    assert inputs.random_rows(10, 50, 0).tolist() == list(range(10))
    assert [s.r for s in inputs.rank_sweep_shapes()] == [1024, 1638, 2048, 2458, 3072]
