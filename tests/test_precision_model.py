"""Why every variant carries Y_p into the second contraction as a hi + lo pair of C's type (the
reading of Algorithm 2's step 3 taken for precision): on a layer from Algorithm 1, rounding Y_p
once to bf16 already breaks the tolerance the GPU path is held to, while the pair keeps the
error more than two orders of magnitude inside it. The emulation uses the oracle's steps on the
same rounded operands the kernels get; only the rounding of Y_p differs between the two arms."""
import numpy as np

import oracle
from paper_2501_19090_gb300 import inputs

REL_FRO, ELEM = 5e-3, 2e-2


def _errors(Y, ref):
    return (np.linalg.norm(Y - ref) / np.linalg.norm(ref), np.max(np.abs(Y - ref) / (np.abs(ref) + 1.0)))


def test_one_bf16_plane_fails_the_tolerance_and_hi_lo_meets_it():
    m = n = 512
    r = 256
    U, V, rng = inputs.make_factors(m, n, r, 0)
    L = oracle.compress(U, V, r, "lapack")
    Wp, C = inputs.round_bf16(L.Wp).astype(np.float64), inputs.round_bf16(L.C).astype(np.float64)
    X = inputs.make_activations(rng, 64, n, "bf16").astype(np.float64)
    ref = oracle.forward(X, Wp, C, L.pivots, L.nonpivots)
    Yp = X @ Wp.T                                     # step 2 (exact here; the kernels use fp32)
    hi = inputs.round_bf16(Yp).astype(np.float64)
    lo = inputs.round_bf16(Yp - hi).astype(np.float64)

    def with_planes(planes):                          # steps 3-5 with Y_p replaced by its planes
        Y = np.empty_like(ref)
        Y[:, L.pivots] = Yp
        Y[:, L.nonpivots] = sum(p @ C.T for p in planes)
        return Y

    rel1, elem1 = _errors(with_planes([hi]), ref)
    rel2, elem2 = _errors(with_planes([hi, lo]), ref)
    assert elem1 > ELEM and rel1 > 0.5 * REL_FRO, (rel1, elem1)          # one plane: out of tolerance
    assert rel2 < 1e-2 * REL_FRO and elem2 < 1e-2 * ELEM, (rel2, elem2)  # the pair: far inside it
    # the cause is cancellation, not large coefficients: |C| stays of order one while each
    # non-pivot output sums r products of that size
    assert np.abs(C).max() < 4.0
