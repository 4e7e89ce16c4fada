"""pifa_compress_device (Algorithm 1 on the GPU, float64) through the C ABI, against the fp64 oracle.

Pivots (I, I^c) must equal the oracle's bit for bit: the plain greedy loop on small and ragged
layers, LAPACK's pivoted QR on the LLaMA-shaped ones. C is pinned by Eq. 2 (||C W_p - W_np|| /
||W'|| <= 1e-10, the lossless reconstruction the paper states) and W_p by Eq. 1, both checked in
fp64 on the host on sampled rows.
"""
import time

import numpy as np
import pytest
import torch

import oracle
from paper_2501_19090_gb300 import inputs
from paper_2501_19090_gb300 import pifa as P

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")


def _device_compress(U, V):
    Ud = torch.from_numpy(np.ascontiguousarray(U, dtype=np.float64)).to(DEV)
    Vd = torch.from_numpy(np.ascontiguousarray(V, dtype=np.float64)).to(DEV)
    piv, nonp, Wp, C, info = P.pifa_compress_device(Ud, Vd)
    return (piv.cpu().numpy().astype(np.int64), nonp.cpu().numpy().astype(np.int64), Wp.cpu().numpy(),
            C.cpu().numpy(), info)


def _check_eqs(U, V, piv, nonp, Wp, C, rows=None):
    """Eq. 1 (W_p = W'[I]) and Eq. 2 (W'[I^c] = C W_p) in fp64 on the host, on sampled rows."""
    Ud, Vd = U.astype(np.float64), V.astype(np.float64)
    Wp_ref = Ud[piv] @ Vd.T
    assert np.abs(Wp - Wp_ref).max() <= 1e-12 * np.abs(Wp_ref).max()
    if nonp.size:
        sel = np.arange(nonp.size) if rows is None else rows
        Wnp = Ud[nonp[sel]] @ Vd.T
        err = np.linalg.norm(C[sel] @ Wp - Wnp) / np.linalg.norm(Wnp)
        assert err <= 1e-10, err


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    P.load()


@pytest.mark.parametrize("m,n,r,seed", [(256, 256, 128, 0), (300, 200, 77, 3), (64, 128, 64, 4), (40, 48, 1, 5),
                                         (1000, 776, 301, 3), (97, 61, 33, 8)])
def test_small_layers_match_the_greedy_oracle(m, n, r, seed):
    U, V, _ = inputs.make_factors(m, n, r, seed)
    L = oracle.compress(U, V, r, "greedy")
    piv, nonp, Wp, C, info = _device_compress(U, V)
    assert np.array_equal(piv, L.pivots)
    assert np.array_equal(nonp, L.nonpivots)
    _check_eqs(U, V, piv, nonp, Wp, C)
    np.testing.assert_allclose(Wp, L.Wp, rtol=0, atol=1e-12 * np.abs(L.Wp).max())
    if C.size:
        np.testing.assert_allclose(C, L.C, rtol=0, atol=1e-9 * max(1.0, np.abs(L.C).max()))
    assert 0 < info.r_ratio <= 1 and info.min_pivot_gap >= 0


def test_worked_example_golden():
    """The hand-derived 5 x 3, rank-2 example (tests/golden): W' = U V^T with U its first two
    columns and V = [e_0, e_1], so the pivots and C printed there must come out exactly."""
    import os
    path = os.path.join(os.path.dirname(__file__), "golden", "worked_example_5x3_r2.txt")
    W, C_ref, kv = [], [], {}
    for ln in open(path):
        if not ln.strip() or ln.startswith("#"):
            continue
        key, *vals = ln.split()
        if key == "W":
            W.append([float(v) for v in vals])
        elif key == "C":
            C_ref.append([float(v) for v in vals])
        else:
            kv[key] = [int(v) for v in vals] if key in ("pivots", "nonpivots") else vals
    W = np.array(W)
    U = W[:, :2].copy()
    V = np.array([[1.0, 0.0], [0.0, 1.0], [0.0, 0.0]])
    assert np.array_equal(U @ V.T, W)
    piv, nonp, Wp, C, _ = _device_compress(U, V)
    assert piv.tolist() == kv["pivots"] and nonp.tolist() == kv["nonpivots"]
    np.testing.assert_allclose(C, np.array(C_ref), rtol=0, atol=1e-14)
    np.testing.assert_allclose(Wp, W[piv], rtol=0, atol=1e-14)


@pytest.mark.parametrize("m,n,r", [(4096, 4096, 2048), (4096, 4096, 1638), (11008, 4096, 2048)])
def test_llama_layers_match_the_lapack_oracle(m, n, r):
    U, V, _ = inputs.make_factors(m, n, r, 0)
    L = oracle.compress(U, V, r, "lapack")
    piv, nonp, Wp, C, info = _device_compress(U, V)
    assert np.array_equal(piv, L.pivots), f"{np.setdiff1d(piv, L.pivots)[:8]}"
    assert np.array_equal(nonp, L.nonpivots)
    _check_eqs(U, V, piv, nonp, Wp, C, rows=inputs.random_rows(m - r, 64, 1))


def test_rank_deficient_is_reported():
    """Two identical columns in U and V make W' = U V^T rank r - 1."""
    U, V, _ = inputs.make_factors(200, 150, 20, 6)
    U[:, 7] = U[:, 3]
    V[:, 7] = V[:, 3]
    with pytest.raises(P.PifaError) as e:
        _device_compress(U, V)
    assert e.value.status == P.PIFA_ERR_RANK_DEFICIENT


def test_llama70b_gate_up_compresses_on_the_gpu():
    """The 28672 x 8192, r = 4096 layer: Eq. 1 and Eq. 2 on sampled rows; its pivots against the
    host route (pifa_compress, itself bit-exact with the oracle on the smaller layers) would take
    minutes on the host, so this checks the relations the pivots must satisfy instead: I and I^c
    partition [0, m), the sampled non-pivot rows are reproduced to 1e-10 (Eq. 2)."""
    m, n, r = 28672, 8192, 4096
    U, V, _ = inputs.make_factors(m, n, r, 0)
    t0 = time.perf_counter()
    piv, nonp, Wp, C, info = _device_compress(U, V)
    dt = time.perf_counter() - t0
    assert P.pifa_validate_indices(piv, nonp, m, r) == P.PIFA_OK
    rows = inputs.random_rows(m - r, 48, 2)
    pr = inputs.random_rows(r, 16, 3)
    Ud, Vd = U.astype(np.float64), V.astype(np.float64)
    Wp_ref = Ud[piv[pr]] @ Vd.T
    assert np.abs(Wp[pr] - Wp_ref).max() <= 1e-12 * np.abs(Wp_ref).max()
    Wnp = Ud[nonp[rows]] @ Vd.T
    assert np.linalg.norm(C[rows] @ Wp - Wnp) / np.linalg.norm(Wnp) <= 1e-10
    print(f"pifa_compress_device 28672 x 8192, r = 4096: {dt:.2f} s, min gap {info.min_pivot_gap:.3e}")
