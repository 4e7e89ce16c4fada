"""Pins of the oracle's M reconstruction (Sec. 4; Algorithm 3, part 1): the accumulation steps and
the two solves, checked against what the paper and the mathematics fix -- not against the oracle's
own formulas retyped.

* The paper states X X^T = sum_i x_i x_i^T: the per-sample accumulation must equal the batched
  matrix product (a different computation: one BLAS GEMM), and splitting the batch in two and
  continuing the accumulators (the online form) must give the same sums.
* lambda = 0 makes the target the low-rank flow's own output, so Y_t X^T = W X X^T exactly;
  lambda = 1 with X_o = X_u gives the same; the target is affine in lambda.
* U_r from the accumulators (Eq. 4) equals the full-batch least-squares solution of Eq. 3 (from
  numpy's lstsq on all samples at once); V_r^T from Eq. 7 likewise; Eq. 8 with alpha > 0 is the
  minimiser of the regularised objective (its gradient vanishes).
* Planted mistakes (a dropped (1 - lambda), a transposed outer product, the target built from
  x_o alone) fail these pins.
"""
import numpy as np
import pytest

import oracle


def _batch(T, n, m, seed):
    rng = np.random.default_rng(seed)
    Xu = rng.standard_normal((T, n))
    Xo = Xu + 0.1 * rng.standard_normal((T, n))     # the dense flow: the low-rank flow plus drift
    W = rng.standard_normal((m, n)) / np.sqrt(n)
    return Xo, Xu, W


def test_accumulators_equal_the_batched_products_and_xxt_is_psd():
    Xo, Xu, W = _batch(40, 12, 9, 0)
    XXt, YtXt = oracle.m_accumulate(Xo, Xu, W, 0.25)
    assert np.allclose(XXt, Xu.T @ Xu, rtol=0, atol=1e-12)
    Yt = 0.25 * Xo @ W.T + 0.75 * Xu @ W.T
    assert np.allclose(YtXt, Yt.T @ Xu, rtol=0, atol=1e-12)
    assert np.allclose(XXt, XXt.T, atol=0) and np.linalg.eigvalsh(XXt).min() > -1e-10


def test_online_accumulation_equals_one_pass():
    Xo, Xu, W = _batch(33, 10, 7, 1)
    full = oracle.m_accumulate(Xo, Xu, W, 0.4)
    part = oracle.m_accumulate(Xo[:13], Xu[:13], W, 0.4)
    both = oracle.m_accumulate(Xo[13:], Xu[13:], W, 0.4, *part)
    for a, b in zip(full, both):
        assert np.allclose(a, b, rtol=0, atol=1e-12)


def test_lambda_special_cases_and_affinity():
    Xo, Xu, W = _batch(25, 8, 6, 2)
    XXt0, Y0 = oracle.m_accumulate(Xo, Xu, W, 0.0)
    assert np.allclose(Y0, W @ XXt0, rtol=0, atol=1e-12)       # target = W x_u
    _, Ysame = oracle.m_accumulate(Xu, Xu, W, 1.0)
    assert np.allclose(Ysame, W @ XXt0, rtol=0, atol=1e-12)    # x_o = x_u, lambda = 1
    _, Y1 = oracle.m_accumulate(Xo, Xu, W, 1.0)
    _, Yh = oracle.m_accumulate(Xo, Xu, W, 0.3)
    assert np.allclose(Yh, 0.7 * Y0 + 0.3 * Y1, rtol=0, atol=1e-12)


def test_row_restriction_matches_the_full_accumulators():
    Xo, Xu, W = _batch(20, 11, 9, 3)
    XXt, YtXt = oracle.m_accumulate(Xo, Xu, W, 0.25)
    rx, ry = np.array([0, 4, 10]), np.array([1, 2, 8])
    a, b = oracle.m_accumulate(Xo, Xu, W, 0.25, rows=(rx, ry))
    assert np.allclose(a, XXt[rx], rtol=0, atol=1e-12) and np.allclose(b, YtXt[ry], rtol=0, atol=1e-12)


def test_reconstruct_u_equals_full_batch_least_squares():
    """Eq. 4 from the accumulators = Eq. 3 solved directly on all samples (lstsq)."""
    T, n, m, r = 200, 16, 12, 5
    Xo, Xu, W = _batch(T, n, m, 4)
    V = np.random.default_rng(5).standard_normal((n, r))
    lam = 0.25
    XXt, YtXt = oracle.m_accumulate(Xo, Xu, W, lam)
    U_r, V_r = oracle.m_reconstruct(XXt, YtXt, V)
    Yt = lam * Xo @ W.T + (1 - lam) * Xu @ W.T           # T x m targets, rows are samples
    D = Xu @ V                                            # T x r = (V^T X)^T
    Ut, *_ = np.linalg.lstsq(D, Yt, rcond=None)           # min ||Y_t - D U^T||
    assert np.allclose(U_r, Ut.T, rtol=0, atol=1e-9)
    # Eq. 7 (alpha = 0): V_r^T minimises ||Y_t - U_r V^T X|| over V, i.e. lstsq in vec form
    K = np.kron(U_r, Xu)                                  # (T m) x (n r) design for vec(V^T) ... row-major
    vt, *_ = np.linalg.lstsq(K, Yt.T.reshape(-1), rcond=None)
    assert np.allclose(V_r.T, vt.reshape(r, n), rtol=0, atol=1e-8)


def test_reconstruct_v_with_regulariser_is_a_stationary_point():
    """Eq. 8: the gradient of ||Y_t - U_r V^T X||^2 + alpha ||W - U_r V^T||^2 w.r.t. V^T vanishes."""
    T, n, m, r = 150, 10, 8, 4
    Xo, Xu, W = _batch(T, n, m, 6)
    V = np.random.default_rng(7).standard_normal((n, r))
    XXt, YtXt = oracle.m_accumulate(Xo, Xu, W, 0.25)
    U_r, V_r = oracle.m_reconstruct(XXt, YtXt, V, W=W, alpha=0.5)
    Yt = 0.25 * Xo @ W.T + 0.75 * Xu @ W.T
    Vt = V_r.T
    grad = -U_r.T @ (Yt.T - U_r @ Vt @ Xu.T) @ Xu - 0.5 * U_r.T @ (W - U_r @ Vt)
    assert np.abs(grad).max() < 1e-8 * (1 + np.abs(U_r.T @ Yt.T @ Xu).max())


def _mutant(kind):
    """The accumulation with one planted mistake (square W, so a transposed product still fits)."""
    def acc(Xo, Xu, W, lam):
        n, m = Xu.shape[1], W.shape[0]
        XXt, YtXt = np.zeros((n, n)), np.zeros((m, n))
        for xo, xu in zip(Xo, Xu):
            XXt += np.outer(xu, xu)
            if kind == "drop_one_minus_lambda":
                yt = lam * (W @ xo) + (W @ xu)
            elif kind == "dense_flow_only":
                yt = W @ xo
            else:
                yt = lam * (W @ xo) + (1 - lam) * (W @ xu)
            YtXt += np.outer(xu, yt) if kind == "transposed_outer" else np.outer(yt, xu)
        return XXt, YtXt
    return acc


@pytest.mark.parametrize("kind", ["drop_one_minus_lambda", "dense_flow_only", "transposed_outer"])
def test_planted_mistakes_fail_a_pin(kind):
    Xo, Xu, W = _batch(30, 9, 9, 8)
    XXt, Y = _mutant(kind)(Xo, Xu, W, 0.25)
    _, Y0 = _mutant(kind)(Xo, Xu, W, 0.0)
    _, Y1 = _mutant(kind)(Xo, Xu, W, 1.0)
    ok_batched = np.allclose(Y, (0.25 * Xo @ W.T + 0.75 * Xu @ W.T).T @ Xu, atol=1e-9)
    ok_lambda0 = np.allclose(Y0, W @ XXt, atol=1e-9)
    ok_affine = np.allclose(Y, 0.75 * Y0 + 0.25 * Y1, atol=1e-9)
    assert not (ok_batched and ok_lambda0 and ok_affine)
