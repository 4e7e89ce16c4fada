"""Pins for the fp64 oracle: checks against what the paper and the mathematics fix, not against
the oracle itself.

* a hand-derived worked example (tests/golden/worked_example_5x3_r2.txt; Sec. 3.2, Eqs. 1-2);
* brute force with exact rationals: at every greedy step the chosen row maximises the Gram
  determinant of the chosen set (= squared volume), ties to the lowest index (Algorithm 1, step 1);
* special cases: zero rows, duplicate rows, rank 1, r = m;
* losslessness (Eq. 2) and Y_PIFA = X W'^T (Algorithm 2 is exact in exact arithmetic);
* invariance of Y under a different valid pivot set (several correct layers exist);
* the closed form C = U_np U_p^{-1} when W' = U V^T;
* the cost counts of Sec. 3.3 against an instrumented naive loop;
* LAPACK's pivoted QR picks the same rows as the plain greedy loop;
* planted mistakes in copies of oracle functions make at least one pin fail;
* the backward pass: exact central differences (Y is linear in each input), Euler's identity for
  degree-one homogeneous maps, the chain rule through the dense weight, the r = m linear-layer
  case, and planted mistakes.
"""
import itertools
import math
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle
from paper_2501_19090_gb300 import inputs

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ---------------------------------------------------------------------------------------------
# helpers: exact rational linear algebra (independent of numpy)
# ---------------------------------------------------------------------------------------------
def _det(M):
    """Determinant of a square list-of-lists of Fractions by fraction-exact elimination."""
    A = [row[:] for row in M]
    n = len(A)
    det = Fraction(1)
    for c in range(n):
        p = next((i for i in range(c, n) if A[i][c] != 0), None)
        if p is None:
            return Fraction(0)
        if p != c:
            A[c], A[p] = A[p], A[c]
            det = -det
        det *= A[c][c]
        for i in range(c + 1, n):
            f = A[i][c] / A[c][c]
            if f:
                for j in range(c, n):
                    A[i][j] -= f * A[c][j]
    return det


def _gram_det(rows):
    if not rows:
        return Fraction(1)
    return _det([[sum(a * b for a, b in zip(u, v)) for v in rows] for u in rows])


def exact_greedy_pivots(W, r):
    """Greedy volume maximisation with exact rationals: returns (order, min relative norm gap).

    At each step every unchosen row i is scored by det(Gram(W[S + [i]])); det(Gram(S + [i])) =
    det(Gram(S)) * residual_i^2, so the argmax is the row of largest residual norm.
    """
    Wq = [[Fraction(int(v)) for v in row] for row in W]
    m = len(Wq)
    chosen, min_gap = [], math.inf
    for _ in range(r):
        scores = []
        for i in range(m):
            if i in chosen:
                continue
            scores.append((_gram_det([Wq[j] for j in chosen] + [Wq[i]]), i))
        best = max(s for s, _ in scores)
        winner = min(i for s, i in scores if s == best)        # lowest index among ties
        rest = [s for s, i in scores if i != winner]
        if best > 0 and rest:
            runner = max(rest)
            min_gap = min(min_gap, 1.0 - math.sqrt(float(runner / best)))
        chosen.append(winner)
    return chosen, min_gap


def exact_coefficients(W, pivots, nonpivots):
    """C with W_np = C W_p in exact rationals (least squares normal equations solved exactly)."""
    Wq = [[Fraction(int(v)) for v in row] for row in W]
    Wp = [Wq[i] for i in pivots]
    r = len(pivots)
    G = [[sum(a * b for a, b in zip(u, v)) for v in Wp] for u in Wp]   # W_p W_p^T (r x r)
    out = []
    for i in nonpivots:
        rhs = [sum(a * b for a, b in zip(Wq[i], v)) for v in Wp]         # W_p w_i
        # Cramer's rule on the r x r system G c = rhs
        d = _det(G)
        row = []
        for k in range(r):
            Gk = [G[a][:k] + [rhs[a]] + G[a][k + 1:] for a in range(r)]
            row.append(_det(Gk) / d)
        out.append(row)
    return out


def read_golden(name):
    d = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            key, *vals = line.split()
            d.setdefault(key, []).append([float(v) for v in vals])
    return d


def random_layer(m, n, r, seed):
    U, V, rng = inputs.make_factors(m, n, r, seed)
    return U.astype(np.float64), V.astype(np.float64), rng


# ---------------------------------------------------------------------------------------------
# pins written as predicates so the planted-mistake tests can run them on mutated oracles
# ---------------------------------------------------------------------------------------------
def pin_golden_example(compress_weight=oracle.compress_weight, forward=oracle.forward):
    g = read_golden("worked_example_5x3_r2.txt")
    W = np.array(g["W"])
    r = int(g["r"][0][0])
    layer = compress_weight(W, r)
    ok = list(layer.info.order) == [int(v) for v in g["order"][0]]
    ok &= list(layer.pivots) == [int(v) for v in g["pivots"][0]]
    ok &= list(layer.nonpivots) == [int(v) for v in g["nonpivots"][0]]
    ok &= np.allclose(layer.C, np.array(g["C"]), atol=1e-14, rtol=0)
    y = forward(np.array(g["x"]), layer.Wp, layer.C, layer.pivots, layer.nonpivots)
    ok &= np.allclose(y, np.array(g["y"]), atol=1e-13, rtol=0)
    return bool(ok)


def pin_bruteforce(select=oracle.select_pivot_rows, trials=60, seed=7):
    """Compare the greedy order with exact volume maximisation on small integer matrices.

    Matrices with an exact tie or a relative gap under 1e-9 at some step are skipped (there the
    floating-point order legitimately depends on rounding); at least half must be usable.
    """
    rng = np.random.default_rng(seed)
    used = 0
    for _ in range(trials):
        m = int(rng.integers(3, 9))
        n = int(rng.integers(2, 7))
        r = int(rng.integers(1, min(m, n, 4) + 1))
        # rank-r integer matrix: product of small integer factors
        A = rng.integers(-3, 4, size=(m, r))
        B = rng.integers(-3, 4, size=(r, n))
        W = A @ B
        if np.linalg.matrix_rank(W) != r:
            continue
        order, gap = exact_greedy_pivots(W.tolist(), r)
        if gap < 1e-9:
            continue
        used += 1
        info = select(W.astype(np.float64), r)
        if list(info.order) != order:
            return False
    return used >= trials // 2


def pin_lossless(compress=oracle.compress, shapes=((64, 48, 20), (40, 96, 40), (33, 33, 33))):
    for seed, (m, n, r) in enumerate(shapes):
        U, V, _ = random_layer(m, n, r, seed)
        W = oracle.form_weight(U, V)
        layer = compress(U, V, r)
        if oracle.lossless_error(W, layer) > 1e-10:
            return False
        if not np.array_equal(layer.Wp, W[layer.pivots]):
            return False
    return True


def pin_forward_equals_dense(forward=oracle.forward, compress=oracle.compress):
    for seed, (m, n, r, T) in enumerate(((64, 48, 20, 7), (96, 40, 32, 5), (50, 50, 50, 3))):
        U, V, rng = random_layer(m, n, r, seed)
        X = inputs.make_activations(rng, T, n, "fp32")
        layer = compress(U, V, r)
        Y = forward(X, layer.Wp, layer.C, layer.pivots, layer.nonpivots)
        Yd = oracle.dense_forward(X, oracle.form_weight(U, V))
        if np.linalg.norm(Y - Yd) > 1e-10 * np.linalg.norm(Yd):
            return False
    return True


# ---------------------------------------------------------------------------------------------
# the tests
# ---------------------------------------------------------------------------------------------
def test_golden_worked_example():
    assert pin_golden_example()


def test_golden_counts():
    g = read_golden("worked_example_5x3_r2.txt")
    m, n, r = int(g["m"][0][0]), int(g["n"][0][0]), int(g["r"][0][0])
    assert oracle.storage_count(m, n, r) == int(g["storage"][0][0])
    assert oracle.storage_count(m, n, r, with_indices=True) == int(g["storage_with_indices"][0][0])
    assert oracle.flop_count(1, m, n, r) == int(g["flops_b1"][0][0])


def test_bruteforce_pivots_greedy():
    assert pin_bruteforce(oracle.select_pivot_rows)


def test_bruteforce_pivots_lapack():
    assert pin_bruteforce(oracle.select_pivot_rows_lapack)


def test_bruteforce_coefficients_exact():
    rng = np.random.default_rng(3)
    done = 0
    for _ in range(20):
        m, n, r = 7, 5, 3
        W = rng.integers(-3, 4, size=(m, r)) @ rng.integers(-3, 4, size=(r, n))
        if np.linalg.matrix_rank(W) != r:
            continue
        layer = oracle.compress_weight(W.astype(np.float64), r)
        Cx = exact_coefficients(W.tolist(), list(layer.pivots), list(layer.nonpivots))
        assert np.allclose(layer.C, np.array([[float(v) for v in row] for row in Cx]),
                           atol=1e-11 * max(1.0, np.abs(layer.C).max()), rtol=0)
        done += 1
    assert done >= 10


def test_zero_row_never_chosen():
    W = np.array([[0, 0, 0], [1, 2, 0], [0, 0, 0], [3, 1, 1], [2, 0, 5]], dtype=np.float64)
    info = oracle.select_pivot_rows(W, 3)
    assert 0 not in info.order and 2 not in info.order


def test_duplicate_rows_lowest_index_once():
    base = np.array([[1.0, 2.0, 2.0], [0.5, -1.0, 0.0], [1.0, 2.0, 2.0], [0.0, 0.0, 1.0]])
    info = oracle.select_pivot_rows(base, 3)
    assert info.order[0] == 0                          # tie between rows 0 and 2 -> row 0
    assert 2 not in info.order                          # its duplicate has zero residual after


def test_rank_one_picks_max_norm_row():
    rng = np.random.default_rng(1)
    u = rng.standard_normal(9)
    v = rng.standard_normal(6)
    W = np.outer(u, v)
    info = oracle.select_pivot_rows(W, 1)
    assert info.order[0] == int(np.argmax(np.abs(u)))


def test_r_equals_m_is_permuted_dense():
    U, V, rng = random_layer(24, 40, 24, 5)
    X = inputs.make_activations(rng, 6, 40, "fp32")
    layer = oracle.compress(U, V, 24)
    assert list(layer.pivots) == list(range(24)) and layer.nonpivots.size == 0
    assert layer.C.shape == (0, 24)
    Y = oracle.forward(X, layer.Wp, layer.C, layer.pivots, layer.nonpivots)
    Yd = oracle.dense_forward(X, oracle.form_weight(U, V))
    assert np.array_equal(Y, Yd)                       # Y_p = X W^T exactly when I = [0, m)


def test_rank_deficient_raises():
    U, V, _ = random_layer(30, 20, 6, 2)
    W = oracle.form_weight(U, V)                       # rank 6
    with pytest.raises(oracle.RankDeficientError):
        oracle.compress_weight(W, 8)
    with pytest.raises(oracle.RankDeficientError):
        oracle.compress_weight(W, 8, "lapack")


def test_lossless():
    assert pin_lossless()


def test_lossless_lapack_rule():
    assert pin_lossless(lambda U, V, r: oracle.compress(U, V, r, "lapack"))


def test_forward_equals_dense():
    assert pin_forward_equals_dense()


def test_closed_form_coefficients():
    """With W' = U V^T and V of full column rank, C = U_np U_p^{-1} (from Eq. 2)."""
    for seed, (m, n, r) in enumerate(((80, 60, 30), (64, 64, 32))):
        U, V, _ = random_layer(m, n, r, seed)
        layer = oracle.compress(U, V, r)
        Cc = np.linalg.solve(U[layer.pivots].T, U[layer.nonpivots].T).T
        assert np.abs(layer.C - Cc).max() <= 1e-10 * max(1.0, np.abs(Cc).max())


def test_pivot_set_invariance():
    """Any r independent rows give a lossless layer; Y does not depend on which were picked."""
    U, V, rng = random_layer(48, 40, 16, 9)
    X = inputs.make_activations(rng, 5, 40, "fp32")
    W = oracle.form_weight(U, V)
    ref = oracle.compress(U, V, 16)
    Y_ref = oracle.forward(X, ref.Wp, ref.C, ref.pivots, ref.nonpivots)
    alt_rng = np.random.default_rng(11)
    for _ in range(3):
        piv = np.sort(alt_rng.choice(48, size=16, replace=False))
        if np.linalg.cond(W[piv]) > 1e6:
            continue
        nonp = oracle.complement(piv, 48)
        C = oracle.solve_coefficients(W[piv], W[nonp])
        Y = oracle.forward(X, W[piv], C, piv, nonp)
        assert np.linalg.norm(Y - Y_ref) <= 1e-9 * np.linalg.norm(Y_ref)


def test_storage_counts():
    for d in (256, 4096, 8192):
        assert oracle.storage_count(d, d, d // 2) == 3 * d * d // 4        # 0.75 d^2 at r = d/2
    m, n, r = 11008, 4096, 2048
    assert oracle.storage_count(m, n, r, True) == r * (m + n) - r * r + r   # Sec. 3.3 formula
    # PIFA stores strictly less than the two-factor low-rank layer, and less than dense for r<min
    for (m, n, r) in ((256, 256, 128), (28672, 8192, 4096), (100, 60, 59)):
        assert oracle.storage_count(m, n, r, True) < r * (m + n)
        assert oracle.storage_count(m, n, r) < m * n


def test_flop_count_matches_instrumented_loop():
    """2 T r (m + n - r) against multiply-adds counted one by one in a naive Algorithm 2."""
    for (T, m, n, r) in ((3, 7, 5, 2), (2, 6, 9, 4), (1, 4, 4, 4)):
        madds = 0
        for _t in range(T):
            for _j in range(r):            # Y_p = W_p x: r outputs of n multiply-adds
                for _k in range(n):
                    madds += 1
            for _i in range(m - r):        # Y_np = C Y_p: m - r outputs of r multiply-adds
                for _j in range(r):
                    madds += 1
        assert oracle.flop_count(T, m, n, r) == 2 * madds


def test_greedy_matches_lapack_medium():
    for seed, (m, n, r) in enumerate(((300, 200, 100), (256, 256, 128), (200, 320, 150))):
        U, V, _ = random_layer(m, n, r, seed)
        W = oracle.form_weight(U, V)
        g = oracle.select_pivot_rows(W, r)
        lp = oracle.select_pivot_rows_lapack(W, r)
        if g.gaps.min() < 1e-9:
            continue
        assert np.array_equal(np.sort(g.order), np.sort(lp.order))


def test_forward_rows_are_independent():
    """Algorithm 2 acts on each token column (row of X) separately: subsets give the same rows."""
    U, V, rng = random_layer(40, 30, 12, 4)
    X = inputs.make_activations(rng, 9, 30, "fp32")
    layer = oracle.compress(U, V, 12)
    Y = oracle.forward(X, layer.Wp, layer.C, layer.pivots, layer.nonpivots)
    rows = [1, 4, 8]
    Ys = oracle.forward(X[rows], layer.Wp, layer.C, layer.pivots, layer.nonpivots)
    assert np.array_equal(Ys, Y[rows])


# ---------------------------------------------------------------------------------------------
# planted mistakes: a plausible slip in the oracle must trip at least one pin
# ---------------------------------------------------------------------------------------------
def _forward_swapped_scatter(X, Wp, C, pivots, nonpivots):
    Yp = np.asarray(X, np.float64) @ np.asarray(Wp).T
    Ynp = Yp @ np.asarray(C).T
    Y = np.empty((Yp.shape[0], len(pivots) + len(nonpivots)))
    Y[:, pivots] = Yp
    Y[:, nonpivots] = np.roll(Ynp, 1, axis=1)          # non-pivot outputs landed one column off
    return Y


def _forward_transposed_c(X, Wp, C, pivots, nonpivots):
    Yp = np.asarray(X, np.float64) @ np.asarray(Wp).T
    Cm = np.asarray(C)
    Ct = Cm.T if Cm.shape[0] == Cm.shape[1] else Cm[:, ::-1]
    Y = np.empty((Yp.shape[0], len(pivots) + len(nonpivots)))
    Y[:, pivots] = Yp
    Y[:, nonpivots] = Yp @ Ct.T
    return Y


def _forward_dropped_term(X, Wp, C, pivots, nonpivots):
    Yp = np.asarray(X, np.float64) @ np.asarray(Wp)[:, :].T
    Yp_short = np.asarray(X, np.float64)[:, 1:] @ np.asarray(Wp)[:, 1:].T   # first input dropped
    Y = np.empty((Yp.shape[0], len(pivots) + len(nonpivots)))
    Y[:, pivots] = Yp_short
    Y[:, nonpivots] = Yp @ np.asarray(C).T
    return Y


def _select_min_norm(W, r):
    """Mutant: picks the smallest nonzero residual instead of the largest."""
    A = np.array(np.asarray(W, np.float64).T)
    n, m = A.shape
    chosen = np.zeros(m, bool)
    order = []
    for k in range(r):
        res = np.sqrt((A[k:] ** 2).sum(0))
        res[chosen] = np.inf
        res[res < 1e-12] = np.inf
        j = int(np.argmin(res))
        x = A[k:, j].copy()
        alpha = -np.copysign(np.linalg.norm(x), x[0] if x[0] else 1.0)
        x[0] -= alpha
        x /= np.linalg.norm(x)
        A[k:] -= 2 * np.outer(x, x @ A[k:])
        chosen[j] = True
        order.append(j)
    return oracle.PivotInfo(np.array(order), np.zeros(r), np.ones(r), 0.0, 1.0)


def _select_sign_slip(W, r):
    """Mutant: Householder update applied with the wrong sign (reflection not orthogonal)."""
    A = np.array(np.asarray(W, np.float64).T)
    n, m = A.shape
    chosen = np.zeros(m, bool)
    order = []
    for k in range(r):
        res = np.sqrt((A[k:] ** 2).sum(0))
        res[chosen] = -1
        j = int(np.argmax(res))
        x = A[k:, j].copy()
        alpha = -np.copysign(np.linalg.norm(x), x[0] if x[0] else 1.0)
        x[0] -= alpha
        x /= np.linalg.norm(x)
        A[k:] += 2 * np.outer(x, x @ A[k:])
        chosen[j] = True
        order.append(j)
    return oracle.PivotInfo(np.array(order), np.zeros(r), np.ones(r), 0.0, 1.0)


def _compress_unsorted(U, V, r):
    """Mutant: C solved against pivots in greedy order but W_p stored in ascending order."""
    W = oracle.form_weight(U, V)
    info = oracle.select_pivot_rows(W, r)
    piv_sorted = np.sort(info.order)
    nonp = oracle.complement(piv_sorted, W.shape[0])
    C = oracle.solve_coefficients(W[info.order], W[nonp])
    return oracle.PifaLayer(piv_sorted, nonp, W[piv_sorted], C, info)


@pytest.mark.parametrize("mutant", [_forward_swapped_scatter, _forward_transposed_c,
                                    _forward_dropped_term])
def test_planted_forward_mistakes_are_caught(mutant):
    assert not (pin_golden_example(forward=mutant) and pin_forward_equals_dense(forward=mutant))


@pytest.mark.parametrize("mutant", [_select_min_norm, _select_sign_slip])
def test_planted_pivot_mistakes_are_caught(mutant):
    assert not pin_bruteforce(mutant)


def test_planted_coefficient_mistake_is_caught():
    assert not pin_lossless(_compress_unsorted)


# ---------------------------------------------------------------------------------------------
# the backward pass (gradients of Algorithm 2 w.r.t. X, W_p and C): pins that do not restate the
# oracle's reverse-order chain rule
# ---------------------------------------------------------------------------------------------
BWD_SHAPES = ((11, 7, 4, 5), (9, 12, 6, 3), (16, 16, 5, 8), (7, 5, 7, 4))   # (m, n, r, T); last: r = m


def _bwd_case(m, n, r, T, seed):
    """A random layer (random ascending I, real W_p and C, not compressed: the gradients hold for
    any operands), X and dY."""
    rng = np.random.default_rng(500 + seed)
    pivots = np.sort(rng.choice(m, size=r, replace=False))
    nonpivots = oracle.complement(pivots, m)
    Wp = rng.standard_normal((r, n))
    C = rng.standard_normal((m - r, r))
    X = rng.standard_normal((T, n))
    dY = rng.standard_normal((T, m))
    return X, Wp, C, pivots, nonpivots, dY, rng


def _safe(pin):
    def run(*a, **k):
        try:
            return bool(pin(*a, **k))
        except (ValueError, IndexError):
            return False
    return run


@_safe
def pin_backward_central_differences(backward=oracle.backward):
    """L = <dY, Y> is linear in each of X, W_p and C (the others fixed), so a central difference
    along any direction E equals <E, dL/d(that input)> up to rounding, whatever the step."""
    for seed, shape in enumerate(BWD_SHAPES):
        X, Wp, C, I, Ic, dY, rng = _bwd_case(*shape, seed)
        dX, dWp, dC = backward(X, Wp, C, I, Ic, dY)
        L = lambda X_, Wp_, C_: float(np.sum(dY * oracle.forward(X_, Wp_, C_, I, Ic)))
        for which, grad, base in ((0, dX, X), (1, dWp, Wp), (2, dC, C)):
            if grad.shape != base.shape:
                return False
            if base.size == 0:
                continue
            E = rng.standard_normal(base.shape)
            args_p = [X, Wp, C]
            args_m = [X, Wp, C]
            args_p[which] = base + E
            args_m[which] = base - E
            fd = (L(*args_p) - L(*args_m)) / 2
            scale = np.linalg.norm(E) * np.linalg.norm(grad) + abs(L(X, Wp, C)) + 1.0
            if abs(fd - float(np.sum(E * grad))) > 1e-11 * scale:
                return False
    return True


@_safe
def pin_backward_euler(backward=oracle.backward):
    """Y is homogeneous of degree one in X and in W_p, and Y_np in C (Euler): <dX, X> = <dY, Y>,
    <dW_p, W_p> = <dY, Y>, <dC, C> = <dY[:, I^c], Y[:, I^c]>."""
    for seed, shape in enumerate(BWD_SHAPES):
        X, Wp, C, I, Ic, dY, _ = _bwd_case(*shape, seed + 10)
        dX, dWp, dC = backward(X, Wp, C, I, Ic, dY)
        Y = oracle.forward(X, Wp, C, I, Ic)
        full = float(np.sum(dY * Y))
        tail = float(np.sum(dY[:, Ic] * Y[:, Ic]))
        tol = 1e-11 * (np.abs(dY).sum() * np.abs(Y).max() + 1.0)
        if abs(float(np.sum(dX * X)) - full) > tol or abs(float(np.sum(dWp * Wp)) - full) > tol:
            return False
        if abs(float(np.sum(dC * C)) - tail) > tol:
            return False
    return True


@_safe
def pin_backward_dense_route(backward=oracle.backward):
    """The same gradients through the dense weight: W'[I] = W_p, W'[I^c] = C W_p (Eqs. 1-2) and
    Y = X W'^T give dX = dY W' and dW' = dY^T X; W_p reaches W' directly and through C, so
    dW_p = dW'[I] + C^T dW'[I^c], and dC = dW'[I^c] W_p^T."""
    for seed, shape in enumerate(BWD_SHAPES):
        X, Wp, C, I, Ic, dY, _ = _bwd_case(*shape, seed + 20)
        m = I.size + Ic.size
        W = np.empty((m, Wp.shape[1]))
        W[I] = Wp
        W[Ic] = C @ Wp
        dW = dY.T @ X
        ref = (dY @ W, dW[I] + C.T @ dW[Ic], dW[Ic] @ Wp.T)
        got = backward(X, Wp, C, I, Ic, dY)
        for g, r_ in zip(got, ref):
            if g.shape != r_.shape or np.linalg.norm(g - r_) > 1e-12 * (np.linalg.norm(r_) + 1.0):
                return False
    return True


def test_backward_central_differences():
    assert pin_backward_central_differences()


def test_backward_euler_identities():
    assert pin_backward_euler()


def test_backward_dense_route():
    assert pin_backward_dense_route()


def test_backward_r_equals_m_is_the_linear_layer_gradient():
    """r = m (C empty): a row-permuted dense layer, whose gradients are the textbook ones."""
    X, Wp, C, I, Ic, dY, _ = _bwd_case(6, 5, 6, 4, 99)
    dX, dWp, dC = oracle.backward(X, Wp, C, I, Ic, dY)
    assert dC.shape == (0, 6)
    np.testing.assert_allclose(dX, dY[:, I] @ Wp, rtol=0, atol=1e-13)
    np.testing.assert_allclose(dWp, dY[:, I].T @ X, rtol=0, atol=1e-13)


def test_backward_on_a_compressed_layer_matches_the_dense_input_gradient():
    """On a layer from Algorithm 1, dX equals the dense layer's input gradient dY W' (lossless)."""
    U, V, rng = random_layer(40, 30, 12, 3)
    layer = oracle.compress(U, V, 12)
    X = rng.standard_normal((6, 30))
    dY = rng.standard_normal((6, 40))
    dX, _, _ = oracle.backward(X, layer.Wp, layer.C, layer.pivots, layer.nonpivots, dY)
    ref = dY @ oracle.form_weight(U, V)
    assert np.linalg.norm(dX - ref) <= 1e-10 * np.linalg.norm(ref)


# planted mistakes in copies of the backward
def _bwd_parts(X, Wp, C, I, Ic, dY):
    X, Wp, C, dY = (np.asarray(a, np.float64) for a in (X, Wp, C, dY))
    return X, Wp, C, dY, X @ Wp.T, dY[:, Ic], dY[:, I].copy()


def _backward_dropped_c_path(X, Wp, C, I, Ic, dY):
    X, Wp, C, dY, Yp, dYnp, dYp = _bwd_parts(X, Wp, C, I, Ic, dY)
    return dYp @ Wp, dYp.T @ X, dYnp.T @ Yp                        # dY_np C never added


def _backward_reversed_c(X, Wp, C, I, Ic, dY):
    X, Wp, C, dY, Yp, dYnp, dYp = _bwd_parts(X, Wp, C, I, Ic, dY)
    dYp = dYp + dYnp[:, ::-1] @ C                                  # rows of C paired with the wrong outputs
    return dYp @ Wp, dYp.T @ X, dYnp.T @ Yp


def _backward_stale_wp(X, Wp, C, I, Ic, dY):
    X, Wp, C, dY, Yp, dYnp, dYp = _bwd_parts(X, Wp, C, I, Ic, dY)
    full = dYp + dYnp @ C
    return full @ Wp, dYp.T @ X, dYnp.T @ Yp                       # dW_p from the pivot outputs only


def _backward_tokens_misaligned(X, Wp, C, I, Ic, dY):
    X, Wp, C, dY, Yp, dYnp, dYp = _bwd_parts(X, Wp, C, I, Ic, dY)
    full = dYp + dYnp @ C
    return full @ Wp, full.T @ X, dYnp.T @ Yp[::-1]                 # dC pairs token t with token T-1-t


@pytest.mark.parametrize("mutant", [_backward_dropped_c_path, _backward_reversed_c, _backward_stale_wp,
                                    _backward_tokens_misaligned])
def test_planted_backward_mistakes_are_caught(mutant):
    assert not (pin_backward_central_differences(mutant) and pin_backward_euler(mutant)
                and pin_backward_dense_route(mutant))
