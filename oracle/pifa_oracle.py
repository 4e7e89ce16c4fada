"""Plain fp64 CPU oracle for the PIFA layer (Pivoting Factorization, Sec. 3.2).

TEST INFRASTRUCTURE ONLY. Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU
baseline (and its reference arm) may import this module. The product path (the C-ABI library
and its binding) never calls it and shares no code with it.

Everything here is deliberately slow and literal: numpy float64, one step of the paper per line
group, library primitives (a matmul, a Householder QR, a triangular solve) used only as whole
steps. Notation follows the paper: W' (m x n, rank r), pivot-row indices I, non-pivot indices I^c,
pivot-row matrix W_p (r x n), coefficient matrix C ((m-r) x r). The paper writes activations as
columns (X in R^{n x b}, Y = W X); here X is row-major (T x n) and Y = X W'^T (T x m) -- the same
map transposed, so Y_p = X W_p^T and Y_np = Y_p C^T.

Functions and the passages they follow:
  form_weight          Sec. 3.2: W' = U V^T.
  select_pivot_rows    Algorithm 1, step 1 (Sec. 3.2): QR with column pivoting (Businger-Golub)
                       applied to W'^T, greedy, residual norms recomputed exactly every step,
                       ties to the lowest row index.
  select_pivot_rows_lapack  the same step through LAPACK's pivoted QR (dgeqp3) -- a library
                       routine for that step, used where the plain loop is too slow.
  compress             Algorithm 1 (Sec. 3.2, Eqs. 1-2): I, I^c, W_p, W_np and C from
                       W_np = C W_p solved by least squares (Householder QR + back substitution).
  forward              Algorithm 2 (Sec. 3.2): Y_p, Y_np and the two index assignments.
  backward             the gradients of Algorithm 2 w.r.t. X, W_p and C (fine-tuning after
                       pruning, Sec. 5.1; differentiability, Sec. 6): its steps in reverse.
  m_accumulate         Algorithm 3 (MPIFA), part 1, the two accumulation steps (Sec. 4): the sums
                       of x_u x_u^T and of y_t x_u^T over calibration samples, y_t the mixed target
                       of Eq. 6 (lambda W x_o + (1 - lambda) W x_u), one sample at a time.
  m_reconstruct        Algorithm 3, part 1, the two reconstruction steps: U_r by Eq. 4 (the online
                       form of Eq. 3) and V_r^T by Eq. 8 (Eq. 7 with the alpha regulariser).
  storage_count        Sec. 3.3 (memory cost): r(m+n) - r^2 (+ r indices).
  flop_count           Sec. 3.3 (computational cost): 2 b r (m + n - r).
  dense_forward, lowrank_forward  the two comparison layers of Sec. 3.3 (Y = W X, Y = U V^T X).

Readings where the paper is silent are listed in the repository's design notes; in short: the
pivot search runs on W'^T because column pivoting selects columns; ties go to the lowest index;
I and I^c are kept in ascending order, which fixes the row order of W_p and the column order of C.
"""
from __future__ import annotations

import dataclasses

import numpy as np
import scipy.linalg


class RankDeficientError(ValueError):
    """W' has fewer than r linearly independent rows (Algorithm 1 assumes rank exactly r)."""


@dataclasses.dataclass
class PivotInfo:
    order: np.ndarray        # pivot rows in the order the greedy search picked them
    gaps: np.ndarray         # per step: (best - runner_up) / best of the residual norms
    r_diag: np.ndarray       # |R_kk| of the pivoted QR, k = 0..r-1
    residual_after: float    # largest residual row norm left after r steps
    max_initial: float       # largest row norm of W'


@dataclasses.dataclass
class PifaLayer:
    pivots: np.ndarray       # I, int64, ascending, length r
    nonpivots: np.ndarray    # I^c, int64, ascending, length m - r
    Wp: np.ndarray           # W_p = W'[I, :], float64 (r x n)
    C: np.ndarray            # C with W_np = C W_p, float64 ((m - r) x r)
    info: PivotInfo


# ---------------------------------------------------------------------------------------------
# Sec. 3.2: the singular matrix W' = U V^T
# ---------------------------------------------------------------------------------------------
def form_weight(U, V) -> np.ndarray:
    """W' = U V^T in float64 (Sec. 3.2, first step of the PIFA process)."""
    U = np.asarray(U, dtype=np.float64)
    V = np.asarray(V, dtype=np.float64)
    return U @ V.T


# ---------------------------------------------------------------------------------------------
# Algorithm 1, step 1: pivot rows by QR with column pivoting on W'^T
# ---------------------------------------------------------------------------------------------
def select_pivot_rows(W, r: int, rank_tol: float = 1e-10, diag_tol: float = 1e-8) -> PivotInfo:
    """Greedy Businger-Golub pivoted QR of A = W'^T; returns the r chosen rows of W'.

    Column j of A is row j of W'. At step k the k columns chosen so far have been reduced by
    Householder reflections H_k ... H_1, so rows k.. of the reflected A hold each column's
    component orthogonal to the chosen ones. The next pivot is the column with the largest such
    residual norm, recomputed from scratch from the reflected matrix every step (no norm
    downdating); among equal norms the lowest index wins.
    """
    A = np.array(np.asarray(W, dtype=np.float64).T, copy=True)   # n x m
    n, m = A.shape
    if not (1 <= r <= min(m, n)):
        raise ValueError(f"need 1 <= r <= min(m, n); got r={r}, m={m}, n={n}")
    max_initial = float(np.sqrt((A * A).sum(axis=0)).max()) if m else 0.0
    chosen = np.zeros(m, dtype=bool)
    order, gaps, r_diag = [], [], []
    for k in range(r):
        res = np.sqrt((A[k:, :] * A[k:, :]).sum(axis=0))
        res[chosen] = -1.0
        best = res.max()
        j = int(np.flatnonzero(res == best)[0])          # lowest index among ties
        others = np.delete(res, j)
        runner = others.max() if others.size else -1.0
        gaps.append((best - max(runner, 0.0)) / best if best > 0 else 0.0)
        # Householder reflection zeroing A[k+1:, j]
        x = A[k:, j].copy()
        alpha = -np.copysign(np.linalg.norm(x), x[0] if x[0] != 0 else 1.0)
        v = x
        v[0] -= alpha
        vnorm = np.linalg.norm(v)
        if vnorm > 0:
            v /= vnorm
            A[k:, :] -= 2.0 * np.outer(v, v @ A[k:, :])
        chosen[j] = True
        order.append(j)
        r_diag.append(abs(alpha))
    res = np.sqrt((A[r:, :] * A[r:, :]).sum(axis=0)) if r < n else np.zeros(m)
    res[chosen] = 0.0
    residual_after = float(res.max()) if m > r else 0.0
    info = PivotInfo(np.array(order, dtype=np.int64), np.array(gaps), np.array(r_diag),
                     residual_after, max_initial)
    _check_rank(info, r, rank_tol, diag_tol)
    return info


def select_pivot_rows_lapack(W, r: int, rank_tol: float = 1e-10, diag_tol: float = 1e-8) -> PivotInfo:
    """Algorithm 1, step 1 through LAPACK's pivoted QR (dgeqp3) of W'^T; first r pivots.

    dgeqp3 is the library form of the same Businger-Golub rule (it downdates norms and
    recomputes them when cancellation is detected); gaps are not available from it.
    """
    W = np.asarray(W, dtype=np.float64)
    m, n = W.shape
    if not (1 <= r <= min(m, n)):
        raise ValueError(f"need 1 <= r <= min(m, n); got r={r}, m={m}, n={n}")
    R, P = scipy.linalg.qr(W.T, mode="r", pivoting=True)
    order = np.asarray(P[:r], dtype=np.int64)
    d = np.abs(np.diag(R))
    residual_after = float(d[r]) if r < min(m, n) else 0.0
    max_initial = float(np.sqrt((W * W).sum(axis=1)).max())
    info = PivotInfo(order, np.full(r, np.nan), d[:r].copy(), residual_after, max_initial)
    _check_rank(info, r, rank_tol, diag_tol)
    return info


def _check_rank(info: PivotInfo, r: int, rank_tol: float, diag_tol: float) -> None:
    """W' must have rank exactly r: r clear pivots, nothing left after them (Algorithm 1 input)."""
    if info.max_initial == 0 or info.r_diag[r - 1] < diag_tol * info.r_diag[0]:
        raise RankDeficientError(
            f"|R_(r-1,r-1)| = {info.r_diag[r - 1]:.3e} < {diag_tol} * |R_00| = {info.r_diag[0]:.3e}")
    if info.residual_after > rank_tol * info.max_initial:
        raise RankDeficientError(
            f"residual {info.residual_after:.3e} after r={r} pivots exceeds {rank_tol} * max row norm")


# ---------------------------------------------------------------------------------------------
# Algorithm 1: the PIFA layer (I, W_p, C)
# ---------------------------------------------------------------------------------------------
def complement(pivots, m: int) -> np.ndarray:
    """I^c = {0..m-1} minus I, ascending (Algorithm 1, step 2)."""
    mask = np.ones(m, dtype=bool)
    mask[np.asarray(pivots, dtype=np.int64)] = False
    return np.flatnonzero(mask).astype(np.int64)


def solve_coefficients(Wp, Wnp) -> np.ndarray:
    """C from W_np = C W_p (Eq. 2; Algorithm 1, step 5) as a least-squares solve.

    Transposed, the system is W_p^T C^T = W_np^T with W_p^T of size n x r and full column rank.
    Householder QR W_p^T = Q R (library), then C^T = R^{-1} Q^T W_np^T (back substitution).
    The system is consistent for a rank-r W', so the least-squares solution is the exact C.
    """
    Wp = np.asarray(Wp, dtype=np.float64)
    Wnp = np.asarray(Wnp, dtype=np.float64)
    r = Wp.shape[0]
    if Wnp.shape[0] == 0:
        return np.zeros((0, r))
    Q, R = np.linalg.qr(Wp.T, mode="reduced")
    Ct = scipy.linalg.solve_triangular(R, Q.T @ Wnp.T, lower=False)
    return Ct.T


def compress(U, V, r: int, pivot_rule: str = "greedy") -> PifaLayer:
    """Algorithm 1 on W' = U V^T: I, I^c (ascending), W_p = W'[I], C with W_np = C W_p.

    ``pivot_rule`` picks the implementation of step 1: 'greedy' (select_pivot_rows, the plain loop)
    or 'lapack' (select_pivot_rows_lapack). Both implement QR with column pivoting on W'^T.
    """
    W = form_weight(U, V)
    return compress_weight(W, r, pivot_rule)


def compress_weight(W, r: int, pivot_rule: str = "greedy") -> PifaLayer:
    """Algorithm 1 on an explicit rank-r W' (m x n)."""
    W = np.asarray(W, dtype=np.float64)
    m = W.shape[0]
    if pivot_rule == "greedy":
        info = select_pivot_rows(W, r)
    elif pivot_rule == "lapack":
        info = select_pivot_rows_lapack(W, r)
    else:
        raise ValueError(pivot_rule)
    pivots = np.sort(info.order)                       # step 1 result, kept ascending
    nonpivots = complement(pivots, m)                  # step 2
    Wp = W[pivots, :].copy()                           # step 3 (Eq. 1)
    Wnp = W[nonpivots, :]                              # step 4 (Eq. 1)
    C = solve_coefficients(Wp, Wnp)                    # step 5 (Eq. 2)
    return PifaLayer(pivots, nonpivots, Wp, C, info)


# ---------------------------------------------------------------------------------------------
# Algorithm 2: the PIFA layer forward pass
# ---------------------------------------------------------------------------------------------
def forward(X, Wp, C, pivots, nonpivots) -> np.ndarray:
    """Algorithm 2 in float64 with row-major activations X (T x n); returns Y (T x m).

    Y_p = X W_p^T (step 2), Y_np = Y_p C^T (step 3), Y[:, I] = Y_p (step 4),
    Y[:, I^c] = Y_np (step 5).
    """
    X = np.asarray(X, dtype=np.float64)
    Wp = np.asarray(Wp, dtype=np.float64)
    C = np.asarray(C, dtype=np.float64)
    pivots = np.asarray(pivots, dtype=np.int64)
    nonpivots = np.asarray(nonpivots, dtype=np.int64)
    m = pivots.size + nonpivots.size
    Yp = X @ Wp.T
    Ynp = Yp @ C.T
    Y = np.empty((X.shape[0], m), dtype=np.float64)
    Y[:, pivots] = Yp
    Y[:, nonpivots] = Ynp
    return Y


def backward(X, Wp, C, pivots, nonpivots, dY):
    """Gradients of Algorithm 2 with respect to its three real inputs, in float64.

    The paper fine-tunes pruned layers, PIFA layers accelerating the backward pass as well as the
    forward (Sec. 5.1, fine-tuning after pruning), and calls PIFA fully differentiable (Sec. 6);
    the trainable inputs are X, W_p and C, the index sets stay fixed. Given dY = dL/dY (T x m), this takes the
    chain rule back through Algorithm 2's steps in reverse order:
      steps 5, 4: dY_np = dY[:, I^c], dY_p = dY[:, I]          (the two index assignments)
      step 3:     Y_np = Y_p C^T  ->  dC = dY_np^T Y_p,  dY_p += dY_np C
      step 2:     Y_p = X W_p^T   ->  dW_p = dY_p^T X,   dX = dY_p W_p
    Y_p is recomputed from X and W_p (step 2). Returns (dX (T x n), dW_p (r x n), dC ((m-r) x r)).
    """
    X = np.asarray(X, dtype=np.float64)
    Wp = np.asarray(Wp, dtype=np.float64)
    C = np.asarray(C, dtype=np.float64)
    dY = np.asarray(dY, dtype=np.float64)
    pivots = np.asarray(pivots, dtype=np.int64)
    nonpivots = np.asarray(nonpivots, dtype=np.int64)
    Yp = X @ Wp.T                      # step 2, recomputed
    dYnp = dY[:, nonpivots]            # step 5 reversed
    dYp = dY[:, pivots].copy()         # step 4 reversed
    dC = dYnp.T @ Yp                   # step 3 reversed
    dYp += dYnp @ C
    dWp = dYp.T @ X                    # step 2 reversed
    dX = dYp @ Wp
    return dX, dWp, dC


# ---------------------------------------------------------------------------------------------
# Sec. 4 / Algorithm 3: the online accumulators of the M reconstruction and its two solves
# ---------------------------------------------------------------------------------------------
def m_accumulate(Xo, Xu, W, lam, XXt=None, YtXt=None, rows=None):
    """The accumulation steps of Algorithm 3 over one calibration batch, in float64.

    Rows of Xo and Xu are samples (the paper's columns x_o^i, x_u^i of X_o, X_u); W is the dense
    m x n weight. For every sample i, in order:
      XXt  += x_u^i (x_u^i)^T                                        (n x n)
      YtXt += (lambda W x_o^i + (1 - lambda) W x_u^i) (x_u^i)^T      (m x n; Eq. 6 target)
    Existing accumulators are continued (the online form: memory independent of the sample count).
    `rows` restricts both accumulators to those rows (for large shapes); the result then has
    len(rows) rows. Returns (XXt, YtXt).
    """
    Xo = np.asarray(Xo, dtype=np.float64)
    Xu = np.asarray(Xu, dtype=np.float64)
    W = np.asarray(W, dtype=np.float64)
    n, m = Xu.shape[1], W.shape[0]
    rx = np.arange(n) if rows is None else np.asarray(rows[0])
    ry = np.arange(m) if rows is None else np.asarray(rows[1])
    XXt = np.zeros((rx.size, n)) if XXt is None else np.array(XXt, dtype=np.float64, copy=True)
    YtXt = np.zeros((ry.size, n)) if YtXt is None else np.array(YtXt, dtype=np.float64, copy=True)
    for i in range(Xu.shape[0]):
        xu, xo = Xu[i], Xo[i]
        XXt += np.outer(xu[rx], xu)
        yt = lam * (W[ry] @ xo) + (1.0 - lam) * (W[ry] @ xu)
        YtXt += np.outer(yt, xu)
    return XXt, YtXt


def m_reconstruct(XXt, YtXt, V, W=None, alpha=0.0):
    """The reconstruction steps of Algorithm 3 from the accumulators, in float64.

    U_r = (Y_t X^T) V (V^T (X X^T) V)^{-1}                                      (Eq. 4)
    V_r^T = (U_r^T U_r)^{-1} U_r^T (Y_t X^T + alpha W) (X X^T + alpha I)^{-1}   (Eq. 8; alpha = 0
                                                                                  gives Eq. 7)
    V is n x r (the paper's V, W ~ U V^T). Returns (U_r (m x r), V_r (n x r)); linear solves, no
    explicit inverses.
    """
    XXt = np.asarray(XXt, dtype=np.float64)
    YtXt = np.asarray(YtXt, dtype=np.float64)
    V = np.asarray(V, dtype=np.float64)
    S = V.T @ XXt @ V                                  # r x r
    U_r = np.linalg.solve(S.T, (YtXt @ V).T).T        # (Y_t X^T V) S^{-1}
    n = XXt.shape[0]
    rhs = YtXt + (alpha * np.asarray(W, dtype=np.float64) if alpha else 0.0)
    G = XXt + alpha * np.eye(n)
    left = np.linalg.solve(U_r.T @ U_r, U_r.T @ rhs)   # (U_r^T U_r)^{-1} U_r^T (...)   r x n
    Vt = np.linalg.solve(G.T, left.T).T                 # (...) (X X^T + alpha I)^{-1}
    return U_r, Vt.T


def dense_forward(X, W) -> np.ndarray:
    """The dense layer of Sec. 3.3 (Y = W X), row-major: Y = X W^T."""
    return np.asarray(X, dtype=np.float64) @ np.asarray(W, dtype=np.float64).T


def lowrank_forward(X, U, V) -> np.ndarray:
    """The two-factor low-rank layer of Sec. 3.3 (Y = U (V^T X)), row-major: Y = (X V) U^T."""
    X = np.asarray(X, dtype=np.float64)
    return (X @ np.asarray(V, dtype=np.float64)) @ np.asarray(U, dtype=np.float64).T


# ---------------------------------------------------------------------------------------------
# Sec. 3.3: memory and computational cost
# ---------------------------------------------------------------------------------------------
def storage_count(m: int, n: int, r: int, with_indices: bool = False) -> int:
    """Stored elements of a PIFA layer: W_p (r n) + C ((m - r) r) [+ I (r)] (Sec. 3.3).

    r n + (m - r) r = r(m + n) - r^2; with the r pivot indices, r(m + n) - r^2 + r.
    """
    count = r * n + (m - r) * r
    return count + r if with_indices else count


def flop_count(T: int, m: int, n: int, r: int) -> int:
    """FLOPs of one PIFA forward over T tokens: 2 T r n + 2 T r (m - r) = 2 T r (m + n - r)."""
    return 2 * T * r * n + 2 * T * r * (m - r)


def lossless_error(W, layer: PifaLayer) -> float:
    """||C W_p - W_np||_F / ||W'||_F: how far the layer is from Eq. 2 holding exactly."""
    W = np.asarray(W, dtype=np.float64)
    Wnp = W[layer.nonpivots, :]
    num = np.linalg.norm(layer.C @ layer.Wp - Wnp) if Wnp.size else 0.0
    return float(num / np.linalg.norm(W))
