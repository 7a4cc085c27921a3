"""Least-squares absorption: accumulate, solve, feasibility (oracle; fp64).

TEST INFRASTRUCTURE ONLY (see the package docstring).

Paper basis (Sec. 3.2)
  * Eq. 4: min_dW || A_loc (W + dW) - A_full W ||^2 + lambda ||dW||^2, both
    norms read as squared Frobenius norms, row-vector convention A @ W.
  * Eq. 5: with R = (A_full - A_loc) W,
        dW = (A_loc^T A_loc + lambda I)^{-1} A_loc^T R.
  * Eq. 6: eps = || A_loc (W + dW) - A_full W ||_F^2.
  * "summing the outer products ... during the standard forward pass" and "a
    single D x D matrix inversion": the sums are accumulated token by token and
    the system is solved once.  The inverse is applied as a Cholesky solve
    (mathematically the same matrix).
  * lambda = 0.001 by default (Sec. 4.1); it is absolute, applied to the
    unnormalised sums.

Accumulated state (delta = A_full - A_loc per token):
    G = sum a a^T,  X = sum a delta^T,  S = sum delta delta^T,  n = #tokens.
A_loc^T R = X W, formed at solve time; eps expands into traces:
    eps = tr(dW^T G dW) - 2 tr(dW^T X W) + tr(W^T S W).
"""
from __future__ import annotations

import math

import numpy as np


class NotSPD(ValueError):
    pass


def ls_state(D: int) -> dict:
    return dict(G=np.zeros((D, D)), X=np.zeros((D, D)), S=np.zeros((D, D)), n=0)


def ls_accumulate(state: dict, a_loc: np.ndarray, a_full: np.ndarray) -> dict:
    """Add one batch of tokens (rows) of A_loc, A_full [T, D] to the sums."""
    a = np.asarray(a_loc, np.float64).reshape(a_loc.shape[0], -1)
    f = np.asarray(a_full, np.float64).reshape(a_full.shape[0], -1)
    delta = f - a
    state["G"] += a.T @ a
    state["X"] += a.T @ delta
    state["S"] += delta.T @ delta
    state["n"] += a.shape[0]
    return state


def cholesky(M: np.ndarray) -> np.ndarray:
    """Textbook column-by-column Cholesky: M = L L^T, L lower triangular.

    For column j: L_jj = sqrt(M_jj - sum_k<j L_jk^2) and, below the diagonal,
    L_ij = (M_ij - sum_k<j L_ik L_jk) / L_jj.  Raises NotSPD on a non-positive
    pivot.
    """
    M = np.asarray(M, np.float64)
    n = M.shape[0]
    L = np.zeros_like(M)
    for j in range(n):
        piv = M[j, j] - L[j, :j] @ L[j, :j]
        if not piv > 0.0:
            raise NotSPD(f"pivot {j} is {piv}")
        L[j, j] = math.sqrt(piv)
        if j + 1 < n:
            L[j + 1:, j] = (M[j + 1:, j] - L[j + 1:, :j] @ L[j, :j]) / L[j, j]
    return L


def forward_sub(L: np.ndarray, B: np.ndarray) -> np.ndarray:
    """Solve L Y = B for lower-triangular L, row by row."""
    n = L.shape[0]
    Y = np.zeros_like(B, dtype=np.float64)
    for i in range(n):
        Y[i] = (B[i] - L[i, :i] @ Y[:i]) / L[i, i]
    return Y


def back_sub(U: np.ndarray, B: np.ndarray) -> np.ndarray:
    """Solve U Z = B for upper-triangular U, row by row from the bottom."""
    n = U.shape[0]
    Z = np.zeros_like(B, dtype=np.float64)
    for i in range(n - 1, -1, -1):
        Z[i] = (B[i] - U[i, i + 1:] @ Z[i + 1:]) / U[i, i]
    return Z


def ls_solve(G, X, S, W, lam: float = 1e-3, factor=None):
    """Eq. 5 and Eq. 6 from the accumulated sums.

    Returns (dW [D, D_out], eps) with eps from the trace expansion.
    factor: the Cholesky factorisation used for G + lambda I; the textbook one above by
    default.  At hidden sizes where its column loop takes too long on the host (D = 5120)
    a library Cholesky (numpy's LAPACK call) serves as that one step; the two agree to
    rounding (pinned in the oracle's tests).
    """
    G = np.asarray(G, np.float64)
    X = np.asarray(X, np.float64)
    S = np.asarray(S, np.float64)
    W = np.asarray(W, np.float64)
    D = G.shape[0]
    L = (factor or cholesky)(G + lam * np.eye(D))
    rhs = X @ W                               # A_loc^T R
    dW = back_sub(L.T, forward_sub(L, rhs))
    eps = float(np.sum(dW * (G @ dW)) - 2.0 * np.sum(dW * rhs) + np.sum(W * (S @ W)))
    return dW, eps


def eps_direct(a_loc, a_full, W, dW) -> float:
    """Eq. 6 evaluated from the stored tokens."""
    a = np.asarray(a_loc, np.float64)
    f = np.asarray(a_full, np.float64)
    W = np.asarray(W, np.float64)
    r = a @ (W + np.asarray(dW, np.float64)) - f @ W
    return float(np.sum(r * r))


def objective(a_loc, a_full, W, dW, lam: float) -> float:
    """Eq. 4's objective at dW."""
    return eps_direct(a_loc, a_full, W, dW) + lam * float(np.sum(np.asarray(dW) ** 2))
