"""Pins for oracle.ls: normal equations, planted recovery, ridge equivalence, Cholesky."""
import numpy as np
import pytest

from oracle import ls


def _planted(seed, T, D, D_out, noise=0.0):
    """Exactly realisable instance: delta = A dW* W^+, so R = delta W = A dW*.

    W has full column rank, so its pseudo-inverse W^+ satisfies W^+ W = I.
    """
    r = np.random.default_rng(seed)
    A = r.standard_normal((T, D))
    W = r.standard_normal((D, D_out)) / np.sqrt(D) + np.eye(D, D_out)
    dW_star = r.standard_normal((D, D_out)) * 0.1
    delta = A @ dW_star @ np.linalg.pinv(W)                    # delta W = A dW*
    delta += noise * r.standard_normal(delta.shape)
    return A, A + delta, W, dW_star


def _state(a_loc, a_full, batches=1):
    st = ls.ls_state(a_loc.shape[1])
    for part in np.array_split(np.arange(a_loc.shape[0]), batches):
        ls.ls_accumulate(st, a_loc[part], a_full[part])
    return st


def test_accumulate_sums():
    r = np.random.default_rng(0)
    a, f = r.standard_normal((50, 6)), r.standard_normal((50, 6))
    st = _state(a, f)
    d = f - a
    # token-by-token outer products (the paper's "summing the outer products")
    G = sum(np.outer(a[t], a[t]) for t in range(50))
    X = sum(np.outer(a[t], d[t]) for t in range(50))
    S = sum(np.outer(d[t], d[t]) for t in range(50))
    assert np.allclose(st["G"], G, atol=1e-12) and np.allclose(st["X"], X, atol=1e-12)
    assert np.allclose(st["S"], S, atol=1e-12) and st["n"] == 50


def test_accumulate_is_additive():
    r = np.random.default_rng(1)
    a, f = r.standard_normal((97, 9)), r.standard_normal((97, 9))
    s1, s5 = _state(a, f, 1), _state(a, f, 5)
    for key in "GXS":
        assert np.allclose(s1[key], s5[key], atol=1e-12)
    assert np.array_equal(s1["G"], s1["G"].T) or np.allclose(s1["G"], s1["G"].T, atol=1e-13)


@pytest.mark.parametrize("lam", [0.0, 1e-3, 1.0])
def test_normal_equations_residual(lam):
    r = np.random.default_rng(2)
    a, f = r.standard_normal((300, 24)), r.standard_normal((300, 24))
    W = r.standard_normal((24, 20))
    st = _state(a, f)
    dW, _ = ls.ls_solve(st["G"], st["X"], st["S"], W, lam)
    lhs = (st["G"] + lam * np.eye(24)) @ dW
    rhs = st["X"] @ W
    assert np.linalg.norm(lhs - rhs) / np.linalg.norm(rhs) <= 1e-10


def test_planted_recovery_exact():
    A, F, W, dW_star = _planted(3, 400, 32, 32)
    st = _state(A, F)
    dW, eps = ls.ls_solve(st["G"], st["X"], st["S"], W, 0.0)
    assert np.max(np.abs(dW - dW_star)) < 1e-9
    ref = float(np.sum((A @ W) ** 2))                # scale of the problem
    assert abs(eps) < 1e-9 * ref
    assert ls.eps_direct(A, F, W, dW) < 1e-15 * ref


def test_planted_recovery_ridge_bias_bound():
    # With lambda > 0: dW = (G + lam I)^{-1} G dW*, so ||dW - dW*|| <= lam/(s_min + lam) ||dW*||.
    A, F, W, dW_star = _planted(4, 400, 32, 16)
    st = _state(A, F)
    lam = 1e-3
    dW, _ = ls.ls_solve(st["G"], st["X"], st["S"], W, lam)
    s_min = np.linalg.eigvalsh(st["G"]).min()
    bound = lam / (s_min + lam) * np.linalg.norm(dW_star)
    assert np.linalg.norm(dW - dW_star) <= bound * (1 + 1e-6)
    assert np.linalg.norm(dW - dW_star) > 0


def test_large_lambda_shrinks_to_zero():
    A, F, W, _ = _planted(5, 200, 16, 16, noise=0.1)
    st = _state(A, F)
    rhs = np.linalg.norm(st["X"] @ W)
    for lam in (1e6, 1e9):
        dW, eps = ls.ls_solve(st["G"], st["X"], st["S"], W, lam)
        assert np.linalg.norm(dW) <= rhs / lam * (1 + 1e-9)
    # eps tends to ||delta W||^2 = tr(W^T S W) (nothing absorbed)
    dW, eps = ls.ls_solve(st["G"], st["X"], st["S"], W, 1e12)
    assert abs(eps - np.sum(W * (st["S"] @ W))) < 1e-6 * eps


def test_ridge_matches_augmented_least_squares():
    # Eq. 4 as an ordinary least-squares problem on [A; sqrt(lam) I] dW = [R; 0].
    r = np.random.default_rng(6)
    T, D, Do = 120, 10, 7
    a, f = r.standard_normal((T, D)), r.standard_normal((T, D))
    W = r.standard_normal((D, Do))
    lam = 0.37
    st = _state(a, f)
    dW, eps = ls.ls_solve(st["G"], st["X"], st["S"], W, lam)
    R = (f - a) @ W
    big = np.vstack([a, np.sqrt(lam) * np.eye(D)])
    tgt = np.vstack([R, np.zeros((D, Do))])
    dW_ls = np.linalg.lstsq(big, tgt, rcond=None)[0]
    assert np.allclose(dW, dW_ls, atol=1e-11)
    assert abs(eps - ls.eps_direct(a, f, W, dW)) < 1e-9 * max(1.0, eps)


def test_solution_is_a_minimum():
    r = np.random.default_rng(7)
    a, f = r.standard_normal((80, 8)), r.standard_normal((80, 8))
    W = r.standard_normal((8, 8))
    lam = 1e-3
    st = _state(a, f)
    dW, _ = ls.ls_solve(st["G"], st["X"], st["S"], W, lam)
    base = ls.objective(a, f, W, dW, lam)
    for _ in range(10):
        E = r.standard_normal(dW.shape) * 1e-3
        assert ls.objective(a, f, W, dW + E, lam) > base


def test_eps_trace_equals_direct():
    r = np.random.default_rng(8)
    a, f = r.standard_normal((64, 12)), r.standard_normal((64, 12))
    W = r.standard_normal((12, 9))
    st = _state(a, f)
    dW, eps = ls.ls_solve(st["G"], st["X"], st["S"], W, 1e-3)
    assert abs(eps - ls.eps_direct(a, f, W, dW)) <= 1e-10 * ls.eps_direct(a, f, W, dW)


def test_cholesky_against_library_and_reconstruction():
    r = np.random.default_rng(9)
    B = r.standard_normal((40, 40))
    M = B @ B.T + 40 * np.eye(40)
    L = ls.cholesky(M)
    assert np.allclose(np.tril(L), L)
    assert np.allclose(L @ L.T, M, atol=1e-11)
    assert np.allclose(L, np.linalg.cholesky(M), atol=1e-11)


def test_cholesky_rejects_indefinite():
    M = np.array([[1.0, 2.0], [2.0, 1.0]])
    with pytest.raises(ls.NotSPD):
        ls.cholesky(M)


def test_triangular_solves_against_library():
    r = np.random.default_rng(10)
    L = np.tril(r.standard_normal((15, 15))) + 5 * np.eye(15)
    B = r.standard_normal((15, 4))
    assert np.allclose(ls.forward_sub(L, B), np.linalg.solve(L, B), atol=1e-12)
    assert np.allclose(ls.back_sub(L.T, B), np.linalg.solve(L.T, B), atol=1e-12)


def test_solve_with_library_factor_matches_textbook():
    # the library Cholesky used at hidden 5120 gives the textbook path's dW and eps
    r = np.random.default_rng(11)
    a, f = r.standard_normal((400, 48)), r.standard_normal((400, 48))
    W = r.standard_normal((48, 7))
    st = _state(a, f)
    dW0, e0 = ls.ls_solve(st["G"], st["X"], st["S"], W, 1e-3)
    dW1, e1 = ls.ls_solve(st["G"], st["X"], st["S"], W, 1e-3, factor=np.linalg.cholesky)
    assert np.linalg.norm(dW1 - dW0) <= 1e-12 * np.linalg.norm(dW0)
    assert abs(e1 - e0) <= 1e-10 * abs(e0)
    # and still satisfies the normal equations to the oracle's bound
    rhs = st["X"] @ W
    assert np.linalg.norm((st["G"] + 1e-3 * np.eye(48)) @ dW1 - rhs) / np.linalg.norm(rhs) <= 1e-10
