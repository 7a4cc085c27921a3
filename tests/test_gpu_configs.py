"""GPU parity at the full workload sizes: rollouts (1.3B / 14B shapes) and the warmup path.

Rows of attention are independent, so the fp64 oracle checks sampled query rows of the
full-size launches exactly.  LS sums are checked on independent synthetic activations
(full size for hidden 1536, sampled 128x128 blocks for hidden 5120); the solve and eps are
checked against the oracle's at both hidden sizes (at 5120 on a narrow output weight, with
numpy's Cholesky as the oracle's factorisation step).
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from gpu_helpers import Step, assert_close_attn, assert_disc_close  # noqa: E402
from oracle import attention as at  # noqa: E402
from oracle import ls as ols  # noqa: E402
from paper_2607_00712_gb300 import abi, synth  # noqa: E402
from paper_2607_00712_gb300.device import LS, Window, bf16_tensor, to_f32  # noqa: E402

pytestmark = pytest.mark.gpu

P, D_HEAD, CHUNK = 1560, 128, 3


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2607_00712_gb300.build import build_library
    build_library()
    abi.lib()


def _rows(seed, n_q, k=48):
    rng = np.random.default_rng(seed)
    fixed = [0, 127, 128, n_q - 73, n_q - 1]
    return np.unique(np.concatenate([fixed, rng.choice(n_q, k, replace=False)]))


def _attn_out(st, mode, win=None):
    n, Dm = st.n_q, st.H * st.d
    out = torch.empty(n, Dm, dtype=torch.bfloat16, device="cuda")
    if mode == "full":
        abi.ispa_attn_full(st.ring.c, st.q, st.kc, st.vc, n, 0.0, out)
    else:
        abi.ispa_attn_local(st.ring.c, Window(*win), st.q, st.kc, st.vc, n, 0.0, out)
    torch.cuda.synchronize()
    return to_f32(out).reshape(n, st.H, st.d)


@pytest.mark.parametrize("heads", [12, 40], ids=["1.3B", "14B"])
@pytest.mark.parametrize("step", [1, 10, 20])
def test_rollout_step(heads, step):
    # AR rollout, chunk s has 3(s-1) past frames: F-layers attend to all of them (ring of 60
    # frames), L-layers to the chunk + 6 newest frames held in a 6-frame ring (evicting).
    n_past = CHUNK * (step - 1)
    seed = 1000 * heads + step
    st_f = Step(seed, P=P, H=heads, d=D_HEAD, n_past=n_past, n_chunk_frames=CHUNK, capacity=60)
    rows = _rows(seed, st_f.n_q)
    got = _attn_out(st_f, "full")
    ref, _ = at.attn_full(*st_f.oracle_args(), rows=rows)
    assert_close_attn(got[rows], ref, f"rollout full s={step}")
    del st_f
    torch.cuda.empty_cache()
    st_l = Step(seed, P=P, H=heads, d=D_HEAD, n_past=n_past, n_chunk_frames=CHUNK, capacity=6)
    got = _attn_out(st_l, "local", (0, 6))
    ref, _ = at.attn_local(*st_l.oracle_args(), 0, 6, rows=rows)
    assert_close_attn(got[rows], ref, f"rollout local s={step}")


@pytest.mark.parametrize("heads", [12, 40], ids=["1.3B", "14B"])
def test_warmup_dual_step(heads):
    # Warmup step in steady state: 24 cached frames + the chunk (42120 keys), window 6 frames.
    st = Step(77 + heads, P=P, H=heads, d=D_HEAD, n_past=24, n_chunk_frames=CHUNK, capacity=24)
    n, Dm = st.n_q, st.H * st.d
    a_full = torch.empty(n, Dm, dtype=torch.bfloat16, device="cuda")
    a_loc = torch.empty_like(a_full)
    disc = torch.empty(n, dtype=torch.float32, device="cuda")
    dsum = torch.zeros(1, dtype=torch.float32, device="cuda")
    wsb = abi.ispa_attn_dual_workspace_size(heads, n)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    abi.ispa_attn_dual(st.ring.c, Window(0, 6), st.q, st.kc, st.vc, n, 0.0, a_full, a_loc, disc, dsum, None, None,
                       ws, wsb)
    torch.cuda.synchronize()
    rows = _rows(heads, n)
    r = at.attn_dual(*st.oracle_args(), 0, 6, rows=rows)
    g_full = to_f32(a_full).reshape(n, heads, D_HEAD)
    g_loc = to_f32(a_loc).reshape(n, heads, D_HEAD)
    assert_close_attn(g_full[rows], r["a_full"], "warmup a_full")
    assert_close_attn(g_loc[rows], r["a_loc"], "warmup a_loc")
    g_disc = to_f32(disc)
    assert_disc_close(g_full[rows], g_loc[rows], g_disc[rows], r, "warmup disc")
    # extra: self-consistency of disc and of the device sum over all tokens
    d_own = np.sqrt(((g_full.astype(np.float64) - g_loc) ** 2).reshape(n, -1).sum(1))
    assert np.allclose(g_disc, d_own, rtol=1e-5, atol=1e-5)
    assert abs(float(dsum.item()) - float((d_own ** 2).sum())) <= 1e-4 * float((d_own ** 2).sum())


def _accumulate_gpu(D, batches):
    st = LS(D)
    T = batches[0][0].shape[0]
    wsb = abi.ispa_ls_accumulate_workspace_size(D, T)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    for a, f in batches:
        abi.ispa_ls_accumulate(st.c, bf16_tensor(a), bf16_tensor(f), a.shape[0], ws, wsb)
    torch.cuda.synchronize()
    return st


def test_warmup_ls_hidden1536_full():
    # 8 warmup steps x 4680 tokens at hidden 1536, then the closed-form solve (lambda = 1e-3).
    D, T = 1536, 4680
    batches = [synth.make_activations(500 + s, T, D) for s in range(8)]
    st = _accumulate_gpu(D, batches)
    a = np.concatenate([b[0] for b in batches]).astype(np.float64)
    f = np.concatenate([b[1] for b in batches]).astype(np.float64)
    ref = ols.ls_accumulate(ols.ls_state(D), a, f)
    G, X, S = st.blocks()
    for name, got, want in [("G", G, ref["G"]), ("X", X, ref["X"]), ("S", S, ref["S"])]:
        if name != "X":
            iu = np.triu_indices(D)
            got, want = got[iu], want[iu]
        assert np.linalg.norm(got - want) / np.linalg.norm(want) <= 1e-3, name
    W = synth.make_weight(9, D, D)
    wsb = abi.ispa_ls_solve_workspace_size(D, D)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    dW = torch.empty(D, D, dtype=torch.float32, device="cuda")
    eps = abi.ispa_ls_solve(st.c, torch.from_numpy(W).cuda(), D, 1e-3, dW, ws, wsb)
    dW_ref, eps_ref = ols.ls_solve(ref["G"], ref["X"], ref["S"], W, 1e-3)
    dWg = to_f32(dW).astype(np.float64)
    assert np.linalg.norm(dWg - dW_ref) / np.linalg.norm(dW_ref) <= 1e-3
    assert abs(eps - eps_ref) <= 1e-3 * abs(eps_ref)


def _sym_upper(M):
    """The symmetric matrix whose upper triangle the state maintains."""
    return np.triu(M) + np.triu(M, 1).T


def test_warmup_ls_hidden5120_sums_solve_and_eps():
    # Hidden 5120 (the 14B shape).  G/X/S on sampled 128x128 blocks against the oracle's sums;
    # then the solve and eps on a narrow output weight (d_out = 96), both sides from the SAME
    # accumulated state (the GPU's, read back), so the comparison isolates the solve.
    D, T, D_OUT, LAM = 5120, 10240, 96, 1e-3
    a, f = synth.make_activations(600, T, D)
    st = _accumulate_gpu(D, [(a, f)])
    G, X, S = st.blocks()
    ref = ols.ls_accumulate(ols.ls_state(D), a, f)
    for (i, j) in [(0, 0), (0, 39), (17, 23), (39, 39), (5, 5)]:
        I, J = slice(128 * i, 128 * i + 128), slice(128 * j, 128 * j + 128)
        for name, got, want in [("G", G[I, J], ref["G"][I, J]), ("X", X[I, J], ref["X"][I, J]),
                                ("S", S[I, J], ref["S"][I, J])]:
            assert np.linalg.norm(got - want) / np.linalg.norm(want) <= 1e-3, (name, i, j)
    W = synth.make_weight(10, D, D_OUT)
    wsb = abi.ispa_ls_solve_workspace_size(D, D_OUT)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    dW = torch.empty(D, D_OUT, dtype=torch.float32, device="cuda")
    eps = abi.ispa_ls_solve(st.c, torch.from_numpy(W).cuda(), D_OUT, LAM, dW, ws, wsb)
    dWg = to_f32(dW).astype(np.float64)
    Gs, Ss = _sym_upper(G), _sym_upper(S)
    dW_or, eps_or = ols.ls_solve(Gs, X, Ss, W, LAM, factor=np.linalg.cholesky)
    # dW: both solves are fp64 on the same state; the GPU stores dW in fp32 (relative
    # rounding <= 2^-24 per entry), and fp64 rounding times cond(G + lambda I) (~34 for
    # T = 2D Gaussian rows) stays far below 1e-6
    assert np.linalg.norm(dWg - dW_or) <= 1e-6 * np.linalg.norm(dW_or)
    # normal equations of the GPU's dW: the residual of the exact solution is fp64 noise, so
    # what remains is |G + lambda I| |round_fp32(dW) - dW| <= 2^-24 |G + lambda I| |dW|
    M = Gs + LAM * np.eye(D)
    rhs = X @ W.astype(np.float64)
    res = np.linalg.norm(M @ dWg - rhs)
    bound = 2.0 ** -24 * np.linalg.norm(np.abs(M) @ np.abs(dWg)) + 1e-12 * np.linalg.norm(rhs)
    assert res <= bound, (res, bound)
    # eps (Eq. 6 through its trace form; Sec. 3.3 ranks layers by it): a difference of large
    # terms, each formed in fp64 on both sides; allow 1e-9 of the terms' magnitude
    terms = (abs(np.sum(dW_or * (Gs @ dW_or))) + 2 * abs(np.sum(dW_or * rhs))
             + abs(np.sum(W.astype(np.float64) * (Ss @ W.astype(np.float64)))))
    assert abs(eps - eps_or) <= 1e-9 * terms, (eps, eps_or, terms)
    assert eps_or > 0
    # end to end: the GPU solve of the GPU sums against the oracle's solve of its own sums,
    # within what the 1e-3 bound on the sums allows through cond(G + lambda I)
    dW_e2e, eps_e2e = ols.ls_solve(ref["G"], ref["X"], ref["S"], W, LAM, factor=np.linalg.cholesky)
    assert np.linalg.norm(dWg - dW_e2e) <= 1e-3 * np.linalg.norm(dW_e2e)
    assert abs(eps - eps_e2e) <= 1e-3 * abs(eps_e2e)
