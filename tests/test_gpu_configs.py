"""GPU parity at the full workload sizes: rollouts (1.3B / 14B shapes) and the warmup path.

Rows of attention are independent, so the fp64 oracle checks sampled query rows of the
full-size launches exactly.  LS sums are checked on independent synthetic activations
(full size for hidden 1536, sampled 128x128 blocks for hidden 5120); the solve is checked
against the oracle at hidden 1536 and through its normal equations at hidden 5120.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from gpu_helpers import Step, assert_close_attn  # noqa: E402
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
    d_own = np.sqrt(((g_full.astype(np.float64) - g_loc) ** 2).reshape(n, -1).sum(1))
    assert np.allclose(to_f32(disc), d_own, rtol=1e-5, atol=1e-5)
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


def test_warmup_ls_hidden5120_sampled_blocks_and_normal_equations():
    # Hidden 5120: G/X/S on sampled 128x128 blocks (each computed by the oracle from its own
    # column slices), and the solve through the normal equations with the oracle's sums.
    D, T = 5120, 10240
    a, f = synth.make_activations(600, T, D)
    st = _accumulate_gpu(D, [(a, f)])
    G, X, S = st.blocks()
    a64, d64 = a.astype(np.float64), f.astype(np.float64) - a.astype(np.float64)
    for (i, j) in [(0, 0), (0, 39), (17, 23), (39, 39), (5, 5)]:
        I, J = slice(128 * i, 128 * i + 128), slice(128 * j, 128 * j + 128)
        for name, got, want in [("G", G[I, J], a64[:, I].T @ a64[:, J]), ("X", X[I, J], a64[:, I].T @ d64[:, J]),
                                ("S", S[I, J], d64[:, I].T @ d64[:, J])]:
            assert np.linalg.norm(got - want) / np.linalg.norm(want) <= 1e-3, (name, i, j)
    W = synth.make_weight(10, D, D)
    wsb = abi.ispa_ls_solve_workspace_size(D, D)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    dW = torch.empty(D, D, dtype=torch.float32, device="cuda")
    abi.ispa_ls_solve(st.c, torch.from_numpy(W).cuda(), D, 1e-3, dW, ws, wsb)
    dWg = to_f32(dW).astype(np.float64)
    Gref = a64.T @ a64
    Xref = a64.T @ d64
    rhs = Xref @ W.astype(np.float64)
    res = (Gref + 1e-3 * np.eye(D)) @ dWg - rhs
    assert np.linalg.norm(res) / np.linalg.norm(rhs) <= 1e-3
