"""GPU parity: the paper-literal decomposed dual pass (Eq. 9-12) and the transition steps
(weight injection, permanent eviction of an L-layer's history)."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from gpu_helpers import Step, assert_close_attn, assert_disc_close  # noqa: E402
from oracle import attention as at  # noqa: E402
from oracle import keysets as ks  # noqa: E402
from paper_2607_00712_gb300 import abi, synth  # noqa: E402
from paper_2607_00712_gb300.device import Ring, Window, bf16_tensor, to_f32  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2607_00712_gb300.build import build_library
    build_library()
    abi.lib()


def _branch(st, fn, *args):
    out = torch.empty(st.n_q, st.H * st.d, dtype=torch.bfloat16, device="cuda")
    lse = torch.empty(st.H, st.n_q, dtype=torch.float32, device="cuda")
    fn(*args, out, lse)
    return out, lse


@pytest.mark.parametrize("win", [(0, 2), (1, 1), (1, 3)])
def test_decomposed_dual_matches_oracle(win):
    # Eq. 9: local branch, Eq. 10: history branch, Eq. 11-12: LSE fusion -> A_full.
    st = Step(31, P=100, H=3, d=128, n_past=9, n_chunk_frames=3, capacity=8, n_sink_pinned=1)
    o_loc, l_loc = _branch(st, lambda o, l: abi.ispa_attn_local(st.ring.c, Window(*win), st.q, st.kc, st.vc,
                                                                   st.n_q, 0.0, o, l))
    o_hist, l_hist = _branch(st, lambda o, l: abi.ispa_attn_hist(st.ring.c, Window(*win), st.q, st.n_q, 0.0, o, l))
    fused = torch.empty_like(o_loc)
    lse = torch.empty_like(l_loc)
    abi.ispa_lse_merge(o_loc, l_loc, o_hist, l_hist, st.n_q, st.H, st.d, fused, lse)
    torch.cuda.synchronize()
    args = st.oracle_args()
    r_hist, rl_hist = at.attn_hist(st.s.q, st.k_hist_res, st.v_hist_res, st.P, *win)
    assert_close_attn(to_f32(o_hist).reshape(r_hist.shape), r_hist, "history branch")
    assert np.abs(to_f32(l_hist) - rl_hist).max() < 2e-3
    r_full, rl_full = at.attn_full(*args)
    assert_close_attn(to_f32(fused).reshape(r_full.shape), r_full, "decomposed A_full")
    assert np.abs(to_f32(lse) - rl_full).max() < 2e-3
    # the decomposed pass's discrepancy (Sec. 3.1 phase 1) from its two stored outputs
    disc = torch.empty(st.n_q, dtype=torch.float32, device="cuda")
    dsum = torch.zeros(1, dtype=torch.float32, device="cuda")
    abi.ispa_discrepancy(fused, o_loc, st.n_q, st.H * st.d, disc, dsum)
    torch.cuda.synchronize()
    r = at.attn_dual(*args, *win)
    g_full = to_f32(fused).reshape(r_full.shape)
    g_loc = to_f32(o_loc).reshape(r_full.shape)
    assert_disc_close(g_full, g_loc, to_f32(disc), r, "decomposed disc", float(dsum.item()))


def test_decomposed_dual_empty_history():
    # window covers the cache: the history branch is empty (O = 0, LSE = -inf) and the merge
    # returns the local branch unchanged.
    st = Step(32, P=64, H=2, d=64, n_past=3, n_chunk_frames=2, capacity=4)
    o_loc, l_loc = _branch(st, lambda o, l: abi.ispa_attn_local(st.ring.c, Window(0, 3), st.q, st.kc, st.vc,
                                                                   st.n_q, 0.0, o, l))
    o_hist, l_hist = _branch(st, lambda o, l: abi.ispa_attn_hist(st.ring.c, Window(0, 3), st.q, st.n_q, 0.0, o, l))
    fused = torch.empty_like(o_loc)
    lse = torch.empty_like(l_loc)
    abi.ispa_lse_merge(o_loc, l_loc, o_hist, l_hist, st.n_q, st.H, st.d, fused, lse)
    torch.cuda.synchronize()
    assert np.all(to_f32(o_hist) == 0) and np.all(np.isneginf(to_f32(l_hist)))
    assert np.array_equal(to_f32(fused), to_f32(o_loc))
    assert np.allclose(to_f32(lse), to_f32(l_loc), rtol=0, atol=1e-6)


def test_lse_merge_in_place():
    # out may alias an input
    r = np.random.default_rng(3)
    n, H, d = 300, 4, 64
    a = bf16_tensor(synth.bf16_round(r.standard_normal((n, H * d)).astype(np.float32)))
    b = bf16_tensor(synth.bf16_round(r.standard_normal((n, H * d)).astype(np.float32)))
    la = torch.from_numpy(r.standard_normal((H, n)).astype(np.float32)).cuda()
    lb = torch.from_numpy(r.standard_normal((H, n)).astype(np.float32)).cuda()
    want, wl = at.lse_fuse(to_f32(a).reshape(n, H, d), to_f32(la), to_f32(b).reshape(n, H, d), to_f32(lb))
    abi.ispa_lse_merge(a, la, b, lb, n, H, d, a, None)
    torch.cuda.synchronize()
    assert np.abs(to_f32(a).reshape(n, H, d) - want).max() <= 2 ** -8 * np.abs(want).max() + 1e-6


def test_ring_compact_keeps_the_window_and_keeps_sliding():
    H, d, P = 2, 128, 40
    n_past, cap = 11, 12
    st = Step(33, P=P, H=H, d=d, n_past=n_past, n_chunk_frames=3, capacity=cap)
    win = Window(1, 3)
    small = Ring(H, d, P, 4, n_sink_frames=1)
    abi.ispa_ring_compact(st.ring.c, win, small.c)
    torch.cuda.synchronize()
    assert small.frames_written == n_past
    k_small = to_f32(small.k)
    for f in ks.local_past_frames(n_past, 1, 3):
        sl = ks.ring_slot(f, 4, 1)
        want = st.s.k_hist[f * P:(f + 1) * P].transpose(1, 0, 2)
        assert np.array_equal(k_small[:, sl * P:(sl + 1) * P], want), f
    # L-layer attention on the compacted ring equals the oracle's local attention
    out = torch.empty(st.n_q, H * d, dtype=torch.bfloat16, device="cuda")
    abi.ispa_attn_local(small.c, win, st.q, st.kc, st.vc, st.n_q, 0.0, out)
    torch.cuda.synchronize()
    ref, _ = at.attn_local(*st.oracle_args(), 1, 3)
    assert_close_attn(to_f32(out).reshape(ref.shape), ref, "local on compacted ring")
    # appending the chunk keeps the window sliding inside the small ring
    abi.ispa_kv_append(small.c, st.kc, st.vc, 3)
    torch.cuda.synchronize()
    k_small = to_f32(small.k)
    for i in range(3):
        sl = ks.ring_slot(n_past + i, 4, 1)
        want = st.s.k_cur[i * P:(i + 1) * P].transpose(1, 0, 2)
        assert np.array_equal(k_small[:, sl * P:(sl + 1) * P], want)
    assert np.array_equal(k_small[:, :P], st.s.k_hist[:P].transpose(1, 0, 2))   # the sink stays


def test_apply_absorption():
    r = np.random.default_rng(4)
    D, Do = 256, 192
    W = r.standard_normal((D, Do)).astype(np.float32)
    dW = (0.01 * r.standard_normal((D, Do))).astype(np.float32)
    Wt = torch.from_numpy(W).cuda()
    abi.ispa_apply_absorption(Wt, torch.from_numpy(dW).cuda(), D, Do)
    torch.cuda.synchronize()
    assert np.array_equal(Wt.cpu().numpy(), W + dW)
    Wb = synth.bf16_round(W)
    Wbt = bf16_tensor(Wb)
    abi.ispa_apply_absorption_bf16(Wbt, torch.from_numpy(dW).cuda(), D, Do)
    torch.cuda.synchronize()
    exact = Wb.astype(np.float64) + dW.astype(np.float64)
    assert np.all(np.abs(to_f32(Wbt) - exact) <= 2 ** -8 * np.abs(exact) + 1e-30)


@pytest.mark.parametrize("n,dim", [(1, 8), (37, 264), (4680, 1536), (1000, 5120)])
def test_discrepancy_of_stored_outputs(n, dim):
    # disc_t = ||a_t - b_t||_2 of two bf16 rows (differences of bf16 values are exact in fp32;
    # the fp32 sums of dim squares stay within 1e-5 relative of the fp64 norms), and the running
    # sum of disc^2 over two calls; ragged word counts (264 = 33 words) and the model widths
    a, b = synth.make_activations(400 + n, n, dim)
    disc = torch.empty(n, dtype=torch.float32, device="cuda")
    dsum = torch.zeros(1, dtype=torch.float32, device="cuda")
    ta, tb = bf16_tensor(a), bf16_tensor(b)
    abi.ispa_discrepancy(ta, tb, n, dim, disc, dsum)
    abi.ispa_discrepancy(ta, tb, n, dim, disc, dsum)
    torch.cuda.synchronize()
    want, want_sq = at.discrepancy(a, b)
    assert np.allclose(to_f32(disc), want, rtol=1e-5, atol=1e-6)
    assert abs(float(dsum.item()) - 2 * want_sq) <= 1e-5 * 2 * want_sq


def test_discrepancy_rejects_bad_arguments():
    x = torch.zeros(16, 64, dtype=torch.bfloat16, device="cuda")
    disc = torch.empty(16, dtype=torch.float32, device="cuda")
    dsum = torch.zeros(1, dtype=torch.float32, device="cuda")
    with pytest.raises(abi.IspaError) as e:
        abi.ispa_discrepancy(x, x, 16, 60, disc, dsum)
    assert e.value.status == abi.ISPA_ERR_UNSUPPORTED
    with pytest.raises(abi.IspaError) as e:
        abi.ispa_discrepancy(x, x, 0, 64, disc, dsum)
    assert e.value.status == abi.ISPA_ERR_INVALID_ARG
