"""GPU parity: chunk-step attention (full / local / dual) through the C-ABI vs the fp64 oracle.

Tolerance (bf16 outputs, fp32 accumulation): max-abs <= 2e-2, mean-abs <= 2e-3.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from gpu_helpers import Step, assert_close_attn, assert_disc_close  # noqa: E402
from oracle import attention as at  # noqa: E402
from paper_2607_00712_gb300 import abi  # noqa: E402
from paper_2607_00712_gb300.device import Window, bf16_tensor, to_f32  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2607_00712_gb300.build import build_library
    build_library()
    abi.lib()


def _run_full(st: Step, scale=0.0):
    out = torch.empty(st.n_q, st.H * st.d, dtype=torch.bfloat16, device="cuda")
    lse = torch.empty(st.H, st.n_q, dtype=torch.float32, device="cuda")
    abi.ispa_attn_full(st.ring.c, st.q, st.kc, st.vc, st.n_q, scale, out, lse)
    torch.cuda.synchronize()
    return to_f32(out).reshape(st.n_q, st.H, st.d), to_f32(lse)


def _run_local(st: Step, win, scale=0.0):
    out = torch.empty(st.n_q, st.H * st.d, dtype=torch.bfloat16, device="cuda")
    lse = torch.empty(st.H, st.n_q, dtype=torch.float32, device="cuda")
    abi.ispa_attn_local(st.ring.c, Window(*win), st.q, st.kc, st.vc, st.n_q, scale, out, lse)
    torch.cuda.synchronize()
    return to_f32(out).reshape(st.n_q, st.H, st.d), to_f32(lse)


def _run_dual(st: Step, win, scale=0.0, disc_sum=None):
    D = st.H * st.d
    a_full = torch.empty(st.n_q, D, dtype=torch.bfloat16, device="cuda")
    a_loc = torch.empty(st.n_q, D, dtype=torch.bfloat16, device="cuda")
    disc = torch.empty(st.n_q, dtype=torch.float32, device="cuda")
    if disc_sum is None:
        disc_sum = torch.zeros(1, dtype=torch.float32, device="cuda")
    lf = torch.empty(st.H, st.n_q, dtype=torch.float32, device="cuda")
    ll = torch.empty(st.H, st.n_q, dtype=torch.float32, device="cuda")
    wsb = abi.ispa_attn_dual_workspace_size(st.H, st.n_q)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    abi.ispa_attn_dual(st.ring.c, Window(*win), st.q, st.kc, st.vc, st.n_q, scale, a_full, a_loc, disc,
                       disc_sum, lf, ll, ws, wsb)
    torch.cuda.synchronize()
    return dict(a_full=to_f32(a_full).reshape(st.n_q, st.H, st.d), a_loc=to_f32(a_loc).reshape(st.n_q, st.H, st.d),
                disc=to_f32(disc), disc_sum=float(disc_sum.item()), lse_full=to_f32(lf), lse_loc=to_f32(ll))


def _check_all_modes(st: Step, win, scale=0.0):
    args = st.oracle_args()
    o, l = _run_full(st, scale)
    ro, rl = at.attn_full(*args, scale=scale)
    assert_close_attn(o, ro, "full")
    assert np.abs(l - rl).max() < 2e-3
    o, l = _run_local(st, win, scale)
    ro, rl = at.attn_local(*args, *win, scale=scale)
    assert_close_attn(o, ro, "local")
    assert np.abs(l - rl).max() < 2e-3
    g = _run_dual(st, win, scale)
    r = at.attn_dual(*args, *win, scale=scale)
    assert_close_attn(g["a_full"], r["a_full"], "dual a_full")
    assert_close_attn(g["a_loc"], r["a_loc"], "dual a_loc")
    assert np.abs(g["lse_full"] - r["lse_full"]).max() < 2e-3
    assert np.abs(g["lse_loc"] - r["lse_loc"]).max() < 2e-3
    # disc and the one-call sum of disc^2 against the oracle's, within the bound the outputs'
    # own errors give (triangle inequality, per token)
    assert_disc_close(g["a_full"], g["a_loc"], g["disc"], r, "dual disc", g["disc_sum"])
    # extra: disc is the norm of the difference of the two stored bf16 outputs
    d_own = np.sqrt(((g["a_full"].astype(np.float64) - g["a_loc"]) ** 2).reshape(st.n_q, -1).sum(1))
    assert np.allclose(g["disc"], d_own, rtol=1e-5, atol=1e-6)


def test_config0_tiny():
    # 2 heads, d = 64, 64 tokens/frame, chunk of 2 frames (128 queries), 4 cached frames
    # (384 keys in the full set), window = chunk + 2 most recent frames.
    st = Step(0, P=64, H=2, d=64, n_past=4, n_chunk_frames=2, capacity=4)
    _check_all_modes(st, (0, 2))


@pytest.mark.parametrize("d", [64, 128])
def test_ragged_tiles_and_ring_wrap(d):
    # 100 tokens per frame (tiles straddle frames), 300 queries (ragged tail), a ring of 7
    # frames with one pinned sink that has wrapped (12 frames written).
    st = Step(1, P=100, H=3, d=d, n_past=12, n_chunk_frames=3, capacity=7, n_sink_pinned=1)
    for win in [(1, 2), (0, 3), (1, 0), (1, 6)]:
        _check_all_modes(st, win)


def test_explicit_scale_and_single_frame_chunk():
    st = Step(2, P=72, H=2, d=64, n_past=5, n_chunk_frames=1, capacity=8)
    _check_all_modes(st, (0, 2), scale=0.21)


def test_no_history():
    # F = 0: every mode sees only the chunk.
    st = Step(3, P=64, H=2, d=128, n_past=0, n_chunk_frames=2, capacity=4)
    o_full, _ = _run_full(st)
    o_loc, _ = _run_local(st, (0, 2))
    assert np.array_equal(o_full, o_loc)
    g = _run_dual(st, (0, 2))
    assert np.array_equal(g["a_full"], g["a_loc"]) and np.all(g["disc"] == 0)


def test_values_all_one():
    st = Step(4, P=64, H=2, d=128, n_past=3, n_chunk_frames=2, capacity=4)
    st.ring.v.fill_(1.0)
    st.vc.fill_(1.0)
    o, _ = _run_full(st)
    assert np.all(o == 1.0)
    o, _ = _run_local(st, (0, 1))
    assert np.all(o == 1.0)


def test_empty_history_dual_is_exact():
    # window covers the whole cache: hist is empty, A_full == A_loc bit for bit, disc == 0
    st = Step(5, P=96, H=2, d=128, n_past=4, n_chunk_frames=2, capacity=6)
    g = _run_dual(st, (0, 4))
    assert np.array_equal(g["a_full"], g["a_loc"])
    assert np.all(g["disc"] == 0) and g["disc_sum"] == 0.0
    # and local over that window matches full within tolerance
    o_full, _ = _run_full(st)
    o_loc, _ = _run_local(st, (0, 4))
    assert_close_attn(o_loc, o_full, "window covering cache")


def test_disc_sum_accumulates():
    st = Step(6, P=64, H=2, d=64, n_past=4, n_chunk_frames=2, capacity=4)
    acc = torch.zeros(1, dtype=torch.float32, device="cuda")
    g1 = _run_dual(st, (0, 1), disc_sum=acc)
    g2 = _run_dual(st, (0, 1), disc_sum=acc)
    one = float((g1["disc"].astype(np.float64) ** 2).sum())
    assert abs(g2["disc_sum"] - 2 * one) <= 1e-4 * 2 * one


def test_config1_sampled_rows():
    # The 1.3B-shaped chunk step the bench times: 12 heads x 128, 1560 tokens/frame, 4680 queries,
    # 18 cached frames (28080 keys + 4680 chunk keys), window = chunk + 6 frames.  Rows are
    # independent, so the oracle on sampled rows is exact for those rows.
    st = Step(7, P=1560, H=12, d=128, n_past=18, n_chunk_frames=3, capacity=18)
    rng = np.random.default_rng(0)
    rows = np.unique(np.concatenate([[0, 127, 128, 4607, 4608, 4679], rng.choice(4680, 58, replace=False)]))
    args = st.oracle_args()
    o, l = _run_full(st)
    ro, rl = at.attn_full(*args, rows=rows)
    assert_close_attn(o[rows], ro, "config1 full")
    assert np.abs(l[:, rows] - rl).max() < 2e-3
    o, _ = _run_local(st, (0, 6))
    ro, _ = at.attn_local(*args, 0, 6, rows=rows)
    assert_close_attn(o[rows], ro, "config1 local")
    g = _run_dual(st, (0, 6))
    r = at.attn_dual(*args, 0, 6, rows=rows)
    assert_close_attn(g["a_full"][rows], r["a_full"], "config1 dual full")
    assert_close_attn(g["a_loc"][rows], r["a_loc"], "config1 dual loc")
    assert_disc_close(g["a_full"][rows], g["a_loc"][rows], g["disc"][rows], r, "config1 disc")
    assert np.isfinite(g["disc"]).all()


@pytest.mark.parametrize("d", [64, 128])
@pytest.mark.parametrize("boost,frames", [(3.0, (4, 5)), (6.0, (4, 5)), (6.0, (5,))])
def test_running_max_rescale_path(boost, frames, d):
    # Late frames whose keys are scaled up make the running row max jump by more than 2^8 for
    # some rows (boost 3: some lanes of a warp, boost 6: nearly all), exercising the lazy O
    # rescale in TMEM, including warps where only part of the lanes need it.  The 6 past frames
    # of 64 keys fill key tiles 0 (keys 0-191) and 1 (192-383); frame 5 (keys 320-383) lies in
    # the second half-row of tile 1 only, so with frames = (5,) one warp of each pair alone sees
    # the jump and the pair's reducing barrier must carry the decision to its partner.
    from paper_2607_00712_gb300 import synth
    st = Step(8, P=64, H=2, d=d, n_past=6, n_chunk_frames=2, capacity=6)
    P = st.P
    for f in frames:
        blk = synth.bf16_round(st.s.k_hist[f * P:(f + 1) * P] * np.float32(boost))
        st.s.k_hist[f * P:(f + 1) * P] = blk
        st.k_hist_res[f * P:(f + 1) * P] = blk
        st.ring.k[:, f * P:(f + 1) * P] = bf16_tensor(blk.transpose(1, 0, 2).copy())
    torch.cuda.synchronize()
    _check_all_modes(st, (0, 2))
    _check_all_modes(st, (0, 1))


def test_back_to_back_calls_without_host_sync():
    # Many launches queued on one stream with no host synchronisation in between (the
    # pattern of a layer loop); results equal the single-call results bit for bit.
    st = Step(9, P=100, H=3, d=128, n_past=9, n_chunk_frames=3, capacity=7)
    o_ref, _ = _run_full(st)
    l_ref, _ = _run_local(st, (0, 3))
    g_ref = _run_dual(st, (0, 2))
    D = st.H * st.d
    outs = [torch.empty(st.n_q, D, dtype=torch.bfloat16, device="cuda") for _ in range(4)]
    disc = torch.empty(st.n_q, dtype=torch.float32, device="cuda")
    dsum = torch.zeros(1, dtype=torch.float32, device="cuda")
    wsb = abi.ispa_attn_dual_workspace_size(st.H, st.n_q)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    for _ in range(6):
        abi.ispa_attn_full(st.ring.c, st.q, st.kc, st.vc, st.n_q, 0.0, outs[0])
        abi.ispa_attn_local(st.ring.c, Window(0, 3), st.q, st.kc, st.vc, st.n_q, 0.0, outs[1])
        abi.ispa_attn_dual(st.ring.c, Window(0, 2), st.q, st.kc, st.vc, st.n_q, 0.0, outs[2], outs[3], disc, dsum,
                           None, None, ws, wsb)
    torch.cuda.synchronize()
    assert abi.ispa_last_device_error()[0] == abi.ISPA_OK
    assert np.array_equal(to_f32(outs[0]).reshape(o_ref.shape), o_ref)
    assert np.array_equal(to_f32(outs[1]).reshape(l_ref.shape), l_ref)
    assert np.array_equal(to_f32(outs[2]).reshape(o_ref.shape), g_ref["a_full"])
    assert np.array_equal(to_f32(outs[3]).reshape(o_ref.shape), g_ref["a_loc"])


@pytest.mark.parametrize("d", [64, 128])
def test_minimum_sizes_one_query_one_head(d):
    # n_q = 1 (one query of a one-token chunk frame), one head, one-token frames: the
    # smallest step the boundary accepts
    st = Step(51, P=1, H=1, d=d, n_past=5, n_chunk_frames=1, capacity=3, n_sink_pinned=1)
    assert st.n_q == 1
    _check_all_modes(st, (1, 1))


def test_work_stealing_covers_every_item():
    # 64 heads x 5 query tiles = 320 (query tile, head) items, about twice the SM count: the
    # CTAs that start first take the items of CTAs that have not started (cluster launch
    # control).  Every row of every item is checked against the oracle, and repeated calls
    # must agree bit for bit whichever CTA ran an item.
    n_sm = torch.cuda.get_device_properties(0).multi_processor_count
    st = Step(61, P=128, H=64, d=128, n_past=3, n_chunk_frames=5, capacity=4)
    assert st.n_q == 640 and 5 * st.H > n_sm
    o, l = _run_full(st)
    ro, rl = at.attn_full(*st.oracle_args())
    assert_close_attn(o, ro, "stolen items full")
    assert np.abs(l - rl).max() < 2e-3
    for _ in range(3):
        o2, l2 = _run_full(st)
        assert np.array_equal(o2, o) and np.array_equal(l2, l)
    g = _run_dual(st, (0, 1))
    r = at.attn_dual(*st.oracle_args(), 0, 1)
    assert_close_attn(g["a_full"], r["a_full"], "stolen items dual full")
    assert_close_attn(g["a_loc"], r["a_loc"], "stolen items dual loc")
    assert_disc_close(g["a_full"], g["a_loc"], g["disc"], r, "stolen items disc", g["disc_sum"])


def test_repeated_launches_at_the_step_shape_are_bit_identical():
    # 444 items at the 1.3B step shape, each launch redistributing them over the SMs by work
    # stealing: 12 rounds of the three modes launched back to back on one stream, with no host
    # synchronisation between them, must reproduce the first launches' outputs bit for bit (the
    # arithmetic of an item does not depend on which CTA runs it, and no item may be skipped or
    # run twice)
    st = Step(62, P=1560, H=12, d=128, n_past=18, n_chunk_frames=3, capacity=18)
    D = st.H * st.d
    ref_f, _ = _run_full(st)
    ref_l, _ = _run_local(st, (0, 6))
    g = _run_dual(st, (0, 6))
    wsb = abi.ispa_attn_dual_workspace_size(st.H, st.n_q)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    dsum = torch.zeros(1, dtype=torch.float32, device="cuda")
    rounds = []
    for _ in range(12):
        outs = [torch.empty(st.n_q, D, dtype=torch.bfloat16, device="cuda") for _ in range(4)]
        disc = torch.empty(st.n_q, dtype=torch.float32, device="cuda")
        abi.ispa_attn_full(st.ring.c, st.q, st.kc, st.vc, st.n_q, 0.0, outs[0])
        abi.ispa_attn_local(st.ring.c, Window(0, 6), st.q, st.kc, st.vc, st.n_q, 0.0, outs[1])
        abi.ispa_attn_dual(st.ring.c, Window(0, 6), st.q, st.kc, st.vc, st.n_q, 0.0, outs[2], outs[3], disc, dsum,
                           None, None, ws, wsb)
        rounds.append((outs, disc))
    torch.cuda.synchronize()
    assert abi.ispa_last_device_error()[0] == abi.ISPA_OK
    bad = []
    for i, (outs, disc) in enumerate(rounds):
        for name, t, ref in [("full", outs[0], ref_f), ("local", outs[1], ref_l), ("dual full", outs[2], g["a_full"]),
                             ("dual loc", outs[3], g["a_loc"])]:
            if not np.array_equal(to_f32(t).reshape(ref.shape), ref):
                bad.append((i, name))
        if not np.array_equal(to_f32(disc), g["disc"]):
            bad.append((i, "disc"))
    assert not bad, bad
