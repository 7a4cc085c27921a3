"""GPU parity of the frame-causal chunk option (ISPA_ATTN_FRAME_CAUSAL) through the C-ABI.

Eq. 3 keeps the chunk dense; the option makes a query of chunk frame a see the chunk's
frames 0..a only.  The oracle (oracle.attention, frame_causal=True) is pinned by a
brute force and special cases in test_oracle_attention.py.
"""
import math

import numpy as np
import pytest

torch = pytest.importorskip("torch")

from gpu_helpers import Step, assert_close_attn, assert_disc_close  # noqa: E402
from oracle import attention as at  # noqa: E402
from paper_2607_00712_gb300 import abi  # noqa: E402
from paper_2607_00712_gb300.device import Window, to_f32  # noqa: E402

pytestmark = pytest.mark.gpu
CAUSAL = abi.ISPA_ATTN_FRAME_CAUSAL


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2607_00712_gb300.build import build_library
    build_library()
    abi.lib()


def _full(st, flags):
    out = torch.empty(st.n_q, st.H * st.d, dtype=torch.bfloat16, device="cuda")
    lse = torch.empty(st.H, st.n_q, dtype=torch.float32, device="cuda")
    abi.ispa_attn_full_ex(st.ring.c, st.q, st.kc, st.vc, st.n_q, 0.0, flags, out, lse)
    torch.cuda.synchronize()
    return to_f32(out).reshape(st.n_q, st.H, st.d), to_f32(lse)


def _local(st, win, flags):
    out = torch.empty(st.n_q, st.H * st.d, dtype=torch.bfloat16, device="cuda")
    lse = torch.empty(st.H, st.n_q, dtype=torch.float32, device="cuda")
    abi.ispa_attn_local_ex(st.ring.c, Window(*win), st.q, st.kc, st.vc, st.n_q, 0.0, flags, out, lse)
    torch.cuda.synchronize()
    return to_f32(out).reshape(st.n_q, st.H, st.d), to_f32(lse)


def _dual(st, win, flags):
    D = st.H * st.d
    a_full = torch.empty(st.n_q, D, dtype=torch.bfloat16, device="cuda")
    a_loc = torch.empty(st.n_q, D, dtype=torch.bfloat16, device="cuda")
    disc = torch.empty(st.n_q, dtype=torch.float32, device="cuda")
    dsum = torch.zeros(1, dtype=torch.float32, device="cuda")
    wsb = abi.ispa_attn_dual_workspace_size(st.H, st.n_q)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    abi.ispa_attn_dual_ex(st.ring.c, Window(*win), st.q, st.kc, st.vc, st.n_q, 0.0, flags, a_full, a_loc, disc,
                          dsum, None, None, ws, wsb)
    torch.cuda.synchronize()
    return (to_f32(a_full).reshape(st.n_q, st.H, st.d), to_f32(a_loc).reshape(st.n_q, st.H, st.d),
            to_f32(disc))


@pytest.mark.parametrize("d", [64, 128])
def test_causal_ragged_tiles_and_ring_wrap(d):
    # 100 tokens per frame: key tiles straddle frame boundaries, so the causal limit falls
    # inside tiles; 300 queries (three chunk frames), a wrapped ring with a pinned sink.
    st = Step(41, P=100, H=3, d=d, n_past=12, n_chunk_frames=3, capacity=7, n_sink_pinned=1)
    args = st.oracle_args()
    o, l = _full(st, CAUSAL)
    ro, rl = at.attn_full(*args, frame_causal=True)
    assert_close_attn(o, ro, "causal full")
    assert np.abs(l - rl).max() < 2e-3
    for win in [(1, 2), (0, 3), (1, 0)]:
        o, l = _local(st, win, CAUSAL)
        ro, rl = at.attn_local(*args, *win, frame_causal=True)
        assert_close_attn(o, ro, f"causal local {win}")
        assert np.abs(l - rl).max() < 2e-3
        af, al, disc = _dual(st, win, CAUSAL)
        r = at.attn_dual(*args, *win, frame_causal=True)
        assert_close_attn(af, r["a_full"], f"causal dual full {win}")
        assert_close_attn(al, r["a_loc"], f"causal dual loc {win}")
        assert_disc_close(af, al, disc, r, f"causal disc {win}")


def test_causal_flag_zero_is_the_plain_call():
    st = Step(42, P=64, H=2, d=128, n_past=5, n_chunk_frames=2, capacity=6)
    o_ex, l_ex = _full(st, 0)
    out = torch.empty(st.n_q, st.H * st.d, dtype=torch.bfloat16, device="cuda")
    lse = torch.empty(st.H, st.n_q, dtype=torch.float32, device="cuda")
    abi.ispa_attn_full(st.ring.c, st.q, st.kc, st.vc, st.n_q, 0.0, out, lse)
    torch.cuda.synchronize()
    assert np.array_equal(o_ex, to_f32(out).reshape(o_ex.shape)) and np.array_equal(l_ex, to_f32(lse))
    # the chunk's last frame sees the whole chunk either way
    o_c, _ = _full(st, CAUSAL)
    assert_close_attn(o_c[64:], o_ex[64:], "last chunk frame")


def test_causal_no_history_first_frame():
    # no past frames: chunk frame 0 attends to itself only
    st = Step(43, P=96, H=2, d=64, n_past=0, n_chunk_frames=3, capacity=4)
    o, _ = _full(st, CAUSAL)
    want, _ = at.attend_heads(st.s.q[:96], st.s.k_cur[:96], st.s.v_cur[:96], 1.0 / math.sqrt(64))
    assert_close_attn(o[:96], want, "frame 0")
    ro, _ = at.attn_full(*st.oracle_args(), frame_causal=True)
    assert_close_attn(o, ro, "no history")


def test_causal_config1_sampled_rows():
    # 1.3B shapes (12 heads x 128, 1560 tokens/frame, 4680 queries, 18 cached frames), rows
    # on both sides of each chunk-frame boundary
    st = Step(44, P=1560, H=12, d=128, n_past=18, n_chunk_frames=3, capacity=18)
    rng = np.random.default_rng(1)
    rows = np.unique(np.concatenate([[0, 1559, 1560, 3119, 3120, 4679], rng.choice(4680, 42, replace=False)]))
    args = st.oracle_args()
    o, _ = _full(st, CAUSAL)
    ro, _ = at.attn_full(*args, rows=rows, frame_causal=True)
    assert_close_attn(o[rows], ro, "config1 causal full")
    af, al, disc = _dual(st, (0, 6), CAUSAL)
    r = at.attn_dual(*args, 0, 6, rows=rows, frame_causal=True)
    assert_close_attn(af[rows], r["a_full"], "config1 causal dual full")
    assert_close_attn(al[rows], r["a_loc"], "config1 causal dual loc")
    assert_disc_close(af[rows], al[rows], disc[rows], r, "config1 causal disc")
