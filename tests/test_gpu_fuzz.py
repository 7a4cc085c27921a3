"""Seeded random chunk steps through every attention mode of the C-ABI, against the oracle.

Frame lengths, head counts, head dims, ring capacities (with and without a pinned sink),
windows, history lengths and the frame-causal option are drawn from a fixed seed; each case
runs F-layer, L-layer, dual and (with history) the two-call decomposition, with the bf16-path
tolerances.  Windows that need an evicted frame must be refused with ISPA_ERR_CAPACITY.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from gpu_helpers import Step, assert_close_attn, assert_disc_close  # noqa: E402
from oracle import attention as at  # noqa: E402
from oracle import keysets as ks  # noqa: E402
from paper_2607_00712_gb300 import abi  # noqa: E402
from paper_2607_00712_gb300.device import Window, to_f32  # noqa: E402

pytestmark = pytest.mark.gpu
CASES = 48


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2607_00712_gb300.build import build_library
    build_library()
    abi.lib()


def _case(i):
    r = np.random.default_rng(1000 + i)
    d = int(r.choice([64, 128]))
    P = int(r.choice([1, 7, 64, 100, 176, 190]))
    H = int(r.integers(1, 4))
    cap = int(r.integers(1, 9))
    pinned = int(r.integers(0, 2)) if cap > 1 else 0
    L = int(r.integers(1, 4))
    n_past = int(r.integers(0, 3 * cap + 2))
    win = (int(r.integers(0, 3)), int(r.integers(0, cap + 1)))
    causal = bool(r.integers(0, 2))
    return dict(d=d, P=P, H=H, cap=cap, pinned=pinned, L=L, n_past=n_past, win=win, causal=causal)


@pytest.mark.parametrize("i", range(CASES))
def test_random_step(i):
    c = _case(i)
    P, H, d = c["P"], c["H"], c["d"]
    st = Step(2000 + i, P=P, H=H, d=d, n_past=c["n_past"], n_chunk_frames=c["L"], capacity=c["cap"],
              n_sink_pinned=c["pinned"])
    flags = abi.ISPA_ATTN_FRAME_CAUSAL if c["causal"] else 0
    args = st.oracle_args()
    n_q, D = st.n_q, H * d
    out = torch.empty(n_q, D, dtype=torch.bfloat16, device="cuda")
    lse = torch.empty(H, n_q, dtype=torch.float32, device="cuda")
    abi.ispa_attn_full_ex(st.ring.c, st.q, st.kc, st.vc, n_q, 0.0, flags, out, lse)
    torch.cuda.synchronize()
    ro, rl = at.attn_full(*args, frame_causal=c["causal"])
    assert_close_attn(to_f32(out).reshape(ro.shape), ro, f"case {i} full {c}")
    assert np.abs(to_f32(lse) - rl).max() < 2e-3

    win = c["win"]
    loc_frames = ks.local_past_frames(c["n_past"], *win)
    if not set(loc_frames) <= set(st.resident):
        with pytest.raises(abi.IspaError) as e:
            abi.ispa_attn_local_ex(st.ring.c, Window(*win), st.q, st.kc, st.vc, n_q, 0.0, flags, out, lse)
        assert e.value.status == abi.ISPA_ERR_CAPACITY
        return
    abi.ispa_attn_local_ex(st.ring.c, Window(*win), st.q, st.kc, st.vc, n_q, 0.0, flags, out, lse)
    torch.cuda.synchronize()
    ro, rl = at.attn_local(*args, *win, frame_causal=c["causal"])
    assert_close_attn(to_f32(out).reshape(ro.shape), ro, f"case {i} local {c}")
    assert np.abs(to_f32(lse) - rl).max() < 2e-3

    a_full = torch.empty(n_q, D, dtype=torch.bfloat16, device="cuda")
    a_loc = torch.empty_like(a_full)
    disc = torch.empty(n_q, dtype=torch.float32, device="cuda")
    dsum = torch.zeros(1, dtype=torch.float32, device="cuda")
    wsb = abi.ispa_attn_dual_workspace_size(H, n_q)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    abi.ispa_attn_dual_ex(st.ring.c, Window(*win), st.q, st.kc, st.vc, n_q, 0.0, flags, a_full, a_loc, disc, dsum,
                          None, None, ws, wsb)
    torch.cuda.synchronize()
    r = at.attn_dual(*args, *win, frame_causal=c["causal"])
    assert_close_attn(to_f32(a_full).reshape(ro.shape), r["a_full"], f"case {i} dual full {c}")
    assert_close_attn(to_f32(a_loc).reshape(ro.shape), r["a_loc"], f"case {i} dual loc {c}")
    assert_disc_close(to_f32(a_full).reshape(ro.shape), to_f32(a_loc).reshape(ro.shape), to_f32(disc), r,
                      f"case {i} disc {c}", float(dsum.item()))

    # the paper's two-call decomposition (Eq. 9-12) on the dense chunk
    if not c["causal"]:
        o_loc = torch.empty(n_q, D, dtype=torch.bfloat16, device="cuda")
        l_loc = torch.empty(H, n_q, dtype=torch.float32, device="cuda")
        o_hist = torch.empty_like(o_loc)
        l_hist = torch.empty_like(l_loc)
        fused = torch.empty_like(o_loc)
        abi.ispa_attn_local(st.ring.c, Window(*win), st.q, st.kc, st.vc, n_q, 0.0, o_loc, l_loc)
        abi.ispa_attn_hist(st.ring.c, Window(*win), st.q, n_q, 0.0, o_hist, l_hist)
        abi.ispa_lse_merge(o_loc, l_loc, o_hist, l_hist, n_q, H, d, fused, None)
        torch.cuda.synchronize()
        rf, _ = at.attn_full(*args)
        assert_close_attn(to_f32(fused).reshape(rf.shape), rf, f"case {i} two-call {c}")
