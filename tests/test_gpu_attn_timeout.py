"""The attention kernel's timeout path: with ispa_debug_drop_k_tile the TMA thread of every CTA
stops before loading one key tile (and the V tile it would issue with it), so a wait of the UMMA
thread never completes; after the wait limit (2 ms here) the CTA raises its abort flag and every
role leaves through its abort path: the softmax warps keep walking every tile through the same
warp-pair barriers, the A_loc snapshot and the epilogue.  The call must return, report
ISPA_ERR_TIMEOUT, and leave the context usable: the same call without the drop then matches a
plain run bit for bit.  The dual pass is run with the drop before and after its A_loc snapshot;
its aborted rows report a NaN discrepancy, so the running sum of disc^2 turns NaN rather than
taking a partial or stale value."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from gpu_helpers import Step  # noqa: E402
from paper_2607_00712_gb300 import abi  # noqa: E402
from paper_2607_00712_gb300.device import Window  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2607_00712_gb300.build import build_library
    build_library()
    abi.lib()


def _host(ts):
    return [t.view(torch.int16).cpu().numpy() if t.dtype == torch.bfloat16 else t.cpu().numpy() for t in ts]


def _run(st, mode):
    n, D = st.n_q, st.H * st.d
    out = torch.zeros(n, D, dtype=torch.bfloat16, device="cuda")
    if mode == "full":
        abi.ispa_attn_full(st.ring.c, st.q, st.kc, st.vc, n, 0.0, out)
        return [out]
    out_loc = torch.zeros_like(out)
    disc = torch.zeros(n, dtype=torch.float32, device="cuda")
    dsum = torch.zeros(1, dtype=torch.float32, device="cuda")
    wsb = abi.ispa_attn_dual_workspace_size(st.H, n)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    abi.ispa_attn_dual(st.ring.c, Window(0, 2), st.q, st.kc, st.vc, n, 0.0, out, out_loc, disc, dsum, None, None,
                       ws, wsb)
    return [out, out_loc, disc, dsum]


@pytest.mark.parametrize("mode,drop", [("full", 3), ("dual", 3), ("dual", 7)])
def test_attention_timeout_is_reported_and_recoverable(mode, drop):
    # 7 past frames of 200 tokens + a 2-frame chunk: 1800 keys in 11 key tiles of 192; the dual
    # pass's local set (2 frames + the chunk: 3 + 3 tiles) comes first, so a drop at tile 3
    # falls before its A_loc snapshot and one at tile 7 after it
    st = Step(8080, P=200, H=3, d=128, n_past=7, n_chunk_frames=2, capacity=8)
    abi.ispa_last_device_error()                 # clear
    plain = _host(_run(st, mode))
    assert abi.ispa_last_device_error()[0] == abi.ISPA_OK
    old = abi.ispa_set_wait_limit_ns(2_000_000)
    abi.ispa_debug_drop_k_tile(drop)
    try:
        aborted = _run(st, mode)
        torch.cuda.synchronize()
    finally:
        abi.ispa_debug_drop_k_tile(-1)
        abi.ispa_set_wait_limit_ns(old)
    st_code, raw = abi.ispa_last_device_error()
    assert st_code == abi.ISPA_ERR_TIMEOUT and raw == 1, (st_code, raw)
    assert abi.ispa_last_device_error()[0] == abi.ISPA_OK   # reading clears it
    if mode == "dual":
        # an aborted row's discrepancy partial is NaN, so the running sum of disc^2 turns NaN
        # rather than silently taking a partial or stale value (the other outputs of a timed-out
        # call are undefined)
        assert np.isnan(aborted[2].cpu().numpy()).any() and np.isnan(float(aborted[3].item()))
    again = _host(_run(st, mode))
    assert abi.ispa_last_device_error()[0] == abi.ISPA_OK
    for a, b in zip(plain, again):
        assert np.array_equal(a, b)
