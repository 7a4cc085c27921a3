"""The traced attention instance (ispa_debug_set_trace) computes what the production instance
computes, bit for bit, and records every tile's events in causal order."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from gpu_helpers import Step  # noqa: E402
from paper_2607_00712_gb300 import abi  # noqa: E402
from paper_2607_00712_gb300.device import Window  # noqa: E402

pytestmark = pytest.mark.gpu
SLOTS = 32


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2607_00712_gb300.build import build_library
    build_library()
    abi.lib()


def _run(st, mode, trace_tiles=0):
    n, D = st.n_q, st.H * st.d
    out = torch.empty(n, D, dtype=torch.bfloat16, device="cuda")
    buf = torch.zeros(max(trace_tiles, 1) * SLOTS, dtype=torch.int64, device="cuda")
    if trace_tiles:
        abi.ispa_debug_set_trace(buf, trace_tiles)
    try:
        if mode == "full":
            abi.ispa_attn_full(st.ring.c, st.q, st.kc, st.vc, n, 0.0, out)
        else:
            abi.ispa_attn_local(st.ring.c, Window(0, 2), st.q, st.kc, st.vc, n, 0.0, out)
        torch.cuda.synchronize()
    finally:
        abi.ispa_debug_set_trace(None, 0)
    return out.view(torch.int16).cpu().numpy(), buf.view(-1, SLOTS).cpu().numpy()


@pytest.mark.parametrize("mode", ["full", "local"])
def test_trace_instance_matches_production_and_orders_events(mode):
    st = Step(4242, P=200, H=3, d=128, n_past=7, n_chunk_frames=2, capacity=8)
    plain, _ = _run(st, mode)
    traced, t = _run(st, mode, trace_tiles=64)
    assert np.array_equal(plain, traced)
    n = int((t[:, 3] != 0).sum())
    assert n >= 2 and np.all(t[:n, 3] != 0) and np.all(t[n:, :] == 0)
    for j in range(n):
        e = t[j]
        # softmax warp 0: S seen <= loaded <= P computed <= rescale decided <= P stored <= arrived
        assert e[0] <= e[8] <= e[9] <= e[1] <= e[10] <= e[2], (j, e[:12])
        # UMMA thread: P seen <= V seen <= PV issued <= the next S issued
        assert e[3] <= e[11] <= e[4] <= e[5], (j, e[:12])
        # TMA thread issued K_j before the UMMA thread saw P_j, V_j before PV_j was issued
        assert e[6] <= e[3] and e[7] <= e[4], (j, e[:12])
        # every softmax warp saw S_j and published P_j (each stamp follows its own arrive, so it
        # is not ordered against the UMMA thread's view of the barrier)
        assert np.all(e[24:32] != 0) and np.all(e[16:24] != 0)
        assert np.all(e[16:24] >= e[24:32])
        if j >= 1:
            # slot 15 (tiles >= 1): the UMMA thread saw K_j land after the TMA thread issued it;
            # S_1 goes out before the first PV, S_j (j >= 2) right after PV_j-2
            assert e[6] <= e[15], (j, e[15])
            if j >= 2:
                assert t[j - 2, 4] <= e[15] <= t[j - 2, 5], (j, e[15])
            else:
                assert e[15] <= t[0, 3], (j, e[15])
