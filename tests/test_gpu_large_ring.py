"""A ring larger than 2^31 bytes per buffer (maximum-size edge case): the window frames and the
appended frames sit at byte offsets beyond 2^31 inside the second head's slab, so every offset
on the path (append, the attention's TMA maps, the key-tile rows) must be 64-bit.

The ring struct is plain data, so the test sets frames_written directly instead of appending
thousands of frames, then appends two frames (checked bit for bit at their slots) and runs the
L-layer attention over a window of those two frames plus the chunk against the oracle."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from gpu_helpers import assert_close_attn  # noqa: E402
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


def test_window_beyond_2gib_offsets():
    P, H, d, cap, chunk = 1560, 2, 128, 5400, 3        # 8.42M slots: 2.16 GB per head and buffer
    slab = cap * P * d * 2
    assert slab > 2 ** 31
    ring = Ring(H, d, P, cap, 0)
    written = cap * 3 - 5                                # the ring has wrapped twice
    ring.c.frames_written = written
    s = synth.make_step(77, 2, P, H, d, n_chunk_frames=chunk)
    k_new, v_new = bf16_tensor(s.k_hist), bf16_tensor(s.v_hist)
    abi.ispa_kv_append(ring.c, k_new, v_new, 2)
    torch.cuda.synchronize()
    assert ring.frames_written == written + 2
    slots = [ks.ring_slot(written + i, cap, 0) for i in range(2)]
    assert min(slots) * P * d * 2 + slab > 2 ** 31     # head 1's copy of them lies past 2 GiB
    for i, sl in enumerate(slots):
        for h in range(H):
            got_k = to_f32(ring.k[h, sl * P:(sl + 1) * P])
            got_v = to_f32(ring.v[h, sl * P:(sl + 1) * P])
            assert np.array_equal(got_k, s.k_hist[i * P:(i + 1) * P, h])
            assert np.array_equal(got_v, s.v_hist[i * P:(i + 1) * P, h])
    n = s.q.shape[0]
    out = torch.empty(n, H * d, dtype=torch.bfloat16, device="cuda")
    abi.ispa_attn_local(ring.c, Window(0, 2), bf16_tensor(s.q), bf16_tensor(s.k_cur), bf16_tensor(s.v_cur), n,
                        0.0, out)
    torch.cuda.synchronize()
    st, code = abi.ispa_last_device_error()
    assert st == abi.ISPA_OK, code
    rows = np.unique(np.concatenate([[0, 127, 128, n - 1], np.random.default_rng(3).choice(n, 40, False)]))
    ref, _ = at.attn_full(s.q, s.k_hist, s.v_hist, s.k_cur, s.v_cur, P, rows=rows)
    assert_close_attn(to_f32(out).reshape(n, H, d)[rows], ref, "window past 2 GiB")
