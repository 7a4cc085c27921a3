"""Seeded fuzz of the two 8-bit paths through the C-ABI.

8-bit Q K^T attention: random frame lengths, heads, ring capacities with and without a pinned
sink, history lengths (wrapped rings included), windows and modes (full / local), each against
the oracle's attention of the dequantised q and k (max-abs 2e-2, mean-abs 2e-3, as for bf16).

8-bit Q K^T and P V attention: the same random steps (frame lengths a multiple of 4) through
full, local and dual, against the oracle's attention of the dequantised q, k and v within the
P-rounding bound of tests/test_gpu_kv8.py.

W8A8 projection: random token counts (ragged row tiles) and hidden sizes (multiples of 128,
both column-tile widths), codes bit for bit and the GEMM within the fp32-summation bound of
tests/test_gpu_w8a8.py.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from gpu_helpers import assert_close_attn  # noqa: E402
from oracle import attention as at  # noqa: E402
from oracle import keysets as ks  # noqa: E402
from oracle import quant as qt  # noqa: E402
from paper_2607_00712_gb300 import abi, synth  # noqa: E402
from test_gpu_kv8 import Kv8Step, assert_close_kv8, p_rounding_bound  # noqa: E402
from test_gpu_qk8 import Qk8Step  # noqa: E402
from test_gpu_w8a8 import _check_linear, _gpu_linear, _gpu_quant_rows, _gpu_quant_weight  # noqa: E402

pytestmark = pytest.mark.gpu
QK8_CASES, KV8_CASES, W8A8_CASES = 32, 16, 16


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2607_00712_gb300.build import build_library
    build_library()
    abi.lib()


@pytest.mark.parametrize("i", range(QK8_CASES))
def test_qk8_attention_fuzz(i):
    r = np.random.default_rng(55_000 + i)
    P = int(r.integers(1, 200))
    H = int(r.integers(1, 4))
    cap = int(r.integers(1, 9))
    sink = int(r.integers(0, min(2, cap - 1) + 1)) if cap > 1 else 0
    chunk = int(r.integers(1, 4))
    n_past = int(r.integers(0, 3 * cap + 1))
    st = Qk8Step(60_000 + i, P=P, H=H, n_past=n_past, n_chunk_frames=chunk, capacity=cap, n_sink_pinned=sink)
    if r.random() < 0.5:
        got, _ = st.full()
        ref, _ = at.attn_full(*st.args)
        assert_close_attn(got, ref, f"case {i} full")
    else:
        win = (int(r.integers(0, 3)), int(r.integers(0, cap + 1)))
        if not set(ks.local_past_frames(n_past, *win)) <= set(st.resident):
            with pytest.raises(abi.IspaError) as e:        # a window frame has been evicted
                st.local(win)
            assert e.value.status == abi.ISPA_ERR_CAPACITY
            return
        got, _ = st.local(win)
        ref, _ = at.attn_local(*st.args, *win)
        assert_close_attn(got, ref, f"case {i} local {win}")


@pytest.mark.parametrize("i", range(KV8_CASES))
def test_kv8_attention_fuzz(i):
    r = np.random.default_rng(57_000 + i)
    P = 4 * int(r.integers(1, 50))
    H = int(r.integers(1, 4))
    cap = int(r.integers(1, 9))
    sink = int(r.integers(0, min(2, cap - 1) + 1)) if cap > 1 else 0
    chunk = int(r.integers(1, 4))
    n_past = int(r.integers(0, 3 * cap + 1))
    st = Kv8Step(62_000 + i, P=P, H=H, n_past=n_past, n_chunk_frames=chunk, capacity=cap, n_sink_pinned=sink)
    q_hat = st.args[0]
    mode = ("full", "local", "dual")[int(r.integers(0, 3))]
    if mode == "full":
        got, _ = st.full()
        K, V = st.key_set()
        assert_close_kv8(got, at.attn_full(*st.args)[0], p_rounding_bound(q_hat, K, V), f"case {i} full")
        return
    win = (int(r.integers(0, 3)), int(r.integers(0, cap + 1)))
    if not set(ks.local_past_frames(n_past, *win)) <= set(st.resident):
        with pytest.raises(abi.IspaError) as e:        # a window frame has been evicted
            st.local(win) if mode == "local" else st.dual(win)
        assert e.value.status == abi.ISPA_ERR_CAPACITY
        return
    F = st.args[1].shape[0] // P
    Kl, Vl = st.key_set(ks.local_past_frames(F, *win))
    if mode == "local":
        got, _ = st.local(win)
        assert_close_kv8(got, at.attn_local(*st.args, *win)[0], p_rounding_bound(q_hat, Kl, Vl), f"case {i} local")
    else:
        af, al, _, _ = st.dual(win)
        ref = at.attn_dual(*st.args, *win)
        K, V = st.key_set()
        assert_close_kv8(af, ref["a_full"], p_rounding_bound(q_hat, K, V), f"case {i} dual full")
        assert_close_kv8(al, ref["a_loc"], p_rounding_bound(q_hat, Kl, Vl), f"case {i} dual loc")


@pytest.mark.parametrize("i", range(W8A8_CASES))
def test_w8a8_fuzz(i):
    r = np.random.default_rng(66_000 + i)
    T = int(r.integers(1, 700))
    D = 128 * int(r.integers(1, 9))
    Do = 128 * int(r.integers(1, 9))
    x, _ = synth.make_activations(67_000 + i, T, D)
    W = synth.make_weight(68_000 + i, D, Do)
    dW = (0.02 * synth.make_weight(69_000 + i, D, Do)).astype(np.float32) if r.random() < 0.5 else None
    aq, sa = _gpu_quant_rows(x)
    wq, sw = _gpu_quant_weight(W, dW)
    raq, rsa = qt.quantize_rows(x)
    rwq, rsw = qt.quantize_weight(W, dW)
    assert np.array_equal(aq.cpu().numpy(), raq) and np.array_equal(sa.cpu().numpy(), rsa)
    assert np.array_equal(wq.cpu().numpy(), rwq) and np.array_equal(sw.cpu().numpy(), rsw)
    y = _gpu_linear(aq, sa, wq, sw)
    _check_linear(y, raq, rsa, rwq, rsw)
