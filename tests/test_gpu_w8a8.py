"""GPU parity of the W8A8 output projection on W + dW (Sec. 4) through the C-ABI.

Quantised codes and scales are integer / exactly-specified fp32 results: they must equal
the oracle's (oracle.quant, pinned in test_oracle_quant.py) bit for bit.  The GEMM output
is compared with the oracle's float64 product of the same codes within a bound derived from
the arithmetic: fp32 accumulation of exact e4m3 products (two chains of D/2 terms, then
their sum), two fp32 scale multiplies, and the final bf16 rounding:
  |y - y_ref| <= 2^-8 |y_ref| + 2 (D/2 + 3) 2^-24 a_scale w_scale sum_k |a_k w_k|.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import quant as qt  # noqa: E402
from paper_2607_00712_gb300 import abi, synth  # noqa: E402
from paper_2607_00712_gb300.device import bf16_tensor, to_f32  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2607_00712_gb300.build import build_library
    build_library()
    abi.lib()


def _activations(seed, T, D):
    a, _ = synth.make_activations(seed, T, D)
    return a


def _gpu_quant_rows(x):
    T, D = x.shape
    xt = bf16_tensor(x)
    q = torch.empty(T, D, dtype=torch.uint8, device="cuda")
    s = torch.empty(T, dtype=torch.float32, device="cuda")
    abi.ispa_quantize_rows_e4m3(xt, T, D, q, s)
    torch.cuda.synchronize()
    return q, s


def _gpu_quant_weight(W, dW):
    D, Do = W.shape
    Wt = torch.from_numpy(W).cuda()
    dWt = torch.from_numpy(dW).cuda() if dW is not None else None
    q = torch.empty(Do, D, dtype=torch.uint8, device="cuda")
    s = torch.empty(Do, dtype=torch.float32, device="cuda")
    abi.ispa_quantize_weight_e4m3(Wt, dWt, D, Do, q, s)
    torch.cuda.synchronize()
    return q, s


def _gpu_linear(aq, sa, wq, sw):
    T, D = aq.shape
    Do = wq.shape[0]
    out = torch.empty(T, Do, dtype=torch.bfloat16, device="cuda")
    abi.ispa_linear_w8a8(aq, sa, wq, sw, T, D, Do, out)
    torch.cuda.synchronize()
    return to_f32(out)


def _check_linear(y, aq, sa, wq, sw, rows=None):
    aq = aq if rows is None else aq[rows]
    sa = sa if rows is None else sa[rows]
    ref = qt.linear_w8a8(aq, sa, wq, sw)
    D = aq.shape[1]
    s_abs = (np.abs(qt.decode(aq)) @ np.abs(qt.decode(wq)).T) * sa[:, None].astype(np.float64) * \
        sw[None, :].astype(np.float64)
    bound = 2.0 ** -8 * np.abs(ref) + 2 * (D / 2 + 3) * 2.0 ** -24 * s_abs
    err = np.abs(y.astype(np.float64) - ref)
    assert np.isfinite(y).all()
    assert np.all(err <= bound), f"max err/bound {np.max(err / np.maximum(bound, 1e-30)):.3f}"
    return float(np.max(err / np.maximum(bound, 1e-30)))


@pytest.mark.parametrize("T,D", [(300, 256), (129, 1536), (1, 128)])
def test_quantize_rows_bit_exact(T, D):
    x = _activations(1, T, D)
    if T > 3:
        x[3] = 0.0                                   # an all-zero token
        x[2] *= 1e4                                  # a large-magnitude token
    x = synth.bf16_round(x)                          # the kernel reads bf16: feed both sides the same
    q, s = _gpu_quant_rows(x)
    rq, rs = qt.quantize_rows(x)
    bad = np.argwhere(q.cpu().numpy() != rq)
    assert len(bad) == 0, f"{len(bad)} codes differ, first at {bad[:3].tolist()}"
    assert np.array_equal(s.cpu().numpy(), rs)


@pytest.mark.parametrize("with_dw", [True, False])
def test_quantize_weight_bit_exact(with_dw):
    D, Do = 256, 384
    W = synth.make_weight(2, D, Do)
    dW = (0.05 * synth.make_weight(3, D, Do)).astype(np.float32) if with_dw else None
    W[:, 7] = 0.0                                    # an all-zero output channel (without dW)
    q, s = _gpu_quant_weight(W, dW)
    rq, rs = qt.quantize_weight(W, dW)
    assert np.array_equal(q.cpu().numpy(), rq)
    assert np.array_equal(s.cpu().numpy(), rs)


@pytest.mark.parametrize("T,D,Do", [(300, 256, 384), (300, 256, 512), (77, 384, 256), (130, 128, 128),
                                    (4611, 256, 1536)])
def test_linear_ragged_and_every_tile_width(T, D, Do):
    # D_out = 384 and 128 take the 128-column tile, 512 and 256 the 256-column tile, and 1536
    # with 37 row tiles the 192-column tile (296 tiles: two waves); T leaves a ragged last row tile
    x = _activations(4, T, D)
    W = synth.make_weight(5, D, Do)
    aq, sa = _gpu_quant_rows(x)
    wq, sw = _gpu_quant_weight(W, None)
    y = _gpu_linear(aq, sa, wq, sw)
    _check_linear(y, aq.cpu().numpy(), sa.cpu().numpy(), wq.cpu().numpy(), sw.cpu().numpy())


def test_projection_on_injected_weight_1p3b_shape():
    # the 1.3B-shaped output projection: 4680 tokens x 1536 -> 1536, weight W + dW
    T, D = 4680, 1536
    x = _activations(6, T, D)
    W = synth.make_weight(7, D, D)
    dW = (0.02 * synth.make_weight(8, D, D)).astype(np.float32)
    aq, sa = _gpu_quant_rows(x)
    wq, sw = _gpu_quant_weight(W, dW)
    raq, rsa = qt.quantize_rows(x)
    rwq, rsw = qt.quantize_weight(W, dW)
    assert np.array_equal(aq.cpu().numpy(), raq) and np.array_equal(sa.cpu().numpy(), rsa)
    assert np.array_equal(wq.cpu().numpy(), rwq) and np.array_equal(sw.cpu().numpy(), rsw)
    y = _gpu_linear(aq, sa, wq, sw)
    _check_linear(y, raq, rsa, rwq, rsw)
    # and the quantised layer tracks the full-precision one (a property, not a parity bound)
    full = x.astype(np.float64) @ (W.astype(np.float64) + dW)
    rel = np.linalg.norm(y - full) / np.linalg.norm(full)
    assert rel < 0.1, rel


def test_projection_14b_shape_sampled_rows():
    T, D = 4680, 5120
    x = _activations(9, T, D)
    W = synth.make_weight(10, D, D)
    aq, sa = _gpu_quant_rows(x)
    wq, sw = _gpu_quant_weight(W, None)
    y = _gpu_linear(aq, sa, wq, sw)
    rows = np.unique(np.concatenate([[0, 127, 128, 4607, 4608, 4679], np.random.default_rng(0).choice(T, 26, False)]))
    _check_linear(y[rows], aq.cpu().numpy(), sa.cpu().numpy(), wq.cpu().numpy(), sw.cpu().numpy(), rows=rows)


def test_back_to_back_calls_reuse_buffers():
    T, D, Do = 256, 256, 256
    x1, x2 = _activations(11, T, D), _activations(12, T, D)
    W = synth.make_weight(13, D, Do)
    wq, sw = _gpu_quant_weight(W, None)
    out = torch.empty(T, Do, dtype=torch.bfloat16, device="cuda")
    ys = []
    for x in (x1, x2):
        aq, sa = _gpu_quant_rows(x)
        abi.ispa_linear_w8a8(aq, sa, wq, sw, T, D, Do, out)
        torch.cuda.synchronize()
        ys.append((to_f32(out), aq.cpu().numpy(), sa.cpu().numpy()))
    for y, aq, sa in ys:
        _check_linear(y, aq, sa, wq.cpu().numpy(), sw.cpu().numpy())
