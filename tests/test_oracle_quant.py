"""Pins for oracle.quant: the e4m3 format against its own definition points, torch's float8
type (a library conversion), round-trip bounds and a brute-force linear layer."""
import math

import numpy as np
import pytest

from oracle import quant as qt

torch = pytest.importorskip("torch")
F8 = getattr(torch, "float8_e4m3fn", None)


def test_format_landmarks():
    # values fixed by the format definition
    assert qt.decode(0x00) == 0.0 and math.copysign(1.0, qt.decode(0x80)) == -1.0
    assert qt.decode(0x01) == 2.0 ** -9                   # smallest subnormal
    assert qt.decode(0x07) == 7 * 2.0 ** -9               # largest subnormal
    assert qt.decode(0x08) == 2.0 ** -6                   # smallest normal
    assert qt.decode(0x38) == 1.0                         # e = 7, m = 0
    assert qt.decode(0x7E) == 448.0 and qt.decode(0xFE) == -448.0
    assert np.isnan(qt.decode(0x7F)) and np.isnan(qt.decode(0xFF))
    finite = qt.DECODE_TABLE[:127]
    assert np.all(np.diff(finite) > 0)                    # codes 0..126 increase


@pytest.mark.skipif(F8 is None, reason="torch without float8_e4m3fn")
def test_decode_matches_torch_float8_for_all_codes():
    codes = torch.arange(256, dtype=torch.int32).to(torch.uint8)
    ref = codes.view(F8).to(torch.float64).numpy()
    ours = qt.decode(np.arange(256))
    both_nan = np.isnan(ref) & np.isnan(ours)
    assert np.all(both_nan | (ref == ours))
    assert np.array_equal(np.signbit(ref[~both_nan]), np.signbit(ours[~both_nan]))


def test_encode_representable_values_exactly():
    codes = np.array([c for c in range(256) if c not in (0x7F, 0xFF)], dtype=np.uint8)
    assert np.array_equal(qt.encode(qt.decode(codes)), codes)


def test_encode_midpoints_round_to_even_and_neighbours_to_nearest():
    v = qt.DECODE_TABLE[:127]
    mid = (v[:-1] + v[1:]) / 2                            # exact in float64
    got = qt.encode(mid)
    lo = np.arange(126)
    want = np.where(lo % 2 == 0, lo, lo + 1)              # the even code of the pair
    assert np.array_equal(got, want.astype(np.uint8))
    eps = np.minimum(v[1:] - v[:-1], 1.0) * 1e-6
    assert np.array_equal(qt.encode(mid - eps), lo.astype(np.uint8))
    assert np.array_equal(qt.encode(mid + eps), (lo + 1).astype(np.uint8))
    assert np.array_equal(qt.encode(-mid), (want | 0x80).astype(np.uint8))


def test_encode_saturates_and_keeps_nan():
    assert qt.encode(448.0) == 0x7E and qt.encode(463.9) == 0x7E and qt.encode(1e30) == 0x7E
    assert qt.encode(-1e30) == 0xFE and qt.encode(np.inf) == 0x7E
    assert qt.encode(np.nan) & 0x7F == 0x7F
    assert qt.encode(-0.0) == 0x80 and qt.encode(0.0) == 0x00
    assert qt.encode(2.0 ** -11) == 0x00                  # below half the smallest subnormal
    assert qt.encode(-(2.0 ** -10)) == 0x80               # exactly half: ties to the even code 0


@pytest.mark.skipif(F8 is None, reason="torch without float8_e4m3fn")
def test_encode_matches_torch_cast_in_range():
    r = np.random.default_rng(1)
    x = np.concatenate([r.standard_normal(20000) * 30, r.standard_normal(20000) * 0.01,
                        r.uniform(-448, 448, 20000)]).astype(np.float32)
    ref = torch.from_numpy(x).to(F8).view(torch.uint8).numpy()
    assert np.array_equal(qt.encode(x), ref)


def test_quantize_rows_round_trip_bound_and_amax_code():
    r = np.random.default_rng(2)
    x = (r.standard_normal((37, 256)) * r.uniform(0.01, 50, (37, 1))).astype(np.float32)
    x[5] = 0.0                                            # an all-zero row
    q, s = qt.quantize_rows(x)
    assert q.dtype == np.uint8 and s.shape == (37,) and s[5] == 1.0 and np.all(q[5] == 0)
    back = qt.decode(q) * s[:, None].astype(np.float64)
    err = np.abs(back - x)
    # relative half-spacing 2^-4 of a normal value; subnormal spacing 2^-9 * scale
    assert np.all(err <= 2.0 ** -4 * np.abs(x) + 2.0 ** -10 * s[:, None] + 1e-30)
    # each row's largest magnitude lands on +-448
    am = np.argmax(np.abs(x), axis=1)
    assert np.all(np.abs(qt.decode(q[np.arange(37), am]))[np.arange(37) != 5] == 448.0)


def test_quantize_weight_is_per_output_channel_of_w_plus_dw():
    r = np.random.default_rng(3)
    W = r.standard_normal((64, 48)).astype(np.float32)
    dW = (0.1 * r.standard_normal((64, 48))).astype(np.float32)
    q, s = qt.quantize_weight(W, dW)
    assert q.shape == (48, 64) and s.shape == (48,)
    Wn = (W + dW).astype(np.float32)
    q_cols, s_cols = qt.quantize_rows(np.ascontiguousarray(Wn.T))   # the same as rows of W'^T
    assert np.array_equal(q, q_cols) and np.array_equal(s, s_cols)


def test_linear_brute_force():
    r = np.random.default_rng(4)
    T, D, Do = 5, 7, 3
    aq = r.integers(0, 256, (T, D)).astype(np.uint8)
    wq = r.integers(0, 256, (Do, D)).astype(np.uint8)
    aq[aq & 0x7F == 0x7F] = 0x38                          # no NaN codes
    wq[wq & 0x7F == 0x7F] = 0x38
    sa = r.uniform(0.1, 2, T).astype(np.float32)
    sw = r.uniform(0.1, 2, Do).astype(np.float32)
    y = qt.linear_w8a8(aq, sa, wq, sw)
    for t in range(T):
        for n in range(Do):
            acc = sum(qt._value_of_code(int(aq[t, k])) * qt._value_of_code(int(wq[n, k])) for k in range(D))
            assert abs(y[t, n] - float(sa[t]) * float(sw[n]) * acc) <= 1e-12 * max(1.0, abs(y[t, n]))


def test_linear_identity_weight_returns_dequantised_activations():
    r = np.random.default_rng(5)
    x = r.standard_normal((9, 32)).astype(np.float32)
    aq, sa = qt.quantize_rows(x)
    wq, sw = qt.quantize_weight(np.eye(32, dtype=np.float32))
    assert np.all(sw == np.float32(1 / 448)) and np.all(qt.decode(np.diag(wq)) == 448.0)
    y = qt.linear_w8a8(aq, sa, wq, sw)
    assert np.allclose(y, qt.decode(aq) * sa[:, None], rtol=1e-6, atol=0)


def test_head_quantisation_and_dequantisation():
    r = np.random.default_rng(6)
    x = (r.standard_normal((50, 3, 16)) * np.array([0.1, 3.0, 40.0])[None, :, None]).astype(np.float32)
    x[:, 1, :] = 0.0                                     # an all-zero head
    q, s = qt.quantize_heads(x)
    assert s.dtype == np.float32 and s[1] == 1.0 and np.all(q[:, 1, :] == 0)
    amax = np.abs(x).max(axis=(0, 2))
    assert s[0] == np.float32(amax[0]) / np.float32(448) and s[2] == np.float32(amax[2]) / np.float32(448)
    back = qt.dequantize_heads(q, s)
    err = np.abs(back - x)
    assert np.all(err <= 2.0 ** -4 * np.abs(x) * (1 + 1e-6) + 2.0 ** -10 * s[None, :, None])
    # the largest magnitude of a head maps to (about) +-448: within one rounding of the division
    for h in (0, 2):
        i = np.unravel_index(np.argmax(np.abs(x[:, h, :])), x[:, h, :].shape)
        assert abs(qt.decode(q[i[0], h, i[1]])) in (416.0, 448.0)


def test_quantize_with_scale_saturates_outliers():
    x = np.array([[[1.0, -2.0, 1000.0, -1e6]]], dtype=np.float32)
    q = qt.quantize_heads_with_scale(x, np.array([1.0], np.float32))
    assert list(qt.decode(q).ravel()) == [1.0, -2.0, 448.0, -448.0]


def test_query_blocks_are_per_head_quantisation_of_each_block():
    r = np.random.default_rng(7)
    x = (r.standard_normal((300, 2, 8)) * r.uniform(0.1, 9, (300, 1, 1))).astype(np.float32)
    q, s = qt.quantize_query_blocks(x, block=128)
    assert s.shape == (2, 3)
    for b in range(3):
        qb, sb = qt.quantize_heads(x[b * 128:(b + 1) * 128])
        assert np.array_equal(q[b * 128:(b + 1) * 128], qb) and np.array_equal(s[:, b], sb)
    back = qt.dequantize_query_blocks(q, s)
    assert np.all(np.abs(back - x) <= 2.0 ** -4 * np.abs(x) * (1 + 1e-6) + 2.0 ** -10 * s.max())
