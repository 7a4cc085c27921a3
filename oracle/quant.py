"""8-bit (e4m3) weight/activation quantisation of a linear layer (oracle; test infrastructure only).

Paper basis
  * Sec. 4 (further analysis, post-training quantisation): the linear layers run with 8-bit
    weights and activations (W8A8) on top of ISPA; the layer whose weight ISPA changes is the
    attention output projection, W_new = W + dW (Sec. 3.2), so the quantised weight is that
    of W + dW.  The paper fixes no format; on this hardware the 8-bit tensor-core type is
    fp8 e4m3, so W8A8 is read as e4m3 codes with one fp32 scale per token (activations) and
    one per output channel (weights), scale = absmax / 448.

Format (OCP 8-bit floating point, e4m3 "fn" variant), restated from its definition:
  code = s eeee mmm.  e = 0: (-1)^s * m * 2^-9 (zero and subnormals);
  0 < e < 15, or e = 15 with m < 7: (-1)^s * (1 + m/8) * 2^(e-7);  e = 15, m = 7: NaN.
  Largest finite magnitude 448 (e = 15, m = 6); there are no infinities.
Encoding rounds to nearest, ties to the even code, keeps the sign of zero, and saturates
magnitudes above 448 to 448 (NaN stays NaN).

Quantisation, in fp32 as both sides compute it:
  amax = max |x| over the group; if amax == 0: inv = 1, scale = 1;
  else inv = fl32(448 / amax), scale = fl32(amax / 448); code = e4m3(fl32(x * inv)).
Linear: y[t, n] = a_scale[t] * w_scale[n] * sum_k dec(a_q[t, k]) * dec(w_q[n, k]), in float64
(the weight codes are stored K-major, [D_out][D]).

8-bit query/key attention (SageAttention's 8-bit Q K^T with 16-bit P V, cited in Sec. 3.4):
one scale per head, scale = fl32(amax / 448) over all the group's tokens (or a given scale, for
keys appended into a cache), code = e4m3(fl32(x * fl32(1 / scale))); queries take one scale
per head and block of 128 tokens (SageAttention's per-block granularity).  The attention is then
the plain attention of the dequantised q and k (codes times scale) with the unquantised v.
"""
from __future__ import annotations

import numpy as np

E4M3_MAX = 448.0


def _value_of_code(c: int) -> float:
    """Value of one e4m3 code from the format definition (NaN for the NaN codes)."""
    s = -1.0 if c & 0x80 else 1.0
    e = (c >> 3) & 0xF
    m = c & 0x7
    if e == 15 and m == 7:
        return float("nan")
    if e == 0:
        return s * m * 2.0 ** -9
    return s * (1.0 + m / 8.0) * 2.0 ** (e - 7)


DECODE_TABLE = np.array([_value_of_code(c) for c in range(256)], dtype=np.float64)
# non-negative finite values in code order (codes 0..126); they increase with the code
_POS = DECODE_TABLE[:127]


def decode(q) -> np.ndarray:
    """uint8 codes -> float64 values."""
    return DECODE_TABLE[np.asarray(q, dtype=np.uint8)]


def encode(x) -> np.ndarray:
    """float values -> uint8 e4m3 codes (round to nearest, ties to even, saturating)."""
    x = np.asarray(x, dtype=np.float64)
    a = np.abs(x)
    sign = np.signbit(x).astype(np.uint8) << 7
    code = np.zeros(x.shape, dtype=np.uint8)
    not_nan = ~np.isnan(x)
    sat = a >= E4M3_MAX
    # nearest code by search over the 127 non-negative finite values
    i = np.clip(np.searchsorted(_POS, a, side="left"), 1, 126)   # _POS[i-1] < a <= _POS[i] (inside)
    lo, hi = _POS[i - 1], _POS[i]
    d_lo, d_hi = a - lo, hi - a
    pick_hi = (d_hi < d_lo) | ((d_hi == d_lo) & ((i & 1) == 0))   # tie: the even code
    c = np.where(pick_hi, i, i - 1).astype(np.uint8)
    c = np.where(a == 0, 0, c).astype(np.uint8)
    c = np.where(sat, 126, c).astype(np.uint8)
    code[...] = np.where(not_nan, c | sign, 0x7F | sign)
    return code


def quantize_groups(x: np.ndarray, axis: int):
    """Per-group e4m3 quantisation along `axis` (the reduced axis): returns (codes, scale fp32)."""
    x = np.asarray(x, dtype=np.float32)
    amax = np.max(np.abs(x), axis=axis, keepdims=True).astype(np.float32)
    zero = amax == 0
    safe = np.where(zero, np.float32(1), amax)
    inv = np.where(zero, np.float32(1), np.float32(E4M3_MAX) / safe).astype(np.float32)
    scale = np.where(zero, np.float32(1), safe / np.float32(E4M3_MAX)).astype(np.float32)
    y = (x * inv).astype(np.float32)                  # one fp32 multiply, rounded to nearest
    return encode(y), np.squeeze(scale, axis=axis)


def quantize_rows(x):
    """Activations [T][D] -> (codes [T][D], scale [T]): one scale per token."""
    return quantize_groups(x, axis=1)


def quantize_weight(W, dW=None):
    """W (+ dW), fp32 [D][D_out] -> (codes [D_out][D] K-major, scale [D_out]): one scale per channel.

    W + dW is summed in fp32 (the weight injection of Sec. 3.2 as stored in fp32)."""
    W = np.asarray(W, dtype=np.float32)
    Wn = W if dW is None else (W + np.asarray(dW, dtype=np.float32)).astype(np.float32)
    codes, scale = quantize_groups(Wn, axis=0)         # per column of W' = per output channel
    return np.ascontiguousarray(codes.T), scale


def linear_w8a8(a_q, a_scale, w_q, w_scale) -> np.ndarray:
    """y [T][D_out] in float64 from e4m3 codes a_q [T][D], w_q [D_out][D] and their scales."""
    A = decode(a_q)
    Wt = decode(w_q)
    acc = A @ Wt.T
    return acc * np.asarray(a_scale, np.float64)[:, None] * np.asarray(w_scale, np.float64)[None, :]


def quantize_heads_with_scale(x, scale) -> np.ndarray:
    """Token-major [n][H][d] values and per-head scales [H] -> codes e4m3(fl32(x * fl32(1 / scale_h)))."""
    x = np.asarray(x, dtype=np.float32)
    inv = (np.float32(1) / np.asarray(scale, dtype=np.float32)).astype(np.float32)[None, :, None]
    return encode((x * inv).astype(np.float32))


def head_scales(x) -> np.ndarray:
    """Per-head scale fl32(amax / 448) of token-major [n][H][d] values (1 for an all-zero head)."""
    x = np.asarray(x, dtype=np.float32)
    amax = np.max(np.abs(x), axis=(0, 2)).astype(np.float32)
    return np.where(amax == 0, np.float32(1), amax / np.float32(E4M3_MAX)).astype(np.float32)


def quantize_heads(x):
    """[n][H][d] -> (codes, per-head scales [H])."""
    s = head_scales(x)
    return quantize_heads_with_scale(x, s), s


def dequantize_heads(q, scale) -> np.ndarray:
    """codes [n][H][d], scales [H] -> float64 values."""
    return decode(q) * np.asarray(scale, np.float64)[None, :, None]


def quantize_query_blocks(x, block: int = 128):
    """Queries [n][H][d] -> (codes, scales [H][ceil(n / block)]): one scale per head and block of
    `block` consecutive tokens, scale = fl32(amax / 448) (1 for an all-zero block)."""
    x = np.asarray(x, dtype=np.float32)
    n, H, _ = x.shape
    nb = (n + block - 1) // block
    scales = np.ones((H, nb), dtype=np.float32)
    codes = np.zeros(x.shape, dtype=np.uint8)
    for b in range(nb):
        xb = x[b * block:(b + 1) * block]
        s = head_scales(xb)
        scales[:, b] = s
        codes[b * block:(b + 1) * block] = quantize_heads_with_scale(xb, s)
    return codes, scales


def dequantize_query_blocks(q, scales, block: int = 128) -> np.ndarray:
    q = np.asarray(q)
    out = decode(q)
    for b in range(scales.shape[1]):
        out[b * block:(b + 1) * block] *= np.asarray(scales[:, b], np.float64)[None, :, None]
    return out

