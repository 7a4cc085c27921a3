"""GPU parity of the 8-bit Q K^T and P V attention (SageAttention's fp8 P V form) through the C-ABI.

Keys and values carry the ring's per-head scales (the chunk's too), queries one scale per head
and block of 128 tokens.  Codes are exact results of fp32 decisions taken alike on both sides:
the key codes and the d-major value codes must equal the oracle's (oracle.quant) bit for bit.
The attention is compared with the oracle's attention of the dequantised q, k and v.  What the
kernel adds beyond the bf16 path is the e4m3 rounding of the probabilities: each weight p_i of a
row is used with relative error <= 2^-4, or absolute error <= 2^-14 / L where e4m3 is subnormal
(P is scaled by 2^4 before rounding against a running maximum within 2^4 of the row's, and
L = sum_i exp(s_i - max s) <= the kernel's row sum), so per output element

    |o_gpu - o| <= 2^-4 sum_i p_i |v_i| + 2^-14 sum_i |v_i| / L   (+ the bf16 path's tolerance),

computed here from the oracle's own weights.  Mean-abs errors must stay within the mean of that
bound plus the bf16 path's mean tolerance.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from gpu_helpers import MAX_ABS, MEAN_ABS, assert_disc_close  # noqa: E402
from oracle import attention as at  # noqa: E402
from oracle import keysets as ks  # noqa: E402
from oracle import quant as qt  # noqa: E402
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


def _vt_ld(n):
    return (n + 15) // 16 * 16


def _quant_vt(x, scale, fill=0):
    n, H, d = x.shape
    ld = _vt_ld(n)
    out = torch.full((H, d, ld), fill, dtype=torch.uint8, device="cuda")
    abi.ispa_quantize_vt_e4m3(bf16_tensor(x), n, H, d, scale, out, ld)
    torch.cuda.synchronize()
    return out, ld


class Kv8Step:
    """A chunk step over a ring with e4m3 keys and d-major e4m3 values, and its oracle view."""

    def __init__(self, seed, P, H, n_past, n_chunk_frames, capacity, n_sink_pinned=0):
        d = 128
        self.s = synth.make_step(seed, n_past, P, H, d, n_chunk_frames)
        self.P, self.H, self.d = P, H, d
        src_k = self.s.k_hist if n_past else self.s.k_cur
        src_v = self.s.v_hist if n_past else self.s.v_cur
        self.k_scale_np = qt.head_scales(src_k).astype(np.float32)
        self.v_scale_np = qt.head_scales(src_v).astype(np.float32)
        self.k_scale = torch.from_numpy(self.k_scale_np).cuda()
        self.v_scale = torch.from_numpy(self.v_scale_np).cuda()
        self.ring = Ring(H, d, P, capacity, n_sink_pinned, kv_e4m3=True)
        g = max(1, min(n_chunk_frames, capacity - n_sink_pinned))
        f = 0
        while f < n_past:
            n = min(g, n_past - f)
            abi.ispa_kv_append_kv8(self.ring.c, bf16_tensor(self.s.k_hist[f * P:(f + n) * P]),
                                   bf16_tensor(self.s.v_hist[f * P:(f + n) * P]), n, self.k_scale, self.v_scale)
            f += n
        self.n_q = self.s.q.shape[0]
        q8 = torch.empty(self.n_q, H, d, dtype=torch.uint8, device="cuda")
        qs = torch.empty(H, (self.n_q + 127) // 128, dtype=torch.float32, device="cuda")
        abi.ispa_quantize_q_e4m3(bf16_tensor(self.s.q), self.n_q, H, d, q8, qs)
        k8 = torch.empty(self.n_q, H, d, dtype=torch.uint8, device="cuda")
        abi.ispa_quantize_k_e4m3(bf16_tensor(self.s.k_cur), self.n_q, H, d, self.k_scale, k8)
        self.q8, self.q_scale, self.k8c = q8, qs, k8
        self.vt8c, self.vt_ld = _quant_vt(self.s.v_cur, self.v_scale)
        torch.cuda.synchronize()
        res = ks.resident_frames(n_past, capacity, n_sink_pinned)
        self.resident = res
        kh = np.concatenate([self.s.k_hist[x * P:(x + 1) * P] for x in res]) if res else self.s.k_hist[:0]
        vh = np.concatenate([self.s.v_hist[x * P:(x + 1) * P] for x in res]) if res else self.s.v_hist[:0]
        deq = lambda x, sc: qt.dequantize_heads(qt.quantize_heads_with_scale(x, sc), sc)  # noqa: E731
        q_hat = qt.dequantize_query_blocks(*qt.quantize_query_blocks(self.s.q))
        self.args = (q_hat, deq(kh, self.k_scale_np), deq(vh, self.v_scale_np), deq(self.s.k_cur, self.k_scale_np),
                     deq(self.s.v_cur, self.v_scale_np), P)

    def full(self):
        out = torch.empty(self.n_q, self.H * self.d, dtype=torch.bfloat16, device="cuda")
        lse = torch.empty(self.H, self.n_q, dtype=torch.float32, device="cuda")
        abi.ispa_attn_full_kv8(self.ring.c, self.k_scale, self.v_scale, self.q8, self.q_scale, self.k8c, self.k_scale,
                               self.vt8c, self.vt_ld, self.n_q, 0.0, out, lse)
        torch.cuda.synchronize()
        return to_f32(out).reshape(self.n_q, self.H, self.d), to_f32(lse)

    def local(self, win):
        out = torch.empty(self.n_q, self.H * self.d, dtype=torch.bfloat16, device="cuda")
        lse = torch.empty(self.H, self.n_q, dtype=torch.float32, device="cuda")
        abi.ispa_attn_local_kv8(self.ring.c, self.k_scale, self.v_scale, Window(*win), self.q8, self.q_scale,
                                self.k8c, self.k_scale, self.vt8c, self.vt_ld, self.n_q, 0.0, out, lse)
        torch.cuda.synchronize()
        return to_f32(out).reshape(self.n_q, self.H, self.d), to_f32(lse)

    def dual(self, win):
        D = self.H * self.d
        a_full = torch.empty(self.n_q, D, dtype=torch.bfloat16, device="cuda")
        a_loc = torch.empty_like(a_full)
        disc = torch.empty(self.n_q, dtype=torch.float32, device="cuda")
        dsum = torch.zeros(1, dtype=torch.float32, device="cuda")
        wsb = abi.ispa_attn_dual_workspace_size(self.H, self.n_q)
        ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
        abi.ispa_attn_dual_kv8(self.ring.c, self.k_scale, self.v_scale, Window(*win), self.q8, self.q_scale,
                               self.k8c, self.k_scale, self.vt8c, self.vt_ld, self.n_q, 0.0, a_full, a_loc, disc,
                               dsum, None, None, ws, wsb)
        torch.cuda.synchronize()
        shape = (self.n_q, self.H, self.d)
        return to_f32(a_full).reshape(shape), to_f32(a_loc).reshape(shape), to_f32(disc), float(dsum.item())

    def key_set(self, frames_local=None):
        """(K, V) of the full set, or of the past frames listed plus the chunk (dequantised)."""
        q_hat, kh, vh, kc, vc, P = self.args
        F = kh.shape[0] // P
        frames = list(range(F)) if frames_local is None else frames_local
        return at.key_set(kh, vh, kc, vc, frames, P)


def p_rounding_bound(q, K, V, rows=None):
    """Per output element: 2^-4 sum_i p_i |v_i| + 2^-14 sum_i |v_i| / L, from the oracle's weights."""
    q = q if rows is None else q[rows]
    n, H, d = q.shape
    b = np.zeros((n, H, d))
    for h in range(H):
        p, L = at.attend_weights(q[:, h], K[:, h], 1.0 / np.sqrt(d))
        av = np.abs(V[:, h])
        b[:, h] = 2.0 ** -4 * (p @ av) + 2.0 ** -14 * av.sum(axis=0)[None, :] / L[:, None]
    return b


def assert_close_kv8(got, want, bound, what=""):
    err = np.abs(np.asarray(got, np.float64) - want)
    assert np.isfinite(got).all(), what
    excess = err - (bound + MAX_ABS)
    i = np.unravel_index(np.argmax(excess), excess.shape)
    assert excess.max() <= 0, f"{what}: err {err[i]:.3e} > bound {bound[i]:.3e} + {MAX_ABS} at {i}"
    assert err.mean() <= bound.mean() + MEAN_ABS, f"{what}: mean-abs {err.mean():.3e}, bound mean {bound.mean():.3e}"
    return float(err.max()), float(err.mean()), float(bound.mean())


@pytest.mark.parametrize("n,H", [(300, 3), (4680, 12), (77, 1)])
def test_quantize_vt_bit_exact_and_padding_untouched(n, H):
    x = synth.make_step(41, 0, n, H, 128, 1).q[:n]
    sc = (qt.head_scales(x) * np.float32(0.8)).astype(np.float32)        # some codes saturate
    out, ld = _quant_vt(x, torch.from_numpy(sc).cuda(), fill=0xAB)
    o = out.cpu().numpy()
    want = qt.quantize_heads_with_scale(x, sc).transpose(1, 2, 0)        # [H][d][n]
    assert np.array_equal(o[:, :, :n], want)
    assert np.all(o[:, :, n:] == 0xAB)


def test_append_kv8_ring_contents_exact():
    P, H, cap = 100, 3, 4
    st = Kv8Step(42, P=P, H=H, n_past=6, n_chunk_frames=2, capacity=cap, n_sink_pinned=1)
    k_ring = st.ring.k.cpu().numpy()
    v_ring = st.ring.v.cpu().numpy()                                     # [H][128][vt_stride]
    assert v_ring.shape[2] == abi.ispa_ring_vt_stride(st.ring.c) == (cap * P + 15) // 16 * 16
    for f in st.resident:
        sl = ks.ring_slot(f, cap, 1)
        want_k = qt.quantize_heads_with_scale(st.s.k_hist[f * P:(f + 1) * P], st.k_scale_np).transpose(1, 0, 2)
        assert np.array_equal(k_ring[:, sl * P:(sl + 1) * P], want_k), f
        want_v = qt.quantize_heads_with_scale(st.s.v_hist[f * P:(f + 1) * P], st.v_scale_np).transpose(1, 2, 0)
        assert np.array_equal(v_ring[:, :, sl * P:(sl + 1) * P], want_v), f
    assert st.ring.frames_written == 6
    assert abi.ispa_ring_bytes(st.ring.c) == H * cap * P * 128 + H * 128 * v_ring.shape[2]


def _check_modes(st, wins, rows=None):
    q_hat = st.args[0]
    o, l = st.full()
    K, V = st.key_set()
    ro, rl = at.attn_full(*st.args, rows=rows)
    sel = slice(None) if rows is None else rows
    assert_close_kv8(o[sel], ro, p_rounding_bound(q_hat, K, V, rows), "kv8 full")
    assert np.abs(l[:, sel] - rl).max() < 2e-3
    F = st.args[1].shape[0] // st.P
    for win in wins:
        frames = ks.local_past_frames(F, *win)
        Kl, Vl = st.key_set(frames)
        o, l = st.local(win)
        ro, rl = at.attn_local(*st.args, *win, rows=rows)
        assert_close_kv8(o[sel], ro, p_rounding_bound(q_hat, Kl, Vl, rows), f"kv8 local {win}")
        assert np.abs(l[:, sel] - rl).max() < 2e-3
        af, al, disc, dsum = st.dual(win)
        r = at.attn_dual(*st.args, *win, rows=rows)
        assert_close_kv8(af[sel], r["a_full"], p_rounding_bound(q_hat, K, V, rows), f"kv8 dual full {win}")
        assert_close_kv8(al[sel], r["a_loc"], p_rounding_bound(q_hat, Kl, Vl, rows), f"kv8 dual loc {win}")
        assert_disc_close(af[sel], al[sel], disc[sel], r, f"kv8 disc {win}", dsum if rows is None else None)


def test_kv8_attention_ragged_wrapped_every_shift():
    # 100 tokens per frame: ring segments start at keys 100 * slot, so the value windows are
    # shifted by 0, 4, 8 and 12 keys; 300 queries (ragged tail), a wrapped ring with a sink
    st = Kv8Step(43, P=100, H=3, n_past=12, n_chunk_frames=3, capacity=7, n_sink_pinned=1)
    _check_modes(st, [(1, 2), (0, 3), (1, 0)])


def test_kv8_attention_small_frames_and_no_history():
    st = Kv8Step(44, P=64, H=2, n_past=5, n_chunk_frames=2, capacity=6)
    _check_modes(st, [(0, 2)])
    st0 = Kv8Step(45, P=36, H=2, n_past=0, n_chunk_frames=3, capacity=4)
    o, _ = st0.full()
    ro, _ = at.attn_full(*st0.args)
    K, V = st0.key_set()
    assert_close_kv8(o, ro, p_rounding_bound(st0.args[0], K, V), "kv8 chunk only")


def test_kv8_values_all_one():
    # every value 1 (codes 448 with scale 1/448): each output is sum_i p^_i / l, within the
    # rounding bound of 1
    st = Kv8Step(46, P=64, H=2, n_past=3, n_chunk_frames=2, capacity=4)
    ones = np.ones((st.s.v_hist.shape[0], 2, 128), np.float32)
    st.v_scale_np[:] = np.float32(1.0 / 448.0)
    st.v_scale.copy_(torch.from_numpy(st.v_scale_np))
    ring = Ring(2, 128, 64, 4, 0, kv_e4m3=True)
    abi.ispa_kv_append_kv8(ring.c, bf16_tensor(st.s.k_hist), bf16_tensor(ones), 3, st.k_scale, st.v_scale)
    st.ring = ring
    st.vt8c, st.vt_ld = _quant_vt(np.ones_like(st.s.v_cur), st.v_scale)
    o, _ = st.full()
    assert np.abs(o - 1.0).max() <= 2.0 ** -4 + 2.0 ** -8


def test_kv8_config1_sampled_rows():
    # the 1.3B-shaped step: 12 heads, 1560 tokens per frame (value windows shifted by 0 or 8
    # keys), 18 cached frames, window of 6
    st = Kv8Step(47, P=1560, H=12, n_past=18, n_chunk_frames=3, capacity=18)
    rows = np.unique(np.concatenate([[0, 127, 128, 4607, 4608, 4679], np.random.default_rng(3).choice(4680, 26, False)]))
    _check_modes(st, [(0, 6)], rows=rows)


def test_kv8_rejects_mismatched_rings_and_strides():
    st = Kv8Step(48, P=64, H=2, n_past=2, n_chunk_frames=1, capacity=4)
    out = torch.empty(st.n_q, 256, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(abi.IspaError) as e:   # a stride below n_q
        abi.ispa_attn_full_kv8(st.ring.c, st.k_scale, st.v_scale, st.q8, st.q_scale, st.k8c, st.k_scale, st.vt8c,
                               8, st.n_q, 0.0, out)
    assert e.value.status == abi.ISPA_ERR_INVALID_ARG
    with pytest.raises(abi.IspaError) as e:   # the 8-bit Q K^T call on a ring with e4m3 values
        abi.ispa_attn_full_qk8(st.ring.c, st.k_scale, st.q8, st.q_scale, st.k8c, st.k_scale, st.vt8c, st.n_q, 0.0,
                               out)
    assert e.value.status == abi.ISPA_ERR_INVALID_ARG
    r1 = Ring(2, 128, 64, 4, 0, k_e4m3=True)
    with pytest.raises(abi.IspaError) as e:   # the 8-bit P V call on a ring with bf16 values
        abi.ispa_attn_full_kv8(r1.c, st.k_scale, st.v_scale, st.q8, st.q_scale, st.k8c, st.k_scale, st.vt8c,
                               st.vt_ld, st.n_q, 0.0, out)
    assert e.value.status == abi.ISPA_ERR_INVALID_ARG
    r2 = abi.KVRing(2, 128, 62, 4, 0, abi.ISPA_KV_KV_E4M3, 0, st.ring.k.data_ptr(), st.ring.v.data_ptr())
    with pytest.raises(abi.IspaError) as e:   # tokens per frame not a multiple of 4
        abi.ispa_attn_full_kv8(r2, st.k_scale, st.v_scale, st.q8, st.q_scale, st.k8c, st.k_scale, st.vt8c,
                               st.vt_ld, st.n_q, 0.0, out)
    assert e.value.status == abi.ISPA_ERR_UNSUPPORTED
