"""GPU parity of the 8-bit query/key attention (e4m3 Q K^T, bf16 P V) through the C-ABI.

Queries carry one scale per head and block of 128 tokens, keys the ring's per-head scales (the
chunk's keys too).  Codes and scales are exact results of fp32 decisions taken alike on both sides: they
must equal the oracle's (oracle.quant) bit for bit.  The attention is then compared with the
oracle's attention of the dequantised q and k (codes times scales) and the bf16 v, within the
same tolerance as the bf16 path: max-abs 2e-2, mean-abs 2e-3 on the bf16 outputs.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from gpu_helpers import assert_close_attn, assert_disc_close  # noqa: E402
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


def _quant_heads(x):
    n, H, d = x.shape
    q = torch.empty(n, H, d, dtype=torch.uint8, device="cuda")
    s = torch.empty(H, dtype=torch.float32, device="cuda")
    abi.ispa_quantize_heads_e4m3(bf16_tensor(x), n, H, d, q, s)
    torch.cuda.synchronize()
    return q, s


def _quant_q(x):
    n, H, d = x.shape
    q = torch.empty(n, H, d, dtype=torch.uint8, device="cuda")
    s = torch.empty(H, (n + 127) // 128, dtype=torch.float32, device="cuda")
    abi.ispa_quantize_q_e4m3(bf16_tensor(x), n, H, d, q, s)
    torch.cuda.synchronize()
    return q, s


def _quant_k(x, scale):
    n, H, d = x.shape
    q = torch.empty(n, H, d, dtype=torch.uint8, device="cuda")
    abi.ispa_quantize_k_e4m3(bf16_tensor(x), n, H, d, scale, q)
    torch.cuda.synchronize()
    return q


class Qk8Step:
    """A chunk step with an e4m3-key ring built by ispa_kv_append_qk8, and its oracle view."""

    def __init__(self, seed, P, H, n_past, n_chunk_frames, capacity, n_sink_pinned=0, k_scale_boost=1.0):
        d = 128
        self.s = synth.make_step(seed, n_past, P, H, d, n_chunk_frames)
        self.P, self.H, self.d = P, H, d
        # the ring's key scales: from the history's keys (a caller would calibrate them once)
        k_ring_scale = qt.head_scales(self.s.k_hist if n_past else self.s.k_cur) * np.float32(k_scale_boost)
        self.k_ring_scale_np = k_ring_scale.astype(np.float32)
        self.k_ring_scale = torch.from_numpy(self.k_ring_scale_np).cuda()
        self.ring = Ring(H, d, P, capacity, n_sink_pinned, k_e4m3=True)
        g = max(1, min(n_chunk_frames, capacity - n_sink_pinned))
        f = 0
        while f < n_past:
            n = min(g, n_past - f)
            abi.ispa_kv_append_qk8(self.ring.c, bf16_tensor(self.s.k_hist[f * P:(f + n) * P]),
                                   bf16_tensor(self.s.v_hist[f * P:(f + n) * P]), n, self.k_ring_scale)
            f += n
        self.q8, self.q_scale = _quant_q(self.s.q)
        self.kc_scale = self.k_ring_scale                      # the chunk's keys use the ring's scales
        self.k8c = _quant_k(self.s.k_cur, self.kc_scale)
        self.vc = bf16_tensor(self.s.v_cur)
        self.n_q = self.s.q.shape[0]
        torch.cuda.synchronize()
        res = ks.resident_frames(n_past, capacity, n_sink_pinned)
        self.resident = res
        kh = np.concatenate([self.s.k_hist[x * P:(x + 1) * P] for x in res]) if res else self.s.k_hist[:0]
        vh = np.concatenate([self.s.v_hist[x * P:(x + 1) * P] for x in res]) if res else self.s.v_hist[:0]
        # oracle view: dequantised q and k, values as they are
        kh_hat = qt.dequantize_heads(qt.quantize_heads_with_scale(kh, k_ring_scale), k_ring_scale)
        q_hat = qt.dequantize_query_blocks(*qt.quantize_query_blocks(self.s.q))
        kc_hat = qt.dequantize_heads(qt.quantize_heads_with_scale(self.s.k_cur, k_ring_scale), k_ring_scale)
        self.args = (q_hat, kh_hat, vh, kc_hat, self.s.v_cur, P)

    def full(self):
        out = torch.empty(self.n_q, self.H * self.d, dtype=torch.bfloat16, device="cuda")
        lse = torch.empty(self.H, self.n_q, dtype=torch.float32, device="cuda")
        abi.ispa_attn_full_qk8(self.ring.c, self.k_ring_scale, self.q8, self.q_scale, self.k8c, self.kc_scale,
                               self.vc, self.n_q, 0.0, out, lse)
        torch.cuda.synchronize()
        return to_f32(out).reshape(self.n_q, self.H, self.d), to_f32(lse)

    def local(self, win):
        out = torch.empty(self.n_q, self.H * self.d, dtype=torch.bfloat16, device="cuda")
        lse = torch.empty(self.H, self.n_q, dtype=torch.float32, device="cuda")
        abi.ispa_attn_local_qk8(self.ring.c, self.k_ring_scale, Window(*win), self.q8, self.q_scale, self.k8c,
                                self.kc_scale, self.vc, self.n_q, 0.0, out, lse)
        torch.cuda.synchronize()
        return to_f32(out).reshape(self.n_q, self.H, self.d), to_f32(lse)


@pytest.mark.parametrize("n,H", [(300, 3), (4680, 12), (1, 1)])
def test_quantize_heads_bit_exact(n, H):
    x = synth.make_step(21, 0, n, H, 128, 1).q[:n]
    if H > 1:
        x[:, 1, :] *= 37.0
        x = synth.bf16_round(x)
    q, s = _quant_heads(x)
    rq, rs = qt.quantize_heads(x)
    assert np.array_equal(s.cpu().numpy(), rs)
    bad = np.argwhere(q.cpu().numpy() != rq)
    assert len(bad) == 0, f"{len(bad)} codes differ, first at {bad[:3].tolist()}"


@pytest.mark.parametrize("n,H", [(300, 3), (4680, 12), (77, 1)])
def test_quantize_q_blocks_and_given_scale_k_bit_exact(n, H):
    x = synth.make_step(27, 0, n, H, 128, 1).q[:n]
    x[: min(n, 50), 0, :] *= 20.0                         # blocks with different ranges
    x = synth.bf16_round(x)
    q, s = _quant_q(x)
    rq, rs = qt.quantize_query_blocks(x)
    assert np.array_equal(s.cpu().numpy(), rs)
    assert np.array_equal(q.cpu().numpy(), rq)
    ks_np = (qt.head_scales(x) * np.float32(0.7)).astype(np.float32)   # some codes saturate
    qk = _quant_k(x, torch.from_numpy(ks_np).cuda())
    assert np.array_equal(qk.cpu().numpy(), qt.quantize_heads_with_scale(x, ks_np))


def test_append_qk8_ring_contents_exact():
    P, H, cap = 100, 3, 4
    st = Qk8Step(22, P=P, H=H, n_past=6, n_chunk_frames=2, capacity=cap, n_sink_pinned=1)
    k_ring = st.ring.k.cpu().numpy()
    v_ring = st.ring.v.view(torch.int16).cpu().numpy()
    for f in st.resident:
        sl = ks.ring_slot(f, cap, 1)
        want_k = qt.quantize_heads_with_scale(st.s.k_hist[f * P:(f + 1) * P], st.k_ring_scale_np).transpose(1, 0, 2)
        assert np.array_equal(k_ring[:, sl * P:(sl + 1) * P], want_k), f
        want_v = synth.bf16_bits(st.s.v_hist[f * P:(f + 1) * P]).view(np.int16).transpose(1, 0, 2)
        assert np.array_equal(v_ring[:, sl * P:(sl + 1) * P], want_v), f
    assert st.ring.frames_written == 6


def test_qk8_attention_ragged_and_wrapped():
    # 100 tokens per frame (tiles straddle frames), 300 queries (ragged tail), a wrapped ring
    # with a pinned sink
    st = Qk8Step(23, P=100, H=3, n_past=12, n_chunk_frames=3, capacity=7, n_sink_pinned=1)
    o, l = st.full()
    ro, rl = at.attn_full(*st.args)
    assert_close_attn(o, ro, "qk8 full")
    assert np.abs(l - rl).max() < 2e-3
    for win in [(1, 2), (0, 3), (1, 0)]:
        o, l = st.local(win)
        ro, rl = at.attn_local(*st.args, *win)
        assert_close_attn(o, ro, f"qk8 local {win}")
        assert np.abs(l - rl).max() < 2e-3


def test_qk8_dual_matches_oracle():
    st = Qk8Step(28, P=100, H=3, n_past=9, n_chunk_frames=3, capacity=8, n_sink_pinned=1)
    D = st.H * st.d
    a_full = torch.empty(st.n_q, D, dtype=torch.bfloat16, device="cuda")
    a_loc = torch.empty_like(a_full)
    disc = torch.empty(st.n_q, dtype=torch.float32, device="cuda")
    dsum = torch.zeros(1, dtype=torch.float32, device="cuda")
    wsb = abi.ispa_attn_dual_workspace_size(st.H, st.n_q)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    abi.ispa_attn_dual_qk8(st.ring.c, st.k_ring_scale, Window(1, 2), st.q8, st.q_scale, st.k8c, st.kc_scale, st.vc,
                           st.n_q, 0.0, a_full, a_loc, disc, dsum, None, None, ws, wsb)
    torch.cuda.synchronize()
    r = at.attn_dual(*st.args, 1, 2)
    assert_close_attn(to_f32(a_full).reshape(r["a_full"].shape), r["a_full"], "qk8 dual full")
    assert_close_attn(to_f32(a_loc).reshape(r["a_loc"].shape), r["a_loc"], "qk8 dual loc")
    got = to_f32(disc)
    assert_disc_close(to_f32(a_full).reshape(r["a_full"].shape), to_f32(a_loc).reshape(r["a_loc"].shape), got, r,
                      "qk8 disc", float(dsum.item()))
    own = np.sqrt(((to_f32(a_full).astype(np.float64) - to_f32(a_loc)) ** 2).sum(1))
    assert np.allclose(got, own, rtol=1e-5, atol=1e-6)


def test_qk8_saturated_ring_keys_still_match_their_dequantised_values():
    # ring scales deliberately too small: the largest keys saturate at +-448 codes, and the
    # attention is that of the saturated (dequantised) keys
    st = Qk8Step(24, P=64, H=2, n_past=5, n_chunk_frames=2, capacity=6, k_scale_boost=0.5)
    o, _ = st.full()
    ro, _ = at.attn_full(*st.args)
    assert_close_attn(o, ro, "qk8 saturated")


def test_qk8_config1_sampled_rows():
    st = Qk8Step(25, P=1560, H=12, n_past=18, n_chunk_frames=3, capacity=18)
    rows = np.unique(np.concatenate([[0, 127, 128, 4607, 4608, 4679], np.random.default_rng(2).choice(4680, 42, False)]))
    o, _ = st.full()
    ro, _ = at.attn_full(*st.args, rows=rows)
    assert_close_attn(o[rows], ro, "qk8 config1 full")
    o, _ = st.local((0, 6))
    ro, _ = at.attn_local(*st.args, 0, 6, rows=rows)
    assert_close_attn(o[rows], ro, "qk8 config1 local")


def test_qk8_rejects_mismatched_ring_formats():
    st = Qk8Step(26, P=64, H=2, n_past=2, n_chunk_frames=1, capacity=4)
    out = torch.empty(st.n_q, st.H * st.d, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(abi.IspaError):
        abi.ispa_attn_full(st.ring.c, st.q8, st.k8c, st.vc, st.n_q, 0.0, out)       # e4m3 ring, bf16 call
    bring = Ring(st.H, st.d, st.P, 4)
    with pytest.raises(abi.IspaError):
        abi.ispa_attn_full_qk8(bring.c, st.k_ring_scale, st.q8, st.q_scale, st.k8c, st.kc_scale, st.vc, st.n_q,
                               0.0, out)
    with pytest.raises(abi.IspaError):
        abi.ispa_kv_append(st.ring.c, st.vc, st.vc, 1)
