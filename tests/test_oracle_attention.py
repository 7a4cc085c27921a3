"""Pins for oracle.attention against closed forms, invariants and brute force.

Each pin is independent of the oracle's own code path: identities that the
softmax attention of Eq. 3 must satisfy, a pure-Python brute force over a
masked dense key list, and the LSE fusion of Eq. 11-12.
"""
import math

import numpy as np
import pytest

from oracle import attention as at
from oracle import keysets as ks
from paper_2607_00712_gb300 import synth


def _rng(seed=0):
    return np.random.default_rng(seed)


def test_values_all_one_gives_one():
    # Softmax rows sum to 1, so V == 1 makes every output exactly 1.
    r = _rng(1)
    q = r.standard_normal((7, 16))
    k = r.standard_normal((33, 16)) * 3
    o, _ = at.attend(q, k, np.ones((33, 16)), 0.25)
    assert np.max(np.abs(o - 1.0)) < 1e-14


def test_single_key_gives_its_value():
    r = _rng(2)
    q = r.standard_normal((5, 8))
    k = r.standard_normal((1, 8))
    v = r.standard_normal((1, 8))
    o, lse = at.attend(q, k, v, 0.7)
    assert np.allclose(o, np.broadcast_to(v, o.shape), atol=1e-15)
    assert np.allclose(lse, 0.7 * (q @ k.T)[:, 0], atol=1e-14)


def test_zero_query_gives_mean():
    r = _rng(3)
    k = r.standard_normal((40, 8))
    v = r.standard_normal((40, 8))
    o, lse = at.attend(np.zeros((3, 8)), k, v, 1.0)
    assert np.allclose(o, v.mean(axis=0), atol=1e-14)
    assert np.allclose(lse, math.log(40.0), atol=1e-14)


def test_key_shift_invariance():
    # Adding one vector c to every key adds q.c to every score of a row: no change.
    r = _rng(4)
    q, k, v = r.standard_normal((6, 8)), r.standard_normal((20, 8)), r.standard_normal((20, 8))
    c = r.standard_normal(8) * 5
    o1, l1 = at.attend(q, k, v, 0.5)
    o2, l2 = at.attend(q, k + c, v, 0.5)
    assert np.allclose(o1, o2, atol=1e-12)
    assert np.allclose(l2 - l1, 0.5 * (q @ c), atol=1e-12)


def test_key_permutation_invariance():
    r = _rng(5)
    q, k, v = r.standard_normal((6, 8)), r.standard_normal((20, 8)), r.standard_normal((20, 8))
    p = r.permutation(20)
    o1, l1 = at.attend(q, k, v, 0.5)
    o2, l2 = at.attend(q, k[p], v[p], 0.5)
    assert np.allclose(o1, o2, atol=1e-13) and np.allclose(l1, l2, atol=1e-13)


def test_empty_key_set():
    o, lse = at.attend(np.ones((2, 4)), np.zeros((0, 4)), np.zeros((0, 4)), 1.0)
    assert np.all(o == 0) and np.all(np.isneginf(lse))


def _brute_force(q, k_hist, v_hist, k_cur, v_cur, P, member, scale, chunk_member=None):
    """Masked dense softmax written with Python loops and math.exp.

    member(f) says whether past frame f is in the key set; chunk key j is in it for
    query i when chunk_member(i, j) (always, by default).
    """
    nq, H, d = q.shape
    nh = k_hist.shape[0]
    keys = [(None, k_hist[j], v_hist[j], member(j // P)) for j in range(nh)]
    keys += [(j, k_cur[j], v_cur[j], True) for j in range(k_cur.shape[0])]
    out = np.zeros((nq, H, d))
    lse = np.zeros((H, nq))
    for h in range(H):
        for i in range(nq):
            scores = []
            for cj, kk, _, use in keys:
                if cj is not None and chunk_member is not None:
                    use = chunk_member(i, cj)
                scores.append(scale * sum(float(q[i, h, c]) * float(kk[h, c]) for c in range(d))
                              if use else -math.inf)
            mx = max(scores)
            w = [math.exp(s - mx) if s != -math.inf else 0.0 for s in scores]
            tot = sum(w)
            for c in range(d):
                out[i, h, c] = sum(w[j] * float(keys[j][2][h, c]) for j in range(len(keys))) / tot
            lse[h, i] = mx + math.log(tot)
    return out, lse


@pytest.mark.parametrize("n_sink,n_recent", [(0, 2), (1, 0), (1, 1), (0, 0)])
def test_brute_force_tiny(n_sink, n_recent):
    P, H, d, F = 3, 2, 4, 5
    s = synth.make_step(11, F, P, H, d, n_chunk_frames=2)
    scale = 1.0 / math.sqrt(d)
    o_f, l_f = at.attn_full(s.q, s.k_hist, s.v_hist, s.k_cur, s.v_cur, P)
    b_f, bl_f = _brute_force(s.q, s.k_hist, s.v_hist, s.k_cur, s.v_cur, P, lambda f: True, scale)
    assert np.allclose(o_f, b_f, atol=1e-12) and np.allclose(l_f, bl_f, atol=1e-12)
    o_l, l_l = at.attn_local(s.q, s.k_hist, s.v_hist, s.k_cur, s.v_cur, P, n_sink, n_recent)
    b_l, bl_l = _brute_force(s.q, s.k_hist, s.v_hist, s.k_cur, s.v_cur, P,
                             lambda f: f < n_sink or f >= F - n_recent, scale)
    assert np.allclose(o_l, b_l, atol=1e-12) and np.allclose(l_l, bl_l, atol=1e-12)


def test_lse_fusion_reconstructs_full():
    # Eq. 11-12 applied to the local and history branches equals direct full attention.
    P, H, d, F = 8, 3, 16, 9
    s = synth.make_step(12, F, P, H, d)
    for n_sink, n_recent in [(0, 2), (1, 0), (1, 3), (2, 2)]:
        o_l, l_l = at.attn_local(s.q, s.k_hist, s.v_hist, s.k_cur, s.v_cur, P, n_sink, n_recent)
        o_h, l_h = at.attn_hist(s.q, s.k_hist, s.v_hist, P, n_sink, n_recent)
        fused, l_fused = at.lse_fuse(o_l, l_l, o_h, l_h)
        o_f, l_f = at.attn_full(s.q, s.k_hist, s.v_hist, s.k_cur, s.v_cur, P)
        assert np.allclose(fused, o_f, atol=1e-12)
        assert np.allclose(l_fused, l_f, atol=1e-12)


def test_lse_fusion_single_key_sets_closed_form():
    # One key per branch: the fused output is the two-way softmax blend of the values.
    a, b = 0.3, -1.1
    va, vb = np.array([[1.0, 2.0]]), np.array([[-3.0, 5.0]])
    fused, lse = at.lse_fuse(va, np.array([a]), vb, np.array([b]))
    wa = math.exp(a) / (math.exp(a) + math.exp(b))
    assert np.allclose(fused, wa * va + (1 - wa) * vb, atol=1e-15)
    assert abs(lse[0] - math.log(math.exp(a) + math.exp(b))) < 1e-15


def test_window_covering_cache_equals_full():
    P, H, d, F = 8, 2, 16, 6
    s = synth.make_step(13, F, P, H, d)
    o_f, l_f = at.attn_full(s.q, s.k_hist, s.v_hist, s.k_cur, s.v_cur, P)
    for n_sink, n_recent in [(0, F), (0, F + 5), (F, 0), (2, F - 2)]:
        o_l, l_l = at.attn_local(s.q, s.k_hist, s.v_hist, s.k_cur, s.v_cur, P, n_sink, n_recent)
        assert np.array_equal(o_l, o_f) and np.array_equal(l_l, l_f)


def test_dual_empty_history_gives_zero_discrepancy():
    P, H, d, F = 8, 2, 16, 3
    s = synth.make_step(14, F, P, H, d)
    r = at.attn_dual(s.q, s.k_hist, s.v_hist, s.k_cur, s.v_cur, P, 0, F)
    assert np.array_equal(r["a_full"], r["a_loc"])
    assert np.all(r["disc"] == 0) and r["disc_sq_sum"] == 0


def test_discrepancy_definition():
    # disc_t is the L2 norm over all H*d features of token t.
    r = _rng(6)
    a = r.standard_normal((5, 3, 4))
    b = a.copy()
    b[2, 1, 3] += 2.0
    b[4, 0, 0] -= 1.0
    b[4, 2, 1] += 1.0
    disc, tot = at.discrepancy(b, a)
    assert np.allclose(disc, [0, 0, 2.0, 0, math.sqrt(2.0)], atol=1e-15)
    assert abs(tot - 6.0) < 1e-14


def test_default_scale():
    assert at.default_scale(64) == 0.125 and at.default_scale(128, 0.3) == 0.3


def test_rows_subset_is_exact():
    P, H, d, F = 8, 2, 16, 4
    s = synth.make_step(15, F, P, H, d)
    rows = np.array([0, 5, 17, 23])
    o_all, l_all = at.attn_full(s.q, s.k_hist, s.v_hist, s.k_cur, s.v_cur, P)
    o_sub, l_sub = at.attn_full(s.q, s.k_hist, s.v_hist, s.k_cur, s.v_cur, P, rows=rows)
    assert np.allclose(o_sub, o_all[rows], atol=1e-15)
    assert np.allclose(l_sub, l_all[:, rows], atol=1e-15)


def test_keysets_used_by_local_match_eq7():
    # The local branch sees exactly the keys of ks.local_past_frames plus the chunk:
    # putting V=1 on exactly those keys and V=0 elsewhere makes full attention's output
    # equal the softmax mass of the local set, which must be exp(lse_loc - lse_full).
    P, H, d, F = 4, 1, 8, 7
    s = synth.make_step(16, F, P, H, d)
    n_sink, n_recent = 1, 2
    loc = ks.local_past_frames(F, n_sink, n_recent)
    v_hist = np.zeros_like(s.v_hist)
    for f in loc:
        v_hist[f * P:(f + 1) * P] = 1.0
    v_cur = np.ones_like(s.v_cur)
    o_f, l_f = at.attn_full(s.q, s.k_hist, v_hist, s.k_cur, v_cur, P)
    _, l_l = at.attn_local(s.q, s.k_hist, s.v_hist, s.k_cur, s.v_cur, P, n_sink, n_recent)
    assert np.allclose(o_f[:, 0, 0], np.exp(l_l[0] - l_f[0]), atol=1e-13)


# ------------------------------------------------------------------ frame-causal chunk option

@pytest.mark.parametrize("n_sink,n_recent", [(0, 2), (1, 0)])
def test_frame_causal_brute_force(n_sink, n_recent):
    # query i of chunk frame i // P sees chunk key j iff j // P <= i // P (frames up to its own)
    P, H, d, F = 3, 2, 4, 4
    s = synth.make_step(12, F, P, H, d, n_chunk_frames=3)
    scale = 1.0 / math.sqrt(d)
    causal = lambda i, j: j // P <= i // P  # noqa: E731
    o_f, l_f = at.attn_full(s.q, s.k_hist, s.v_hist, s.k_cur, s.v_cur, P, frame_causal=True)
    b_f, bl_f = _brute_force(s.q, s.k_hist, s.v_hist, s.k_cur, s.v_cur, P, lambda f: True, scale, causal)
    assert np.allclose(o_f, b_f, atol=1e-12) and np.allclose(l_f, bl_f, atol=1e-12)
    o_l, l_l = at.attn_local(s.q, s.k_hist, s.v_hist, s.k_cur, s.v_cur, P, n_sink, n_recent,
                             frame_causal=True)
    b_l, bl_l = _brute_force(s.q, s.k_hist, s.v_hist, s.k_cur, s.v_cur, P,
                             lambda f: f < n_sink or f >= F - n_recent, scale, causal)
    assert np.allclose(o_l, b_l, atol=1e-12) and np.allclose(l_l, bl_l, atol=1e-12)


def test_frame_causal_special_cases():
    P, H, d, F = 5, 2, 8, 3
    s = synth.make_step(13, F, P, H, d, n_chunk_frames=3)
    dense, ld = at.attn_full(s.q, s.k_hist, s.v_hist, s.k_cur, s.v_cur, P)
    causal, lc = at.attn_full(s.q, s.k_hist, s.v_hist, s.k_cur, s.v_cur, P, frame_causal=True)
    # the chunk's last frame sees the whole chunk: identical to the dense chunk
    assert np.array_equal(causal[2 * P:], dense[2 * P:]) and np.array_equal(lc[:, 2 * P:], ld[:, 2 * P:])
    # earlier frames do differ
    assert np.abs(causal[:P] - dense[:P]).max() > 1e-3
    # no past, chunk frame 0: plain attention over the chunk's first frame
    s0 = synth.make_step(14, 0, P, H, d, n_chunk_frames=3)
    o0, _ = at.attn_full(s0.q, s0.k_hist, s0.v_hist, s0.k_cur, s0.v_cur, P, frame_causal=True)
    want, _ = at.attend_heads(s0.q[:P], s0.k_cur[:P], s0.v_cur[:P], 1.0 / math.sqrt(d))
    assert np.allclose(o0[:P], want, atol=1e-13)
    # a one-frame chunk is unchanged by the option
    s1 = synth.make_step(15, F, P, H, d, n_chunk_frames=1)
    a, _ = at.attn_full(s1.q, s1.k_hist, s1.v_hist, s1.k_cur, s1.v_cur, P)
    b, _ = at.attn_full(s1.q, s1.k_hist, s1.v_hist, s1.k_cur, s1.v_cur, P, frame_causal=True)
    assert np.array_equal(a, b)
    # row subsets stay exact
    rows = np.array([0, 4, 7, 11, 14])
    sub, lsub = at.attn_full(s.q, s.k_hist, s.v_hist, s.k_cur, s.v_cur, P, rows=rows, frame_causal=True)
    assert np.allclose(sub, causal[rows], atol=1e-14) and np.allclose(lsub, lc[:, rows], atol=1e-14)


def test_frame_causal_fusion_identity():
    # Eq. 11-12 still reconstruct the full set: history frames are past frames, unmasked
    P, H, d, F = 4, 2, 8, 7
    s = synth.make_step(16, F, P, H, d, n_chunk_frames=3)
    loc, ll = at.attn_local(s.q, s.k_hist, s.v_hist, s.k_cur, s.v_cur, P, 1, 2, frame_causal=True)
    hist, lh = at.attn_hist(s.q, s.k_hist, s.v_hist, P, 1, 2)
    fused, lf = at.lse_fuse(loc, ll, hist, lh)
    full, lfull = at.attn_full(s.q, s.k_hist, s.v_hist, s.k_cur, s.v_cur, P, frame_causal=True)
    assert np.allclose(fused, full, atol=1e-12) and np.allclose(lf, lfull, atol=1e-12)


def test_frame_causal_needs_whole_frames():
    P, H, d = 4, 1, 4
    s = synth.make_step(17, 2, P, H, d, n_chunk_frames=2)
    with pytest.raises(ValueError):
        at.attn_full(s.q[:6], s.k_hist, s.v_hist, s.k_cur[:6], s.v_cur[:6], P, frame_causal=True)


def test_attend_weights_are_the_softmax_of_attend():
    # the weights reproduce attend's output and log-sum-exp (p V = O, max s + log L = LSE)
    r = np.random.default_rng(31)
    q, k, v = r.standard_normal((5, 8)), r.standard_normal((11, 8)), r.standard_normal((11, 3))
    p, L = at.attend_weights(q, k, 0.4)
    o, lse = at.attend(q, k, v, 0.4)
    assert np.allclose(p.sum(axis=1), 1.0, atol=1e-14) and np.allclose(p @ v, o, atol=1e-13)
    s = 0.4 * q @ k.T
    assert np.allclose(s.max(axis=1) + np.log(L), lse, atol=1e-13) and np.all(L >= 1.0)
