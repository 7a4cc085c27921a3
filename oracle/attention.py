"""Attention over key sets, dual warmup outputs, LSE fusion (oracle; fp64).

TEST INFRASTRUCTURE ONLY (see the package docstring).

Paper basis
  * Eq. 3: O = softmax(scale * Q K^T) V with K = [K_past; K_cur]; the chunk is
    dense inside itself (no mask within the step).
  * Sec. 3.1 phase 1 / Sec. 3.2: A_loc is the attention output over the local
    context only, A_full over the whole history; both are taken just before
    the output projection, so per token they are the heads concatenated,
    D = H * d.
  * Eq. 9-10: each branch returns (O, LSE), LSE the natural log-sum-exp of the
    scaled scores.
  * Eq. 11-12: LSE_full = log(exp(LSE_loc) + exp(LSE_hist)) and
    A_full = exp(LSE_loc - LSE_full) O_loc + exp(LSE_hist - LSE_full) O_hist.
  * Discrepancy (Sec. 3.1, tracked between the two branches): the paper does
    not define it; the reading used is disc_t = || A_full,t - A_loc,t ||_2
    over all D features of token t, plus the sum of disc_t^2 over tokens.

Frame-causal option (a variant beyond Eq. 3, which keeps the chunk dense): with
frame_causal=True a query of the chunk's frame a (rows a*P .. a*P+P-1) sees the
chunk's frames 0..a only; past frames stay fully visible.

Softmax scale: the paper does not state it; 1/sqrt(d) is used when scale is 0.
Each attention row is computed by materialising the whole score row and
taking two passes over it (max, then exponentials); there is no tiling and no
online rescaling.
"""
from __future__ import annotations

import math

import numpy as np

from .keysets import hist_past_frames, local_past_frames


def default_scale(d: int, scale: float = 0.0) -> float:
    return 1.0 / math.sqrt(d) if scale == 0.0 else float(scale)


def attend(q: np.ndarray, k: np.ndarray, v: np.ndarray, scale: float):
    """Softmax attention of one head.

    q [n, d], k [m, d], v [m, dv] -> (o [n, dv], lse [n]).  For m == 0 the
    output is 0 and lse is -inf (an empty key set contributes nothing).
    """
    q = np.asarray(q, dtype=np.float64)
    k = np.asarray(k, dtype=np.float64)
    v = np.asarray(v, dtype=np.float64)
    n = q.shape[0]
    if k.shape[0] == 0:
        return np.zeros((n, v.shape[1])), np.full(n, -np.inf)
    s = scale * (q @ k.T)                     # scores, one materialised row per query
    m = s.max(axis=1)                         # pass 1: row maximum
    e = np.exp(s - m[:, None])                # pass 2: exponentials
    l = e.sum(axis=1)
    o = (e @ v) / l[:, None]
    lse = m + np.log(l)
    return o, lse


def attend_weights(q: np.ndarray, k: np.ndarray, scale: float):
    """The softmax weights of one head, as `attend` forms them: q [n, d], k [m, d] ->
    (p [n, m], L [n]) with p = exp(s - max s) / L and L = sum exp(s - max s), s = scale q k^T."""
    q = np.asarray(q, dtype=np.float64)
    k = np.asarray(k, dtype=np.float64)
    s = scale * (q @ k.T)
    e = np.exp(s - s.max(axis=1)[:, None])
    L = e.sum(axis=1)
    return e / L[:, None], L


def attend_heads(q: np.ndarray, k: np.ndarray, v: np.ndarray, scale: float):
    """All heads: q [n, H, d], k/v [m, H, d] -> (o [n, H, d], lse [H, n])."""
    n, H, _ = q.shape
    o = np.zeros((n, H, v.shape[2]))
    lse = np.zeros((H, n))
    for h in range(H):
        o[:, h, :], lse[h] = attend(q[:, h, :], k[:, h, :], v[:, h, :], scale)
    return o, lse


def gather_frames(block: np.ndarray, frames: list[int], P: int) -> np.ndarray:
    """Rows of the given logical frames from a token-major [F*P, H, d] history."""
    if not frames:
        return block[:0]
    return np.concatenate([block[f * P:(f + 1) * P] for f in frames], axis=0)


def key_set(k_hist, v_hist, k_cur, v_cur, frames: list[int], P: int, with_chunk: bool = True):
    """(K, V) of a key set: the listed past frames, then the chunk (Eq. 3)."""
    ks = [gather_frames(k_hist, frames, P)]
    vs = [gather_frames(v_hist, frames, P)]
    if with_chunk:
        ks.append(k_cur)
        vs.append(v_cur)
    return np.concatenate(ks, axis=0), np.concatenate(vs, axis=0)


def _rows(x, rows):
    return x if rows is None else x[rows]


def _attend_with_chunk(q, k_past, v_past, k_cur, v_cur, P: int, scale: float, rows, frame_causal: bool):
    """Queries against the given past keys plus the chunk, dense or frame-causal."""
    if not frame_causal:
        K = np.concatenate([k_past, k_cur], axis=0)
        V = np.concatenate([v_past, v_cur], axis=0)
        return attend_heads(_rows(q, rows), K, V, scale)
    n = k_cur.shape[0]
    if n % P:
        raise ValueError("frame-causal attention needs whole chunk frames")
    idx = np.arange(q.shape[0]) if rows is None else np.asarray(rows)
    H, d = q.shape[1], v_cur.shape[2]
    out = np.zeros((len(idx), H, d))
    lse = np.zeros((H, len(idx)))
    for a in range(n // P):                   # queries of chunk frame a
        sel = np.nonzero(idx // P == a)[0]
        if len(sel) == 0:
            continue
        K = np.concatenate([k_past, k_cur[:(a + 1) * P]], axis=0)
        V = np.concatenate([v_past, v_cur[:(a + 1) * P]], axis=0)
        out[sel], lse[:, sel] = attend_heads(q[idx[sel]], K, V, scale)
    return out, lse


def attn_full(q, k_hist, v_hist, k_cur, v_cur, P: int, scale: float = 0.0, rows=None,
              frame_causal: bool = False):
    """F-layer step: every past frame plus the chunk (Eq. 3).

    rows: optional query-row indices (rows are independent, so a subset is
    exact for those rows).  Returns (out [n, H, d], lse [H, n]).
    """
    F = k_hist.shape[0] // P
    frames = list(range(F))
    return _attend_with_chunk(q, gather_frames(k_hist, frames, P), gather_frames(v_hist, frames, P), k_cur,
                              v_cur, P, default_scale(q.shape[2], scale), rows, frame_causal)


def attn_local(q, k_hist, v_hist, k_cur, v_cur, P: int, n_sink: int, n_recent: int,
               scale: float = 0.0, rows=None, frame_causal: bool = False):
    """L-layer step: sink frames, the n_recent newest past frames, the chunk (Eq. 7)."""
    F = k_hist.shape[0] // P
    frames = local_past_frames(F, n_sink, n_recent)
    return _attend_with_chunk(q, gather_frames(k_hist, frames, P), gather_frames(v_hist, frames, P), k_cur,
                              v_cur, P, default_scale(q.shape[2], scale), rows, frame_causal)


def attn_hist(q, k_hist, v_hist, P: int, n_sink: int, n_recent: int, scale: float = 0.0,
              rows=None):
    """History branch of Eq. 10: the past frames outside the local set, no chunk."""
    F = k_hist.shape[0] // P
    K, V = key_set(k_hist, v_hist, None, None, hist_past_frames(F, n_sink, n_recent), P,
                   with_chunk=False)
    return attend_heads(_rows(q, rows), K, V, default_scale(q.shape[2], scale))


def discrepancy(a_full: np.ndarray, a_loc: np.ndarray):
    """disc_t = ||A_full,t - A_loc,t||_2 over all features; and sum_t disc_t^2.

    a_full, a_loc: [n, H, d] or [n, D].
    """
    n = a_full.shape[0]
    delta = (np.asarray(a_full, np.float64) - np.asarray(a_loc, np.float64)).reshape(n, -1)
    sq = (delta * delta).sum(axis=1)
    return np.sqrt(sq), float(sq.sum())


def attn_dual(q, k_hist, v_hist, k_cur, v_cur, P: int, n_sink: int, n_recent: int,
              scale: float = 0.0, rows=None, frame_causal: bool = False):
    """Warmup dual step: A_full and A_loc of the same queries (Sec. 3.1, 3.4).

    A_full is computed directly over the full set (not through the fusion of
    Eq. 11-12, which is a separate function checked against this one).
    Returns dict with a_full, a_loc [n, H, d], lse_full, lse_loc [H, n],
    disc [n], disc_sq_sum.
    """
    a_full, lse_full = attn_full(q, k_hist, v_hist, k_cur, v_cur, P, scale, rows, frame_causal)
    a_loc, lse_loc = attn_local(q, k_hist, v_hist, k_cur, v_cur, P, n_sink, n_recent, scale, rows,
                                frame_causal)
    disc, disc_sq_sum = discrepancy(a_full, a_loc)
    return dict(a_full=a_full, a_loc=a_loc, lse_full=lse_full, lse_loc=lse_loc,
                disc=disc, disc_sq_sum=disc_sq_sum)


def lse_fuse(o_loc, lse_loc, o_hist, lse_hist):
    """Eq. 11-12: merge two (O, LSE) branches over disjoint key sets.

    o_* [n, dv] with lse_* [n] (or o_* [n, H, d] with lse_* [H, n]).
    A branch with lse = -inf (empty set) gets weight 0.
    """
    o_loc = np.asarray(o_loc, np.float64)
    o_hist = np.asarray(o_hist, np.float64)
    lse_loc = np.asarray(lse_loc, np.float64)
    lse_hist = np.asarray(lse_hist, np.float64)
    mx = np.maximum(lse_loc, lse_hist)
    lse_full = mx + np.log(np.exp(lse_loc - mx) + np.exp(lse_hist - mx))
    w_loc = np.exp(lse_loc - lse_full)
    w_hist = np.exp(lse_hist - lse_full)
    if o_loc.ndim == 3:                     # [n, H, d] with lse [H, n]
        w_loc = w_loc.T[:, :, None]
        w_hist = w_hist.T[:, :, None]
    else:
        w_loc = w_loc[:, None]
        w_hist = w_hist[:, None]
    return w_loc * o_loc + w_hist * o_hist, lse_full
