"""Shared set-up of the GPU parity tests: seeded inputs -> device ring + oracle view."""
from __future__ import annotations

import numpy as np

from oracle import keysets as ks
from paper_2607_00712_gb300 import abi, synth

# Tolerances on bf16 outputs with fp32 accumulation (attention).
MAX_ABS = 2e-2
MEAN_ABS = 2e-3


def assert_close_attn(got: np.ndarray, want: np.ndarray, what: str = ""):
    err = np.abs(np.asarray(got, np.float64) - np.asarray(want, np.float64))
    assert np.isfinite(got).all(), what
    assert err.max() <= MAX_ABS, f"{what}: max-abs {err.max():.3e}"
    assert err.mean() <= MEAN_ABS, f"{what}: mean-abs {err.mean():.3e}"
    return float(err.max()), float(err.mean())


def disc_bound(g_full, g_loc, g_disc, o_full, o_loc):
    """Per-token bound on |disc_gpu - disc_oracle| derived from the outputs themselves.

    disc_gpu,t = ||Gf_t - Gl_t|| is taken in fp32 over the stored bf16 outputs, disc_or,t =
    ||Of_t - Ol_t|| in fp64 over the exact ones.  By the triangle inequality
    | ||x|| - ||y|| | <= ||x - y||, so
        |disc_gpu,t - disc_or,t| <= ||(Gf_t - Of_t) - (Gl_t - Ol_t)|| + fp32 rounding,
    the rounding of a sum of D squares in chains of at most 64 + 2 + H terms being below
    1e-5 relative for every shape here (1e-6 absolute covers an exactly-zero discrepancy).
    """
    n = g_full.shape[0]
    e = (np.asarray(g_full, np.float64) - o_full).reshape(n, -1) - \
        (np.asarray(g_loc, np.float64) - o_loc).reshape(n, -1)
    return np.linalg.norm(e, axis=1) + 1e-5 * np.asarray(g_disc, np.float64) + 1e-6


def assert_disc_close(g_full, g_loc, g_disc, ref, what="", g_disc_sq_sum=None):
    """The dual pass's discrepancy against the oracle's, row by row and summed.

    ref: the oracle's attn_dual result for the same rows.  Per token the bound is
    disc_bound; for the sum of squares |sum g^2 - sum o^2| = |sum (g - o)(g + o)| <=
    sum b_t (g_t + o_t).  g_disc_sq_sum (optional) is the device accumulator of one call
    over exactly these rows; its fp32 summation adds at most 1e-5 relative.
    """
    g = np.asarray(g_disc, np.float64)
    o = np.asarray(ref["disc"], np.float64)
    b = disc_bound(g_full, g_loc, g, ref["a_full"], ref["a_loc"])
    err = np.abs(g - o)
    bad = np.nonzero(err > b)[0]
    assert len(bad) == 0, f"{what}: disc off by {err[bad[:4]]} > bound {b[bad[:4]]} at rows {bad[:4]}"
    sq_bound = float((b * (g + o)).sum())
    so = float((o * o).sum())
    assert abs(float((g * g).sum()) - so) <= sq_bound, f"{what}: sum disc^2"
    if g_disc_sq_sum is not None:
        assert abs(float(g_disc_sq_sum) - so) <= sq_bound + 1e-5 * so + 1e-6, f"{what}: disc_sq_sum"
    return float(err.max()), float(b.max())


class Step:
    """A chunk step on the device and the matching oracle inputs.

    The history is appended into the ring `group` frames at a time, the way an
    AR rollout appends each finished chunk.  `hist_res` is the history the
    oracle sees: the frames still resident in the ring, in logical order.
    """

    def __init__(self, seed, P, H, d, n_past, n_chunk_frames, capacity, n_sink_pinned=0, group=None,
                 device="cuda"):
        import torch

        from paper_2607_00712_gb300.device import Ring, bf16_tensor
        self.s = synth.make_step(seed, n_past, P, H, d, n_chunk_frames)
        self.P, self.H, self.d = P, H, d
        self.ring = Ring(H, d, P, capacity, n_sink_pinned, device)
        g = group or max(1, min(n_chunk_frames, capacity - n_sink_pinned))
        f = 0
        while f < n_past:
            n = min(g, n_past - f)
            k = bf16_tensor(self.s.k_hist[f * P:(f + n) * P], device)
            v = bf16_tensor(self.s.v_hist[f * P:(f + n) * P], device)
            abi.ispa_kv_append(self.ring.c, k, v, n)
            f += n
        torch.cuda.synchronize()
        res = ks.resident_frames(n_past, capacity, n_sink_pinned)
        self.resident = res
        self.k_hist_res = np.concatenate([self.s.k_hist[x * P:(x + 1) * P] for x in res]) if res else \
            self.s.k_hist[:0]
        self.v_hist_res = np.concatenate([self.s.v_hist[x * P:(x + 1) * P] for x in res]) if res else \
            self.s.v_hist[:0]
        self.q = bf16_tensor(self.s.q, device)
        self.kc = bf16_tensor(self.s.k_cur, device)
        self.vc = bf16_tensor(self.s.v_cur, device)
        self.n_q = self.s.q.shape[0]

    def oracle_args(self):
        return (self.s.q, self.k_hist_res, self.v_hist_res, self.s.k_cur, self.s.v_cur, self.P)
