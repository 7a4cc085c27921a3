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
