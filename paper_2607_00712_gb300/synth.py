"""Seeded synthetic inputs shared by the tests, the bench and the oracle checks.

This module only draws random numbers and rounds them to bfloat16; it holds
none of ISPA's arithmetic (no attention, no least squares, no ring mapping).
Both the CUDA path and the fp64 oracle consume exactly the arrays made here.

Input recipe (stand-in for the post-RoPE activations of an autoregressive
video DiT, Sec. 2, the KV injection of Eq. 3):
  * q, k, v ~ N(0, 1), drawn in fp32 with numpy's PCG64: each array gets its
    own child of SeedSequence(seed), split into 2^20-value chunks with one
    grandchild stream each (drawn in parallel threads, so the values depend
    only on the seed and the array shapes);
  * every key of frame f and head h additionally gets an offset vector
    mu[f, h, :] ~ N(0, 0.5^2) (0.5 read as the standard deviation), so the
    softmax over frames is non-uniform;
  * everything is rounded to bfloat16 (round to nearest even) before use, and
    both paths read the rounded values.
Token-major layout everywhere: a block of n frames is [n*P, H, d].
"""
from __future__ import annotations

import os
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass

import numpy as np

_CHUNK = 1 << 20

KEY_OFFSET_STD = 0.5


def bf16_round(x: np.ndarray) -> np.ndarray:
    """Round fp32 values to the nearest bfloat16 (ties to even); returns fp32."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32)
    # finite inputs: the sum stays below 2^32 (only NaN bit patterns are above 0xFFFF0000)
    r = (u >> 16) & np.uint32(1)
    r += np.uint32(0x7FFF)
    r += u
    r &= np.uint32(0xFFFF0000)
    return r.view(np.float32).reshape(x.shape)


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """Bit pattern (uint16) of fp32 values that are already bf16-representable."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    return (x.view(np.uint32) >> 16).astype(np.uint16)


def bits_to_f32(b: np.ndarray) -> np.ndarray:
    """fp32 values of a uint16 bf16 bit pattern."""
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def _normal(ss: np.random.SeedSequence, shape, std: float = 1.0) -> np.ndarray:
    """N(0, std^2) fp32 array of the given shape from the seed sequence ss."""
    n = int(np.prod(shape))
    out = np.empty(n, np.float32)
    n_chunks = max(1, (n + _CHUNK - 1) // _CHUNK)
    kids = ss.spawn(n_chunks)

    def work(i):
        g = np.random.Generator(np.random.PCG64(kids[i]))
        lo, hi = i * _CHUNK, min(n, (i + 1) * _CHUNK)
        if hi > lo:
            g.standard_normal(out=out[lo:hi], dtype=np.float32)

    if n_chunks == 1:
        work(0)
    else:
        with ThreadPoolExecutor(max_workers=min(16, os.cpu_count() or 1)) as ex:
            list(ex.map(work, range(n_chunks)))
    if std != 1.0:
        out *= np.float32(std)
    return out.reshape(shape)


def frame_block(ss: np.random.SeedSequence, n_frames: int, P: int, H: int, d: int,
                with_offset: bool = True) -> np.ndarray:
    """Keys of n_frames frames, [n*P, H, d] fp32, with the per-(frame, head) offset."""
    a, b = ss.spawn(2)
    k = _normal(a, (n_frames, P, H, d))
    if with_offset:
        mu = _normal(b, (n_frames, 1, H, d), KEY_OFFSET_STD)
        k += mu
    return k.reshape(n_frames * P, H, d)


@dataclass
class StepInputs:
    """One layer's inputs for one chunk step, all bf16-representable fp32.

    q, k_cur, v_cur : [n_chunk_frames*P, H, d]  (the chunk being denoised)
    k_hist, v_hist  : [n_past_frames*P, H, d]   (all past frames, logical order)
    """
    q: np.ndarray
    k_cur: np.ndarray
    v_cur: np.ndarray
    k_hist: np.ndarray
    v_hist: np.ndarray
    P: int
    H: int
    d: int

    @property
    def n_past_frames(self) -> int:
        return self.k_hist.shape[0] // self.P

    @property
    def n_q(self) -> int:
        return self.q.shape[0]


def make_step(seed: int, n_past_frames: int, P: int, H: int, d: int,
              n_chunk_frames: int = 3) -> StepInputs:
    """Seeded inputs of one chunk step (recipe in the module docstring)."""
    s_q, s_kc, s_vc, s_kh, s_vh = np.random.SeedSequence(seed).spawn(5)
    nq = n_chunk_frames * P
    q = bf16_round(_normal(s_q, (nq, H, d)))
    k_cur = bf16_round(frame_block(s_kc, n_chunk_frames, P, H, d))
    v_cur = bf16_round(_normal(s_vc, (nq, H, d)))
    k_hist = bf16_round(frame_block(s_kh, n_past_frames, P, H, d))
    v_hist = bf16_round(_normal(s_vh, (n_past_frames * P, H, d)))
    return StepInputs(q, k_cur, v_cur, k_hist, v_hist, P, H, d)


def make_activations(seed: int, T: int, D: int, coupling: float = 0.5):
    """Synthetic (A_loc, A_full) pair, [T, D] each, bf16-representable.

    A_full = A_loc + coupling * N(0,1) noise, so the discrepancy is of the size
    an attention output sees when half its history is removed.
    """
    s_a, s_n = np.random.SeedSequence(seed).spawn(2)
    a_loc = bf16_round(_normal(s_a, (T, D)))
    a_full = bf16_round(a_loc + _normal(s_n, (T, D), coupling))
    return a_loc, a_full


def make_weight(seed: int, D: int, D_out: int) -> np.ndarray:
    """A synthetic output-projection weight W [D, D_out] (row-vector convention A @ W)."""
    return (_normal(np.random.SeedSequence(seed), (D, D_out)) / np.float32(np.sqrt(D))).astype(np.float32)
