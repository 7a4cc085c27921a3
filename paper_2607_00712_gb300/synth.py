"""Seeded synthetic inputs shared by the tests, the bench and the oracle checks.

This module only draws random numbers and rounds them to bfloat16; it holds
none of ISPA's arithmetic (no attention, no least squares, no ring mapping).
Both the CUDA path and the fp64 oracle consume exactly the arrays made here.

Input recipe (stand-in for the post-RoPE activations of an autoregressive
video DiT, Sec. 2 "KV injection", Eq. 3):
  * q, k, v ~ N(0, 1), drawn in fp32 from numpy's PCG64 with the given seed;
  * every key of frame f and head h additionally gets an offset vector
    mu[f, h, :] ~ N(0, 0.5^2) (0.5 read as the standard deviation), so the
    softmax over frames is non-uniform;
  * everything is rounded to bfloat16 (round to nearest even) before use, and
    both paths read the rounded values.
Token-major layout everywhere: a block of n frames is [n*P, H, d].
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

KEY_OFFSET_STD = 0.5


def bf16_round(x: np.ndarray) -> np.ndarray:
    """Round fp32 values to the nearest bfloat16 (ties to even); returns fp32."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32).reshape(x.shape)


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """Bit pattern (uint16) of fp32 values that are already bf16-representable."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    return (x.view(np.uint32) >> 16).astype(np.uint16)


def bits_to_f32(b: np.ndarray) -> np.ndarray:
    """fp32 values of a uint16 bf16 bit pattern."""
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def _normal(rng: np.random.Generator, shape, std: float = 1.0) -> np.ndarray:
    a = rng.standard_normal(size=shape, dtype=np.float32)
    if std != 1.0:
        a *= np.float32(std)
    return a


def frame_block(rng: np.random.Generator, n_frames: int, P: int, H: int, d: int,
                with_offset: bool = True) -> np.ndarray:
    """Keys of n_frames frames, [n*P, H, d] fp32, with the per-(frame, head) offset."""
    k = _normal(rng, (n_frames, P, H, d))
    if with_offset:
        mu = _normal(rng, (n_frames, 1, H, d), KEY_OFFSET_STD)
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
    rng = np.random.Generator(np.random.PCG64(seed))
    nq = n_chunk_frames * P
    q = bf16_round(_normal(rng, (nq, H, d)))
    k_cur = bf16_round(frame_block(rng, n_chunk_frames, P, H, d))
    v_cur = bf16_round(_normal(rng, (nq, H, d)))
    k_hist = bf16_round(frame_block(rng, n_past_frames, P, H, d))
    v_hist = bf16_round(_normal(rng, (n_past_frames * P, H, d)))
    return StepInputs(q, k_cur, v_cur, k_hist, v_hist, P, H, d)


def make_activations(seed: int, T: int, D: int, coupling: float = 0.5):
    """Synthetic (A_loc, A_full) pair, [T, D] each, bf16-representable.

    A_full = A_loc + coupling * N(0,1) noise, so the discrepancy is of the size
    an attention output sees when half its history is removed.
    """
    rng = np.random.Generator(np.random.PCG64(seed))
    a_loc = bf16_round(_normal(rng, (T, D)))
    a_full = bf16_round(a_loc + _normal(rng, (T, D), coupling))
    return a_loc, a_full


def make_weight(seed: int, D: int, D_out: int) -> np.ndarray:
    """A synthetic output-projection weight W [D, D_out] (row-vector convention A @ W)."""
    rng = np.random.Generator(np.random.PCG64(seed))
    return (_normal(rng, (D, D_out)) / np.float32(np.sqrt(D))).astype(np.float32)
