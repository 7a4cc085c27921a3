"""Device-memory helpers (PyTorch allocates; libispa computes)."""
from __future__ import annotations

import numpy as np
import torch

from ._lib import KVRing, LSState, Window, ispa_ls_state_bytes


def bf16_tensor(x: np.ndarray, device="cuda") -> torch.Tensor:
    """bf16 tensor holding the (already bf16-representable) fp32 array x, bit for bit."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    bits = (x.view(np.uint32) >> 16).astype(np.uint16).view(np.int16)
    return torch.from_numpy(bits).view(torch.bfloat16).to(device)


def to_f32(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy()


class Ring:
    """A caller-owned KV ring: K and V [H][cap*P][d] tensors plus the C struct.

    k_e4m3: keys as e4m3 codes (uint8), for the 8-bit query/key attention entry points.
    kv_e4m3: keys as e4m3 codes and values as d-major e4m3 codes [H][d][vt_stride], for the
    8-bit Q K^T and P V entry points."""

    def __init__(self, num_heads: int, head_dim: int, tokens_per_frame: int, capacity_frames: int,
                 n_sink_frames: int = 0, device="cuda", k_e4m3: bool = False, kv_e4m3: bool = False):
        keys = capacity_frames * tokens_per_frame
        shape = (num_heads, keys, head_dim)
        fmt = 2 if kv_e4m3 else (1 if k_e4m3 else 0)
        self.k = torch.zeros(shape, dtype=torch.uint8 if fmt else torch.bfloat16, device=device)
        if kv_e4m3:
            self.vt_stride = (keys + 15) // 16 * 16
            self.v = torch.zeros(num_heads, head_dim, self.vt_stride, dtype=torch.uint8, device=device)
        else:
            self.v = torch.zeros(shape, dtype=torch.bfloat16, device=device)
        self.c = KVRing(num_heads, head_dim, tokens_per_frame, capacity_frames, n_sink_frames, fmt,
                        0, self.k.data_ptr(), self.v.data_ptr())

    @property
    def frames_written(self) -> int:
        return self.c.frames_written


class LS:
    """A caller-owned least-squares state: fp32 [2D][2D] gram plus the C struct."""

    def __init__(self, dim: int, device="cuda"):
        self.gram = torch.zeros(ispa_ls_state_bytes(dim) // 4, dtype=torch.float32, device=device)
        self.c = LSState(dim, 0, 0, self.gram.data_ptr())

    def blocks(self):
        D = self.c.dim
        g = self.gram.view(2 * D, 2 * D).double().cpu().numpy()
        return g[:D, :D], g[:D, D:], g[D:, D:]


def window(n_sink: int, n_recent: int) -> Window:
    return Window(n_sink, n_recent)
