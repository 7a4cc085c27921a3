"""Per-key-tile role timeline of the attention kernel (a debug aid; not on the hot path).

    python -m paper_2607_00712_gb300.trace [--model 1.3b|14b] [--mode full|local|dual] [--frames F]

Builds one synthetic chunk step at the model's attention shape (head_dim 128, 1560 tokens per
frame, a 3-frame chunk, a ring of F past frames, a 6-frame window), runs the chosen attention
call a few times, then once with ispa_debug_set_trace switched on, and prints for the first
CTA the median over its middle key tiles of the intervals between the events the kernel
records (see ispa_debug_set_trace in include/ispa.h).  Values are SM clock cycles.
"""
from __future__ import annotations

import argparse
import statistics

import torch

from . import abi
from .build import build_library
from .device import Ring, Window

HEADS = {"1.3b": 12, "14b": 40}
P, D_HEAD, CHUNK, WINDOW = 1560, 128, 3, 6
SLOTS = 32


def _qkv(g, n_tok, H):
    """q, k, v [n_tok, H, 128] bf16: N(0, 1) entries, keys shifted per (frame, head) by an
    N(0, 0.5^2) offset vector, as in the synthetic workloads of the tests and the bench."""
    n_fr = n_tok // P
    q = torch.randn(n_tok, H, D_HEAD, device="cuda", generator=g)
    k = torch.randn(n_fr, P, H, D_HEAD, device="cuda", generator=g)
    k += 0.5 * torch.randn(n_fr, 1, H, D_HEAD, device="cuda", generator=g)
    v = torch.randn(n_tok, H, D_HEAD, device="cuda", generator=g)
    return [x.reshape(n_tok, H, D_HEAD).to(torch.bfloat16) for x in (q, k, v)]


def run(model: str = "1.3b", mode: str = "full", frames: int = 18, warmup: int = 5) -> dict:
    build_library()
    H = HEADS[model]
    nq, D = CHUNK * P, H * D_HEAD
    g = torch.Generator(device="cuda")
    g.manual_seed(5)
    ring = Ring(H, D_HEAD, P, frames if mode != "local" else WINDOW, 0)
    for _ in range(0, ring.c.capacity_frames, CHUNK):
        _, k, v = _qkv(g, CHUNK * P, H)
        abi.ispa_kv_append(ring.c, k, v, CHUNK)
    q, kc, vc = _qkv(g, nq, H)
    win = Window(0, WINDOW)
    out = torch.empty(nq, D, dtype=torch.bfloat16, device="cuda")
    out2 = torch.empty_like(out)
    disc = torch.empty(nq, dtype=torch.float32, device="cuda")
    dsum = torch.zeros(1, dtype=torch.float32, device="cuda")
    wsb = abi.ispa_attn_dual_workspace_size(H, nq)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")

    def call():
        if mode == "full":
            abi.ispa_attn_full(ring.c, q, kc, vc, nq, 0.0, out)
        elif mode == "local":
            abi.ispa_attn_local(ring.c, win, q, kc, vc, nq, 0.0, out)
        else:
            abi.ispa_attn_dual(ring.c, win, q, kc, vc, nq, 0.0, out, out2, disc, dsum, None, None, ws, wsb)

    for _ in range(warmup):
        call()
    torch.cuda.synchronize()
    n_tiles = 1024
    buf = torch.zeros(n_tiles * SLOTS, dtype=torch.int64, device="cuda")
    abi.ispa_debug_set_trace(buf, n_tiles)
    try:
        call()
        torch.cuda.synchronize()
    finally:
        abi.ispa_debug_set_trace(None, 0)
    return summarise(buf.view(n_tiles, SLOTS).cpu().numpy().astype("int64"))


def summarise(t) -> dict:
    """Medians of the per-tile intervals over the middle tiles, and the first CTA's fill and
    drain, from the event array t[tile, slot] (clock64 values; 0 where nothing was recorded)."""
    n = int((t[:, 3] != 0).sum())
    J = list(range(10, n - 10)) if n > 30 else list(range(3, max(n - 4, 4)))
    J = [j for j in J if j + 2 < n]   # every row reads tiles j .. j + 2: traced tiles only

    last_arrive = lambda j: max(t[j, 16 + w] for w in range(8))  # noqa: E731
    rows = {
        "period (UMMA thread sees P_j -> sees P_j+1)": lambda j: t[j + 1, 3] - t[j, 3],
        "UMMA: sees P_j -> sees V_j": lambda j: t[j, 11] - t[j, 3],
        "UMMA: sees V_j -> PV_j issued (12 UMMAs)": lambda j: t[j, 4] - t[j, 11],
        "UMMA: PV_j issued -> K_j+2 landed": lambda j: t[j + 2, 15] - t[j, 4],
        "UMMA: K_j+2 landed -> S_j+2 issued (8 UMMAs)": lambda j: t[j, 5] - t[j + 2, 15],
        "UMMA: S_j+2 issued -> sees P_j+1": lambda j: t[j + 1, 3] - t[j, 5],
        "S_j+2 issued -> softmax warp 0 sees it (clocks of two sub-partitions)": lambda j: t[j + 2, 0] - t[j, 5],
        "softmax w0: S_j seen -> loaded": lambda j: t[j, 8] - t[j, 0],
        "softmax w0: loaded -> tile max": lambda j: t[j, 9] - t[j, 8],
        "softmax w0: tile max -> rescale decided (pair barrier)": lambda j: t[j, 1] - t[j, 9],
        "softmax w0: rescale decided -> exp loop done": lambda j: t[j, 10] - t[j, 1],
        "softmax w0: exp loop done -> P_j arrived": lambda j: t[j, 2] - t[j, 10],
        "softmax w0: S_j seen -> P_j arrived": lambda j: t[j, 2] - t[j, 0],
        "softmax w0: P_j arrived -> S_j+1 seen (waiting for S)": lambda j: t[j + 1, 0] - t[j, 2],
        # one clock: the chain PV_j -> S_j+2 with both hand-offs; the period is about half of this
        # plus half of the softmax's own time per tile
        "softmax w0: P_j arrived -> S_j+2 seen (UMMA chain)": lambda j: t[j + 2, 0] - t[j, 2],
        "spread of S_j seen over the 8 softmax warps": lambda j: max(t[j, 24 + w] for w in range(8)) - min(
            t[j, 24 + w] for w in range(8)),
        "last softmax warp's P_j arrival -> UMMA sees P_j (two clocks)": lambda j: t[j, 3] - last_arrive(j),
    }
    # too few traced tiles for a steady-state middle: no interval rows at all
    res = {k: int(statistics.median(f(j) for j in J)) for k, f in rows.items()} if J else {}
    res["tiles traced"] = n
    if n == 0:
        return res
    # fill and drain of the first CTA (one sample each)
    res["CTA: entry -> TMEM allocated"] = int(t[0, 13] - t[0, 12])
    res["CTA: TMEM allocated -> Q landed"] = int(t[0, 14] - t[0, 13])
    res["CTA: Q landed -> S_0 seen by softmax warp 0"] = int(t[0, 0] - t[0, 14])
    res["CTA: entry -> P_0 seen (first PV can start)"] = int(t[0, 3] - t[0, 12])
    res["CTA: entry -> last P seen"] = int(t[n - 1, 3] - t[0, 12])
    res["CTA: last P seen -> epilogue stored"] = int(t[0, 15] - t[n - 1, 3])
    res["CTA: entry -> epilogue stored"] = int(t[0, 15] - t[0, 12])
    return res


def main() -> None:
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--model", choices=sorted(HEADS), default="1.3b")
    ap.add_argument("--mode", choices=["full", "local", "dual"], default="full")
    ap.add_argument("--frames", type=int, default=18, help="past frames in the ring (full / dual)")
    a = ap.parse_args()
    for k, v in run(a.model, a.mode, a.frames).items():
        print(f"{k:56s} {v:8d}")


if __name__ == "__main__":
    main()
