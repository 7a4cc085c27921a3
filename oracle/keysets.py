"""Key sets, ring slots and cache accounting (oracle; test infrastructure only).

Paper basis
  * Eq. 3 (Sec. 2, KV injection): the chunk's queries attend to
    K = [K_past ; K_cur], V = [V_past ; V_cur].
  * Eq. 7-8 (Sec. 3.4): the local set is the sink frame plus the current
    frames, the history set is everything in between; the full set is their
    disjoint union.  The window is parameterised as (n_sink, n_recent): the
    n_sink oldest past frames plus the n_recent newest past frames are local.
  * Sec. 3.1 phase 3 / Sec. 3.3: an L-layer permanently evicts its history and
    keeps only the local context.
  * Tables 1-2 "KVCache": fraction of KV memory kept when K = x*N layers are
    L-layers.

Frames are numbered logically 0, 1, 2, ... in generation order.  A step with F
past frames has past frames 0..F-1; the chunk is not part of the cache.
"""
from __future__ import annotations

import math


def local_past_frames(F: int, n_sink: int, n_recent: int) -> list[int]:
    """Past frames in the local set: {f < n_sink} united with {F-n_recent <= f < F}."""
    sink = set(range(min(n_sink, F)))
    recent = set(range(max(0, F - n_recent), F))
    return sorted(sink | recent)


def hist_past_frames(F: int, n_sink: int, n_recent: int) -> list[int]:
    """Past frames in the history set: the full past minus the local past (Eq. 8)."""
    loc = set(local_past_frames(F, n_sink, n_recent))
    return [f for f in range(F) if f not in loc]


def ring_slot(f: int, capacity: int, n_pinned: int) -> int:
    """Ring slot holding logical frame f.

    The first n_pinned frames (sink frames) keep slots 0..n_pinned-1 for
    good; every later frame f goes to slot n_pinned + (f - n_pinned) mod
    (capacity - n_pinned), i.e. it overwrites the oldest non-sink frame.
    """
    if f < n_pinned:
        return f
    return n_pinned + (f - n_pinned) % (capacity - n_pinned)


def resident_frames(frames_written: int, capacity: int, n_pinned: int) -> list[int]:
    """Logical frames still stored in a ring after frames_written appends."""
    out = []
    for f in range(frames_written):
        if f < n_pinned or frames_written - f <= capacity - n_pinned:
            out.append(f)
    return out


def slot_ranges(frames: list[int], capacity: int, n_pinned: int) -> list[tuple[int, int]]:
    """Collapse the slots of the given frames into maximal contiguous runs.

    Returns (first_slot, n_slots) pairs in increasing slot order.
    """
    slots = sorted(ring_slot(f, capacity, n_pinned) for f in frames)
    runs: list[tuple[int, int]] = []
    for s in slots:
        if runs and runs[-1][0] + runs[-1][1] == s:
            runs[-1] = (runs[-1][0], runs[-1][1] + 1)
        else:
            runs.append((s, 1))
    return runs


def select_layers(eps, k: int) -> list[int]:
    """Sec. 3.3: rank layers by ascending feasibility score and pick the k lowest as L-layers.

    Returns a 0/1 list (1 = L-layer).  Ties keep the lower layer index first (the paper
    gives only "ascending order"); a NaN score ranks after every number.
    """
    n = len(eps)
    key = [(1 if math.isnan(e) else 0, 0.0 if math.isnan(e) else e, i) for i, e in enumerate(eps)]
    chosen = [i for _, _, i in sorted(key)[:k]]
    return [1 if i in chosen else 0 for i in range(n)]


def ring_bytes(num_heads: int, head_dim: int, tokens_per_frame: int,
               capacity_frames: int, elem_bytes: int = 2) -> int:
    """Bytes of one layer's K and V rings together."""
    return 2 * num_heads * capacity_frames * tokens_per_frame * head_dim * elem_bytes


def kv_cache_fraction(n_layers: int, n_l_layers: int, f_layer_frames: int,
                      l_layer_frames: int) -> float:
    """Fraction of KV-cache bytes kept when n_l_layers layers are L-layers.

    F-layers keep f_layer_frames frames, L-layers keep l_layer_frames frames
    (Sec. 3.3: L-layers evict their history).  All layers have the same head
    shape, so per-layer bytes are proportional to the frames kept.
    """
    per_frame = ring_bytes(1, 1, 1, 1)
    full = n_layers * f_layer_frames * per_frame
    kept = ((n_layers - n_l_layers) * f_layer_frames + n_l_layers * l_layer_frames) * per_frame
    return kept / full
