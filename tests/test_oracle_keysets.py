"""Pins for oracle.keysets: Eq. 7-8 set algebra, ring slots, Tables 1-2 accounting."""
import os

import pytest

from oracle import keysets as ks

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "kvcache_tables.txt")


def _golden_rows():
    rows = []
    with open(GOLDEN) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            t, model, n, x, pct, ff, lf = line.split()
            rows.append((t, model, int(n), float(x), float(pct), int(ff), int(lf)))
    return rows


@pytest.mark.parametrize("row", _golden_rows(), ids=lambda r: f"{r[0]}-{r[1]}-{r[3]}")
def test_kv_cache_fraction_matches_tables(row):
    # Tables 1-2: KVCache column, printed to 0.1 %.
    _, _, n_layers, x, pct, f_frames, l_frames = row
    K = round(x * n_layers)
    assert abs(K - x * n_layers) < 1e-9          # K = x N is an integer for these models
    frac = ks.kv_cache_fraction(n_layers, K, f_frames, l_frames)
    assert abs(100.0 * frac - pct) <= 0.05 + 1e-9


def test_kv_cache_fraction_limits():
    assert ks.kv_cache_fraction(30, 0, 12, 1) == 1.0
    assert abs(ks.kv_cache_fraction(30, 30, 12, 1) - 1.0 / 12) < 1e-15


@pytest.mark.parametrize("F", [0, 1, 2, 5, 18, 24])
@pytest.mark.parametrize("n_sink,n_recent", [(0, 0), (0, 2), (0, 6), (1, 0), (1, 6), (2, 3), (0, 40)])
def test_local_hist_disjoint_union(F, n_sink, n_recent):
    # Eq. 8: the full past is the disjoint union of local and history frames.
    loc = ks.local_past_frames(F, n_sink, n_recent)
    hist = ks.hist_past_frames(F, n_sink, n_recent)
    assert set(loc).isdisjoint(hist)
    assert sorted(loc + hist) == list(range(F))
    # Eq. 7 membership, restated frame by frame
    for f in range(F):
        assert (f in loc) == (f < n_sink or f >= F - n_recent)


def test_paper_literal_local_set():
    # Eq. 7 with one sink frame and no recent past frame: local = {K_1} (+ chunk);
    # history = {K_2 .. K_{t-1}}.
    assert ks.local_past_frames(6, 1, 0) == [0]
    assert ks.hist_past_frames(6, 1, 0) == [1, 2, 3, 4, 5]


def _simulate_ring(n_frames_total, capacity, n_pinned):
    """Brute-force ring: a list of slots overwritten in arrival order."""
    slots = [None] * capacity
    order = []                         # non-pinned slots in the order they were last filled
    for f in range(n_frames_total):
        if f < n_pinned:
            slots[f] = f
            continue
        free = [s for s in range(n_pinned, capacity) if slots[s] is None]
        if free:
            s = free[0]
        else:
            s = order.pop(0)           # evict the oldest non-sink frame
        slots[s] = f
        order.append(s)
    return slots


@pytest.mark.parametrize("capacity,n_pinned", [(1, 0), (4, 0), (7, 1), (24, 0), (9, 2)])
def test_ring_slot_matches_brute_force(capacity, n_pinned):
    for total in range(0, 3 * capacity + 5):
        slots = _simulate_ring(total, capacity, n_pinned)
        resident = ks.resident_frames(total, capacity, n_pinned)
        assert sorted(f for f in slots if f is not None) == resident
        for f in resident:
            assert slots[ks.ring_slot(f, capacity, n_pinned)] == f


def test_full_set_is_one_slot_run():
    for capacity in (3, 8, 24):
        for total in range(1, 3 * capacity):
            runs = ks.slot_ranges(ks.resident_frames(total, capacity, 0), capacity, 0)
            assert runs == [(0, min(total, capacity))]


def test_slot_ranges_wrap():
    # capacity 8, 11 frames written: frames 3..10 resident, slots of 9, 10 are 1, 2
    frames = [9, 10]
    assert ks.slot_ranges(frames, 8, 0) == [(1, 2)]
    frames = [7, 8]                    # slots 7 and 0: wrap splits the run
    assert ks.slot_ranges(frames, 8, 0) == [(0, 1), (7, 1)]


def test_ring_bytes():
    # config "1.3B": 12 heads x 128 x 1560 tokens, 18 frames, K and V, bf16
    assert ks.ring_bytes(12, 128, 1560, 18) == 2 * 12 * 18 * 1560 * 128 * 2


def test_select_layers_ascending_with_ties_and_nan():
    # Sec. 3.3: the k layers with the lowest eps become L-layers.
    eps = [3.0, 1.0, float("nan"), 1.0, 0.5, 7.0]
    assert ks.select_layers(eps, 0) == [0, 0, 0, 0, 0, 0]
    assert ks.select_layers(eps, 1) == [0, 0, 0, 0, 1, 0]
    assert ks.select_layers(eps, 2) == [0, 1, 0, 0, 1, 0]      # tie 1.0: lower index first
    assert ks.select_layers(eps, 3) == [0, 1, 0, 1, 1, 0]
    assert ks.select_layers(eps, 6) == [1, 1, 1, 1, 1, 1]
    assert ks.select_layers(eps, 5) == [1, 1, 0, 1, 1, 1]      # NaN last


def test_select_layers_matches_sort_brute_force():
    import random
    rnd = random.Random(3)
    for _ in range(50):
        n = rnd.randint(1, 12)
        eps = [rnd.choice([0.0, 1.0, 2.0, rnd.random()]) for _ in range(n)]
        k = rnd.randint(0, n)
        want = sorted(range(n), key=lambda i: (eps[i], i))[:k]
        got = ks.select_layers(eps, k)
        assert [i for i in range(n) if got[i]] == sorted(want)
