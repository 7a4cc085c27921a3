"""The interval arithmetic of paper_2607_00712_gb300.trace (the per-tile role timeline printed from
ispa_debug_set_trace events) on a synthetic, strictly periodic event array: every reported median
must equal the offset it was built with (no GPU)."""
import numpy as np

from paper_2607_00712_gb300.trace import SLOTS, summarise

PERIOD = 2600
# per-tile event offsets from "S_j seen by softmax warp 0" (slot 0)
OFF = {8: 600, 9: 800, 1: 1050, 10: 2100, 2: 2150, 3: 2400, 11: 2480, 4: 3200, 5: 3900}


def _trace(n=40):
    t = np.zeros((n, SLOTS), dtype=np.int64)
    for j in range(n):
        base = 10_000 + PERIOD * j
        t[j, 0] = base
        for slot, off in OFF.items():
            t[j, slot] = base + off
        if j >= 1:
            t[j, 15] = base - 2 * PERIOD + 3300            # K_j landed, seen by the UMMA thread
        for w in range(8):
            t[j, 16 + w] = base + 2150 + 3 * w              # P_j arrivals of the 8 softmax warps
            t[j, 24 + w] = base + 5 * w                     # S_j seen by the 8 softmax warps
    # first CTA: entry, TMEM allocated, Q landed; epilogue stored after the last tile
    t[0, 12], t[0, 13], t[0, 14] = 1000, 2400, 4600
    t[0, 15] = 10_000 + PERIOD * (n - 1) + 2400 + 5000
    return t


def test_summarise_recovers_the_planted_intervals():
    r = summarise(_trace())
    assert r["period (UMMA thread sees P_j -> sees P_j+1)"] == PERIOD
    assert r["UMMA: sees P_j -> sees V_j"] == 80
    assert r["UMMA: sees V_j -> PV_j issued (12 UMMAs)"] == 720
    assert r["UMMA: PV_j issued -> K_j+2 landed"] == 100
    assert r["UMMA: K_j+2 landed -> S_j+2 issued (8 UMMAs)"] == 600
    assert r["UMMA: S_j+2 issued -> sees P_j+1"] == PERIOD + 2400 - 3900
    assert r["softmax w0: S_j seen -> loaded"] == 600
    assert r["softmax w0: loaded -> tile max"] == 200
    assert r["softmax w0: tile max -> rescale decided (pair barrier)"] == 250
    assert r["softmax w0: rescale decided -> exp loop done"] == 1050
    assert r["softmax w0: exp loop done -> P_j arrived"] == 50
    assert r["softmax w0: S_j seen -> P_j arrived"] == 2150
    assert r["softmax w0: P_j arrived -> S_j+1 seen (waiting for S)"] == PERIOD - 2150
    assert r["softmax w0: P_j arrived -> S_j+2 seen (UMMA chain)"] == 2 * PERIOD - 2150
    assert r["spread of S_j seen over the 8 softmax warps"] == 35
    assert r["last softmax warp's P_j arrival -> UMMA sees P_j (two clocks)"] == 2400 - 2150 - 21
    assert r["tiles traced"] == 40
    assert r["CTA: entry -> TMEM allocated"] == 1400
    assert r["CTA: TMEM allocated -> Q landed"] == 2200
    assert r["CTA: last P seen -> epilogue stored"] == 5000


def test_short_traces_report_only_traced_tiles():
    # 6 tiles: the one middle tile j = 3 has j + 2 = 5 traced, so every row is a real interval
    r = summarise(_trace(6))
    assert r["period (UMMA thread sees P_j -> sees P_j+1)"] == PERIOD
    assert r["softmax w0: P_j arrived -> S_j+2 seen (UMMA chain)"] == 2 * PERIOD - 2150
    assert r["tiles traced"] == 6
    # 4 tiles: no middle tile with two traced successors, so no interval row is printed
    r = summarise(_trace(4))
    assert "period (UMMA thread sees P_j -> sees P_j+1)" not in r and r["tiles traced"] == 4
