"""libispa on the host (no GPU): symbols, struct layouts, ring bookkeeping, validation.

Ring slots and key-set runs must equal the oracle's exactly (integer work).
"""
import ctypes
import os
import re
import subprocess
import tempfile

import pytest

from oracle import keysets as ks
from paper_2607_00712_gb300 import abi
from paper_2607_00712_gb300._lib import KeySets, KVRing, LSState, SlotRange, Window

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "ispa.h")


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2607_00712_gb300.build import build_library
    build_library()


def _declared():
    txt = open(HEADER).read()
    return re.findall(r"ISPA_API\s+[\w\s\*]+?\b(ispa_\w+)\s*\(", txt)


def test_every_declared_symbol_is_exported():
    names = _declared()
    assert len(names) >= 19
    L = abi.lib()
    for n in names:
        assert hasattr(L, n), n
    # and the binding declares a signature for every one of them
    assert set(names) == set(abi._SIGS)


def test_struct_layout_matches_header():
    # Compile a tiny C program against the header and compare sizeof/offsetof with ctypes.
    prog = r"""
#include <stdio.h>
#include <stddef.h>
#include "ispa.h"
int main(void) {
  printf("%zu %zu %zu %zu %zu\n", sizeof(ispa_kv_ring), sizeof(ispa_window), sizeof(ispa_slot_range),
         sizeof(ispa_key_sets), sizeof(ispa_ls_state));
  printf("%zu %zu %zu %zu\n", offsetof(ispa_kv_ring, frames_written), offsetof(ispa_kv_ring, k),
         offsetof(ispa_kv_ring, v), offsetof(ispa_key_sets, hist));
  printf("%zu %zu\n", offsetof(ispa_ls_state, n_tokens), offsetof(ispa_ls_state, gram));
  return 0;
}
"""
    with tempfile.TemporaryDirectory() as d:
        src = os.path.join(d, "t.c")
        exe = os.path.join(d, "t")
        open(src, "w").write(prog)
        subprocess.run(["gcc", "-I", os.path.dirname(HEADER), src, "-o", exe], check=True)
        out = subprocess.run([exe], capture_output=True, text=True, check=True).stdout.split()
    got = list(map(int, out))
    want = [ctypes.sizeof(KVRing), ctypes.sizeof(Window), ctypes.sizeof(SlotRange), ctypes.sizeof(KeySets),
            ctypes.sizeof(LSState), KVRing.frames_written.offset, KVRing.k.offset, KVRing.v.offset,
            KeySets.hist.offset, LSState.n_tokens.offset, LSState.gram.offset]
    assert got == want


def test_status_strings():
    assert abi.status_string(0) == "ok"
    assert abi.status_string(abi.ISPA_ERR_NOT_SPD) == "matrix not positive definite"
    assert abi.status_string(99) == "unknown status"


def _ring(cap, n_sink, F, H=2, d=64, P=16):
    return KVRing(H, d, P, cap, n_sink, 0, F, 0, 0)


@pytest.mark.parametrize("cap,n_sink", [(1, 0), (4, 0), (6, 1), (9, 2), (24, 0)])
def test_ring_slot_matches_oracle(cap, n_sink):
    for F in range(0, 3 * cap + 4):
        r = _ring(cap, n_sink, F)
        resident = set(ks.resident_frames(F, cap, n_sink))
        for f in range(F + 2):
            got = abi.ispa_ring_slot(r, f)
            want = ks.ring_slot(f, cap, n_sink) if f in resident else -1
            assert got == want, (cap, n_sink, F, f)


@pytest.mark.parametrize("cap,n_sink", [(4, 0), (6, 1), (9, 2), (12, 0), (24, 1)])
@pytest.mark.parametrize("w_sink,w_recent", [(0, 0), (0, 2), (1, 0), (1, 3), (2, 2), (0, 6)])
def test_window_resolve_matches_oracle(cap, n_sink, w_sink, w_recent):
    for F in range(0, 3 * cap + 3):
        r = _ring(cap, n_sink, F)
        resident = ks.resident_frames(F, cap, n_sink)
        loc = ks.local_past_frames(F, w_sink, w_recent)
        if not set(loc) <= set(resident):
            with pytest.raises(abi.IspaError) as e:
                abi.ispa_window_resolve(r, Window(w_sink, w_recent))
            assert e.value.status == abi.ISPA_ERR_CAPACITY
            continue
        got = abi.ispa_window_resolve(r, Window(w_sink, w_recent))
        hist = [f for f in resident if f not in set(loc)]
        assert got.ranges("full") == ks.slot_ranges(resident, cap, n_sink)
        assert got.ranges("local") == ks.slot_ranges(loc, cap, n_sink)
        assert got.ranges("hist") == ks.slot_ranges(hist, cap, n_sink)


def test_ring_bytes_matches_oracle():
    r = KVRing(12, 128, 1560, 18, 0, 0, 0, 0, 0)
    assert abi.ispa_ring_bytes(r) == ks.ring_bytes(12, 128, 1560, 18)


def test_validation_errors_without_gpu():
    L = abi.lib()
    # null ring
    assert L.ispa_attn_full(None, 16, 16, 16, 128, 0.0, 16, None, None) == abi.ISPA_ERR_INVALID_ARG
    # unsupported head_dim
    r = KVRing(2, 96, 16, 4, 0, 0, 0, 16, 16)
    assert L.ispa_attn_full(ctypes.byref(r), 16, 16, 16, 128, 0.0, 16, None, None) == abi.ISPA_ERR_UNSUPPORTED
    # misaligned pointer
    r = KVRing(2, 64, 16, 4, 0, 0, 0, 16, 16)
    assert L.ispa_attn_full(ctypes.byref(r), 18, 16, 16, 128, 0.0, 16, None, None) == abi.ISPA_ERR_INVALID_ARG
    # window needs an evicted frame
    r = KVRing(2, 64, 16, 4, 0, 0, 10, 16, 16)
    assert L.ispa_attn_local(ctypes.byref(r), Window(1, 0), 16, 16, 16, 128, 0.0, 16, None,
                             None) == abi.ISPA_ERR_CAPACITY
    # append larger than the non-sink capacity
    r = KVRing(2, 64, 16, 4, 1, 0, 0, 16, 16)
    assert L.ispa_kv_append(ctypes.byref(r), 16, 16, 4, None) == abi.ISPA_ERR_CAPACITY
    assert r.frames_written == 0
    # dual without workspace
    r = KVRing(2, 64, 16, 4, 0, 0, 2, 16, 16)
    assert L.ispa_attn_dual(ctypes.byref(r), Window(0, 1), 16, 16, 16, 128, 0.0, 16, 16, 16, 16, None, None,
                            None, 0, None) == abi.ISPA_ERR_WORKSPACE
    # ls: dim not a multiple of 128
    st = LSState(100, 0, 0, 16)
    assert L.ispa_ls_accumulate(ctypes.byref(st), 16, 16, 10, 16, 1 << 30, None) == abi.ISPA_ERR_UNSUPPORTED
    st = LSState(128, 0, 0, 16)
    assert L.ispa_ls_accumulate(ctypes.byref(st), 16, 16, 10, None, 0, None) == abi.ISPA_ERR_WORKSPACE
    assert L.ispa_ls_solve(ctypes.byref(st), 16, 128, -1.0, 16, None, 16, 1 << 30, None) == abi.ISPA_ERR_INVALID_ARG


def test_attention_option_validation_without_gpu():
    L = abi.lib()
    r = KVRing(2, 64, 16, 4, 0, 0, 2, 16, 16)
    # unknown option bit
    assert L.ispa_attn_full_ex(ctypes.byref(r), 16, 16, 16, 32, 0.0, 2, 16, None, None) == abi.ISPA_ERR_INVALID_ARG
    # frame-causal needs whole chunk frames (n_q a multiple of tokens_per_frame = 16)
    assert L.ispa_attn_full_ex(ctypes.byref(r), 16, 16, 16, 24, 0.0, abi.ISPA_ATTN_FRAME_CAUSAL, 16, None,
                               None) == abi.ISPA_ERR_INVALID_ARG
    assert L.ispa_attn_local_ex(ctypes.byref(r), Window(0, 1), 16, 16, 16, 24, 0.0, abi.ISPA_ATTN_FRAME_CAUSAL,
                                16, None, None) == abi.ISPA_ERR_INVALID_ARG
    assert L.ispa_attn_dual_ex(ctypes.byref(r), Window(0, 1), 16, 16, 16, 32, 0.0, 4, 16, 16, 16, 16, None, None,
                               16, 1 << 20, None) == abi.ISPA_ERR_INVALID_ARG


def test_ls_accumulate_option_validation_without_gpu():
    L = abi.lib()
    st = LSState(128, 0, 0, 16)
    # an unknown option bit
    assert L.ispa_ls_accumulate_ex(ctypes.byref(st), 16, 16, 10, 2, 16, 1 << 30, None) == abi.ISPA_ERR_INVALID_ARG
    # the exact form still needs its workspace; dim not a multiple of 128 is unsupported in both
    assert L.ispa_ls_accumulate_ex(ctypes.byref(st), 16, 16, 10, abi.ISPA_LS_EXACT_DELTA, None, 0,
                                   None) == abi.ISPA_ERR_WORKSPACE
    st = LSState(100, 0, 0, 16)
    assert L.ispa_ls_accumulate_ex(ctypes.byref(st), 16, 16, 10, abi.ISPA_LS_EXACT_DELTA, 16, 1 << 30,
                                   None) == abi.ISPA_ERR_UNSUPPORTED
    assert st.n_tokens == 0


def test_w8a8_validation_without_gpu():
    L = abi.lib()
    assert L.ispa_linear_w8a8(16, 16, 16, 16, 100, 192, 256, 16, None) == abi.ISPA_ERR_UNSUPPORTED   # D % 128
    assert L.ispa_linear_w8a8(16, 16, 16, 16, 100, 256, 192, 16, None) == abi.ISPA_ERR_UNSUPPORTED   # D_out % 128
    assert L.ispa_linear_w8a8(16, 16, 16, 16, 0, 256, 256, 16, None) == abi.ISPA_ERR_INVALID_ARG
    assert L.ispa_linear_w8a8(16, 16, 16, 20, 10, 256, 256, 16, None) == abi.ISPA_ERR_INVALID_ARG   # w_scale
    assert L.ispa_linear_w8a8(24, 16, 16, 16, 10, 256, 256, 16, None) == abi.ISPA_ERR_INVALID_ARG    # misaligned
    assert L.ispa_quantize_rows_e4m3(16, 10, 24, 16, 16, None) == abi.ISPA_ERR_UNSUPPORTED           # cols % 16
    assert L.ispa_quantize_rows_e4m3(None, 10, 32, 16, 16, None) == abi.ISPA_ERR_INVALID_ARG
    assert L.ispa_quantize_weight_e4m3(16, None, 24, 32, 16, 16, None) == abi.ISPA_ERR_UNSUPPORTED   # D % 16
    assert L.ispa_quantize_weight_e4m3(16, None, 32, 0, 16, 16, None) == abi.ISPA_ERR_INVALID_ARG


def test_workspace_sizes():
    assert abi.ispa_attn_dual_workspace_size(12, 4680) == 12 * 4680 * 4
    assert abi.ispa_ls_state_bytes(1536) == 4 * 1536 * 1536 * 4
    assert abi.ispa_ls_accumulate_workspace_size(1536, 4680) >= 2 * 4680 * 1536 * 2
    assert abi.ispa_ls_solve_workspace_size(1536, 1536) >= 3 * 1536 * 1536 * 8


def test_select_layers_matches_oracle():
    import random
    rnd = random.Random(5)
    for _ in range(40):
        n = rnd.randint(1, 40)
        eps = [rnd.choice([0.25, 1.0, rnd.random(), float("nan")]) for _ in range(n)]
        k = rnd.randint(0, n)
        assert abi.ispa_select_layers(eps, k) == ks.select_layers(eps, k)
    with pytest.raises(abi.IspaError):
        abi.ispa_select_layers([1.0, 2.0], 3)


def test_ring_compact_validation_without_gpu():
    L = abi.lib()
    src = KVRing(2, 64, 16, 10, 0, 0, 13, 16, 16)
    dst = KVRing(2, 64, 16, 5, 1, 0, 0, 16, 16)          # wrong capacity for window (1, 3)
    assert L.ispa_ring_compact(ctypes.byref(src), Window(1, 3), ctypes.byref(dst), None) == abi.ISPA_ERR_INVALID_ARG
    dst = KVRing(2, 64, 16, 4, 1, 0, 0, 16, 16)
    # frame 0 (the sink) was evicted from src (no pinned sink there): the window cannot be kept
    assert L.ispa_ring_compact(ctypes.byref(src), Window(1, 3), ctypes.byref(dst), None) == abi.ISPA_ERR_CAPACITY
    assert dst.frames_written == 0


def test_empty_calls_are_argument_errors_without_gpu():
    # every count must be >= 1; an empty call is rejected before anything is enqueued
    L = abi.lib()
    r = KVRing(2, 64, 16, 4, 0, 0, 2, 16, 16)
    assert L.ispa_attn_full(ctypes.byref(r), 16, 16, 16, 0, 0.0, 16, None, None) == abi.ISPA_ERR_INVALID_ARG
    assert L.ispa_attn_local(ctypes.byref(r), Window(0, 1), 16, 16, 16, 0, 0.0, 16, None,
                             None) == abi.ISPA_ERR_INVALID_ARG
    assert L.ispa_attn_dual(ctypes.byref(r), Window(0, 1), 16, 16, 16, 0, 0.0, 16, 16, 16, 16, None, None,
                            16, 1 << 20, None) == abi.ISPA_ERR_INVALID_ARG
    assert L.ispa_kv_append(ctypes.byref(r), 16, 16, 0, None) == abi.ISPA_ERR_INVALID_ARG
    assert r.frames_written == 2
    st = LSState(128, 0, 0, 16)
    assert L.ispa_ls_accumulate(ctypes.byref(st), 16, 16, 0, 16, 1 << 30, None) == abi.ISPA_ERR_INVALID_ARG
    assert st.n_tokens == 0
    assert L.ispa_quantize_rows_e4m3(16, 0, 128, 16, 16, None) == abi.ISPA_ERR_INVALID_ARG
    assert L.ispa_linear_w8a8(16, 16, 16, 16, 0, 128, 128, 16, None) == abi.ISPA_ERR_INVALID_ARG
    assert L.ispa_discrepancy(16, 16, 0, 128, 16, 16, None) == abi.ISPA_ERR_INVALID_ARG
    assert L.ispa_discrepancy(16, 16, 4, 0, 16, 16, None) == abi.ISPA_ERR_INVALID_ARG
    assert L.ispa_discrepancy(16, 24, 4, 128, 16, 16, None) == abi.ISPA_ERR_INVALID_ARG   # misaligned row
    assert L.ispa_discrepancy(16, 16, 4, 100, 16, 16, None) == abi.ISPA_ERR_UNSUPPORTED


def test_append_of_more_than_sixteen_frames_is_rejected_without_gpu():
    L = abi.lib()
    r = KVRing(2, 64, 16, 40, 0, 0, 0, 16, 16)
    assert L.ispa_kv_append(ctypes.byref(r), 16, 16, 17, None) == abi.ISPA_ERR_CAPACITY
    assert r.frames_written == 0
