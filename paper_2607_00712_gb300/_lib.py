"""ctypes binding of libispa (include/ispa.h).  Argument marshalling only.

Every function here has the name of the C entry point it calls and passes its
arguments straight through: tensors become device pointers (``data_ptr()``),
streams become ``cudaStream_t`` handles, and a non-OK status raises
``IspaError``.  No computation happens in Python.  If libispa.so is missing
the import of the library fails loudly; there is no fallback path.
"""
from __future__ import annotations

import ctypes
import os
from ctypes import (POINTER, Structure, c_char_p, c_double, c_float, c_int32, c_int64, c_size_t, c_uint32, c_uint64,
                    c_void_p)

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libispa.so")

ISPA_OK = 0
ISPA_ERR_INVALID_ARG = 1
ISPA_ERR_UNSUPPORTED = 2
ISPA_ERR_CAPACITY = 3
ISPA_ERR_NOT_SPD = 4
ISPA_ERR_TIMEOUT = 5
ISPA_ERR_CUDA = 6
ISPA_ERR_WORKSPACE = 7
ISPA_ATTN_FRAME_CAUSAL = 1   # option bit of the *_ex attention entry points
ISPA_LS_EXACT_DELTA = 1      # option bit of ispa_ls_accumulate_ex
ISPA_KV_BF16 = 0             # ring k_format values
ISPA_KV_K_E4M3 = 1
ISPA_KV_KV_E4M3 = 2
MAX_RANGES = 4


class KVRing(Structure):
    _fields_ = [("num_heads", c_int32), ("head_dim", c_int32), ("tokens_per_frame", c_int32),
                ("capacity_frames", c_int32), ("n_sink_frames", c_int32), ("k_format", c_int32),
                ("frames_written", c_int64), ("k", c_void_p), ("v", c_void_p)]


class Window(Structure):
    _fields_ = [("n_sink_frames", c_int32), ("n_recent_frames", c_int32)]


class SlotRange(Structure):
    _fields_ = [("first_slot", c_int32), ("n_slots", c_int32)]


class KeySets(Structure):
    _fields_ = [("n_full", c_int32), ("n_local", c_int32), ("n_hist", c_int32), ("reserved", c_int32),
                ("full", SlotRange * MAX_RANGES), ("local", SlotRange * MAX_RANGES),
                ("hist", SlotRange * MAX_RANGES)]

    def ranges(self, which: str) -> list[tuple[int, int]]:
        n = getattr(self, "n_" + which)
        arr = getattr(self, which)
        return [(arr[i].first_slot, arr[i].n_slots) for i in range(n)]


class LSState(Structure):
    _fields_ = [("dim", c_int32), ("reserved", c_int32), ("n_tokens", c_int64), ("gram", c_void_p)]


class IspaError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} (status {status})")


_lib = None

# name -> (restype, argtypes)
_SIGS = {
    "ispa_status_string": (c_char_p, [c_int32]),
    "ispa_last_device_error": (c_int32, [POINTER(c_int32)]),
    "ispa_set_wait_limit_ns": (c_uint64, [c_uint64]),
    "ispa_debug_wait_probe": (c_int32, [c_uint64, c_void_p]),
    "ispa_debug_error_record": (c_int32, [POINTER(c_int32)]),
    "ispa_debug_set_heartbeat": (c_int32, [c_void_p, c_int32]),
    "ispa_debug_set_trace": (c_int32, [c_void_p, c_int32]),
    "ispa_debug_drop_k_tile": (c_int32, [c_int32]),
    "ispa_debug_static_scratch": (c_int32, [POINTER(c_void_p), POINTER(c_uint64), POINTER(c_uint32)]),
    "ispa_ring_bytes": (c_size_t, [POINTER(KVRing)]),
    "ispa_ring_slot": (c_int32, [POINTER(KVRing), c_int64]),
    "ispa_window_resolve": (c_int32, [POINTER(KVRing), Window, POINTER(KeySets)]),
    "ispa_kv_append": (c_int32, [POINTER(KVRing), c_void_p, c_void_p, c_int32, c_void_p]),
    "ispa_kv_append_layers": (c_int32, [POINTER(KVRing), c_int32, POINTER(c_void_p), POINTER(c_void_p),
                                        c_int32, c_void_p]),
    "ispa_attn_full": (c_int32, [POINTER(KVRing), c_void_p, c_void_p, c_void_p, c_int32, c_float, c_void_p,
                                 c_void_p, c_void_p]),
    "ispa_attn_local": (c_int32, [POINTER(KVRing), Window, c_void_p, c_void_p, c_void_p, c_int32, c_float,
                                  c_void_p, c_void_p, c_void_p]),
    "ispa_attn_full_ex": (c_int32, [POINTER(KVRing), c_void_p, c_void_p, c_void_p, c_int32, c_float, c_uint32,
                                    c_void_p, c_void_p, c_void_p]),
    "ispa_attn_local_ex": (c_int32, [POINTER(KVRing), Window, c_void_p, c_void_p, c_void_p, c_int32, c_float,
                                     c_uint32, c_void_p, c_void_p, c_void_p]),
    "ispa_attn_dual_ex": (c_int32, [POINTER(KVRing), Window, c_void_p, c_void_p, c_void_p, c_int32, c_float,
                                    c_uint32, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                                    c_void_p, c_size_t, c_void_p]),
    "ispa_attn_dual_workspace_size": (c_size_t, [c_int32, c_int32]),
    "ispa_attn_dual": (c_int32, [POINTER(KVRing), Window, c_void_p, c_void_p, c_void_p, c_int32, c_float,
                                 c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                                 c_size_t, c_void_p]),
    "ispa_attn_dual_static": (c_int32, [POINTER(KVRing), Window, c_void_p, c_void_p, c_void_p, c_int32, c_float,
                                        c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p]),
    "ispa_attn_hist": (c_int32, [POINTER(KVRing), Window, c_void_p, c_int32, c_float, c_void_p, c_void_p, c_void_p]),
    "ispa_lse_merge": (c_int32, [c_void_p, c_void_p, c_void_p, c_void_p, c_int32, c_int32, c_int32, c_void_p, c_void_p,
                                 c_void_p]),
    "ispa_discrepancy": (c_int32, [c_void_p, c_void_p, c_int32, c_int32, c_void_p, c_void_p, c_void_p]),
    "ispa_select_layers": (c_int32, [POINTER(c_double), c_int32, c_int32, POINTER(c_int32)]),
    "ispa_apply_absorption": (c_int32, [c_void_p, c_void_p, c_int32, c_int32, c_void_p]),
    "ispa_apply_absorption_bf16": (c_int32, [c_void_p, c_void_p, c_int32, c_int32, c_void_p]),
    "ispa_ring_compact": (c_int32, [POINTER(KVRing), Window, POINTER(KVRing), c_void_p]),
    "ispa_ls_state_bytes": (c_size_t, [c_int32]),
    "ispa_ls_state_reset": (c_int32, [POINTER(LSState), c_void_p]),
    "ispa_ls_accumulate_workspace_size": (c_size_t, [c_int32, c_int64]),
    "ispa_ls_accumulate": (c_int32, [POINTER(LSState), c_void_p, c_void_p, c_int64, c_void_p, c_size_t,
                                     c_void_p]),
    "ispa_ls_accumulate_ex": (c_int32, [POINTER(LSState), c_void_p, c_void_p, c_int64, c_uint32, c_void_p,
                                        c_size_t, c_void_p]),
    "ispa_ls_solve_workspace_size": (c_size_t, [c_int32, c_int32]),
    "ispa_quantize_heads_e4m3": (c_int32, [c_void_p, c_int64, c_int32, c_int32, c_void_p, c_void_p, c_void_p]),
    "ispa_quantize_q_e4m3": (c_int32, [c_void_p, c_int64, c_int32, c_int32, c_void_p, c_void_p, c_void_p]),
    "ispa_quantize_k_e4m3": (c_int32, [c_void_p, c_int64, c_int32, c_int32, c_void_p, c_void_p, c_void_p]),
    "ispa_kv_append_qk8": (c_int32, [POINTER(KVRing), c_void_p, c_void_p, c_int32, c_void_p, c_void_p]),
    "ispa_ring_vt_stride": (c_int64, [POINTER(KVRing)]),
    "ispa_quantize_vt_e4m3": (c_int32, [c_void_p, c_int64, c_int32, c_int32, c_void_p, c_void_p, c_int64, c_void_p]),
    "ispa_kv_append_kv8": (c_int32, [POINTER(KVRing), c_void_p, c_void_p, c_int32, c_void_p, c_void_p, c_void_p]),
    "ispa_attn_full_kv8": (c_int32, [POINTER(KVRing), c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                                     c_void_p, c_int64, c_int32, c_float, c_void_p, c_void_p, c_void_p]),
    "ispa_attn_local_kv8": (c_int32, [POINTER(KVRing), c_void_p, c_void_p, Window, c_void_p, c_void_p, c_void_p,
                                      c_void_p, c_void_p, c_int64, c_int32, c_float, c_void_p, c_void_p, c_void_p]),
    "ispa_attn_dual_kv8": (c_int32, [POINTER(KVRing), c_void_p, c_void_p, Window, c_void_p, c_void_p, c_void_p,
                                     c_void_p, c_void_p, c_int64, c_int32, c_float, c_void_p, c_void_p, c_void_p,
                                     c_void_p, c_void_p, c_void_p, c_void_p, c_size_t, c_void_p]),
    "ispa_attn_full_qk8": (c_int32, [POINTER(KVRing), c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                                     c_int32, c_float, c_void_p, c_void_p, c_void_p]),
    "ispa_attn_dual_qk8": (c_int32, [POINTER(KVRing), c_void_p, Window, c_void_p, c_void_p, c_void_p, c_void_p,
                                     c_void_p, c_int32, c_float, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                                     c_void_p, c_void_p, c_size_t, c_void_p]),
    "ispa_attn_local_qk8": (c_int32, [POINTER(KVRing), c_void_p, Window, c_void_p, c_void_p, c_void_p, c_void_p,
                                      c_void_p, c_int32, c_float, c_void_p, c_void_p, c_void_p]),
    "ispa_quantize_rows_e4m3": (c_int32, [c_void_p, c_int64, c_int32, c_void_p, c_void_p, c_void_p]),
    "ispa_quantize_weight_e4m3": (c_int32, [c_void_p, c_void_p, c_int32, c_int32, c_void_p, c_void_p, c_void_p]),
    "ispa_linear_w8a8": (c_int32, [c_void_p, c_void_p, c_void_p, c_void_p, c_int64, c_int32, c_int32, c_void_p,
                                   c_void_p]),
    "ispa_ls_solve": (c_int32, [POINTER(LSState), c_void_p, c_int32, c_double, c_void_p, POINTER(c_double),
                                c_void_p, c_size_t, c_void_p]),
}


def lib() -> ctypes.CDLL:
    """The loaded libispa.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"libispa.so not built ({LIB_PATH}); run "
                               "python -m paper_2607_00712_gb300.build")
        L = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in _SIGS.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


def _ptr(x) -> int | None:
    """Device pointer of a tensor (or an int / None passed through)."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return x.data_ptr()


def _stream(s) -> int | None:
    if s is None:
        return None
    if isinstance(s, int):
        return s
    return s.cuda_stream


def _check(st: int, where: str) -> None:
    if st != ISPA_OK:
        raise IspaError(st, where)


def status_string(st: int) -> str:
    return lib().ispa_status_string(st).decode()


def ispa_last_device_error() -> tuple[int, int]:
    code = c_int32(0)
    st = lib().ispa_last_device_error(ctypes.byref(code))
    return st, code.value


def ispa_set_wait_limit_ns(ns: int) -> int:
    return lib().ispa_set_wait_limit_ns(ns)


def ispa_debug_wait_probe(limit_ns: int, stream=None) -> None:
    _check(lib().ispa_debug_wait_probe(limit_ns, _stream(stream)), "ispa_debug_wait_probe")


def ispa_debug_error_record() -> list[int]:
    rec = (c_int32 * 8)()
    _check(lib().ispa_debug_error_record(rec), "ispa_debug_error_record")
    return list(rec)


def ispa_debug_set_heartbeat(counters, n_slots: int) -> None:
    _check(lib().ispa_debug_set_heartbeat(_ptr(counters), n_slots), "ispa_debug_set_heartbeat")


def ispa_debug_set_trace(buf, n_tiles: int) -> None:
    _check(lib().ispa_debug_set_trace(_ptr(buf), n_tiles), "ispa_debug_set_trace")


def ispa_debug_drop_k_tile(tile: int) -> None:
    _check(lib().ispa_debug_drop_k_tile(tile), "ispa_debug_drop_k_tile")


def ispa_debug_static_scratch() -> tuple[int, int, int]:
    """(device address, context id, lookups so far) of ispa_attn_dual_static's scratch array."""
    a, c, n = c_void_p(), c_uint64(), c_uint32()
    _check(lib().ispa_debug_static_scratch(ctypes.byref(a), ctypes.byref(c), ctypes.byref(n)),
           "ispa_debug_static_scratch")
    return int(a.value or 0), int(c.value), int(n.value)


def ispa_ring_bytes(ring: KVRing) -> int:
    return lib().ispa_ring_bytes(ctypes.byref(ring))


def ispa_ring_slot(ring: KVRing, frame: int) -> int:
    return lib().ispa_ring_slot(ctypes.byref(ring), frame)


def ispa_window_resolve(ring: KVRing, win: Window) -> KeySets:
    ks = KeySets()
    _check(lib().ispa_window_resolve(ctypes.byref(ring), win, ctypes.byref(ks)), "ispa_window_resolve")
    return ks


def ispa_kv_append(ring: KVRing, k_new, v_new, n_frames: int, stream=None) -> None:
    _check(lib().ispa_kv_append(ctypes.byref(ring), _ptr(k_new), _ptr(v_new), n_frames, _stream(stream)),
           "ispa_kv_append")


def ispa_kv_append_layers(rings, k_new: list, v_new: list, n_frames: int, stream=None) -> None:
    """rings: a ctypes array of KVRing (advanced in place)."""
    n = len(rings)
    ks = (c_void_p * n)(*[_ptr(x) for x in k_new])
    vs = (c_void_p * n)(*[_ptr(x) for x in v_new])
    _check(lib().ispa_kv_append_layers(rings, n, ks, vs, n_frames, _stream(stream)), "ispa_kv_append_layers")


def ispa_attn_full(ring: KVRing, q, k_cur, v_cur, n_q: int, scale: float, out, lse=None, stream=None) -> None:
    _check(lib().ispa_attn_full(ctypes.byref(ring), _ptr(q), _ptr(k_cur), _ptr(v_cur), n_q, scale, _ptr(out),
                                _ptr(lse), _stream(stream)), "ispa_attn_full")


def ispa_attn_local(ring: KVRing, win: Window, q, k_cur, v_cur, n_q: int, scale: float, out, lse=None,
                    stream=None) -> None:
    _check(lib().ispa_attn_local(ctypes.byref(ring), win, _ptr(q), _ptr(k_cur), _ptr(v_cur), n_q, scale,
                                 _ptr(out), _ptr(lse), _stream(stream)), "ispa_attn_local")


def ispa_attn_full_ex(ring: KVRing, q, k_cur, v_cur, n_q: int, scale: float, flags: int, out, lse=None,
                      stream=None) -> None:
    _check(lib().ispa_attn_full_ex(ctypes.byref(ring), _ptr(q), _ptr(k_cur), _ptr(v_cur), n_q, scale, flags,
                                   _ptr(out), _ptr(lse), _stream(stream)), "ispa_attn_full_ex")


def ispa_attn_local_ex(ring: KVRing, win: Window, q, k_cur, v_cur, n_q: int, scale: float, flags: int, out,
                       lse=None, stream=None) -> None:
    _check(lib().ispa_attn_local_ex(ctypes.byref(ring), win, _ptr(q), _ptr(k_cur), _ptr(v_cur), n_q, scale,
                                    flags, _ptr(out), _ptr(lse), _stream(stream)), "ispa_attn_local_ex")


def ispa_attn_dual_ex(ring: KVRing, win: Window, q, k_cur, v_cur, n_q: int, scale: float, flags: int, a_full,
                      a_loc, disc, disc_sq_sum, lse_full=None, lse_loc=None, workspace=None, ws_bytes: int = 0,
                      stream=None) -> None:
    _check(lib().ispa_attn_dual_ex(ctypes.byref(ring), win, _ptr(q), _ptr(k_cur), _ptr(v_cur), n_q, scale,
                                   flags, _ptr(a_full), _ptr(a_loc), _ptr(disc), _ptr(disc_sq_sum),
                                   _ptr(lse_full), _ptr(lse_loc), _ptr(workspace), ws_bytes, _stream(stream)),
           "ispa_attn_dual_ex")


def ispa_attn_dual_workspace_size(num_heads: int, n_q: int) -> int:
    return lib().ispa_attn_dual_workspace_size(num_heads, n_q)


def ispa_attn_dual(ring: KVRing, win: Window, q, k_cur, v_cur, n_q: int, scale: float, a_full, a_loc, disc,
                   disc_sq_sum, lse_full=None, lse_loc=None, workspace=None, ws_bytes: int = 0,
                   stream=None) -> None:
    _check(lib().ispa_attn_dual(ctypes.byref(ring), win, _ptr(q), _ptr(k_cur), _ptr(v_cur), n_q, scale,
                                _ptr(a_full), _ptr(a_loc), _ptr(disc), _ptr(disc_sq_sum), _ptr(lse_full),
                                _ptr(lse_loc), _ptr(workspace), ws_bytes, _stream(stream)), "ispa_attn_dual")


def ispa_attn_dual_static(ring: KVRing, win: Window, q, k_cur, v_cur, n_q: int, scale: float, a_full, a_loc,
                          disc, disc_sq_sum, lse_full=None, lse_loc=None, stream=None) -> None:
    """ispa_attn_dual with the library's own fixed scratch (for callers that cannot allocate)."""
    _check(lib().ispa_attn_dual_static(ctypes.byref(ring), win, _ptr(q), _ptr(k_cur), _ptr(v_cur), n_q, scale,
                                       _ptr(a_full), _ptr(a_loc), _ptr(disc), _ptr(disc_sq_sum), _ptr(lse_full),
                                       _ptr(lse_loc), _stream(stream)), "ispa_attn_dual_static")


def ispa_attn_hist(ring: KVRing, win: Window, q, n_q: int, scale: float, out, lse, stream=None) -> None:
    _check(lib().ispa_attn_hist(ctypes.byref(ring), win, _ptr(q), n_q, scale, _ptr(out), _ptr(lse), _stream(stream)),
           "ispa_attn_hist")


def ispa_lse_merge(o_a, lse_a, o_b, lse_b, n_q: int, num_heads: int, head_dim: int, out, lse_out=None,
                   stream=None) -> None:
    _check(lib().ispa_lse_merge(_ptr(o_a), _ptr(lse_a), _ptr(o_b), _ptr(lse_b), n_q, num_heads, head_dim, _ptr(out),
                                _ptr(lse_out), _stream(stream)), "ispa_lse_merge")


def ispa_discrepancy(a_full, a_loc, n_q: int, dim: int, disc, disc_sq_sum, stream=None) -> None:
    _check(lib().ispa_discrepancy(_ptr(a_full), _ptr(a_loc), n_q, dim, _ptr(disc), _ptr(disc_sq_sum),
                                  _stream(stream)), "ispa_discrepancy")


def ispa_select_layers(eps, k: int) -> list[int]:
    n = len(eps)
    e = (c_double * n)(*eps)
    out = (c_int32 * n)()
    _check(lib().ispa_select_layers(e, n, k, out), "ispa_select_layers")
    return list(out)


def ispa_apply_absorption(W, dW, dim: int, d_out: int, stream=None) -> None:
    _check(lib().ispa_apply_absorption(_ptr(W), _ptr(dW), dim, d_out, _stream(stream)), "ispa_apply_absorption")


def ispa_apply_absorption_bf16(W, dW, dim: int, d_out: int, stream=None) -> None:
    _check(lib().ispa_apply_absorption_bf16(_ptr(W), _ptr(dW), dim, d_out, _stream(stream)),
           "ispa_apply_absorption_bf16")


def ispa_ring_compact(src: KVRing, win: Window, dst: KVRing, stream=None) -> None:
    _check(lib().ispa_ring_compact(ctypes.byref(src), win, ctypes.byref(dst), _stream(stream)), "ispa_ring_compact")


def ispa_ls_state_bytes(dim: int) -> int:
    return lib().ispa_ls_state_bytes(dim)


def ispa_ls_state_reset(state: LSState, stream=None) -> None:
    _check(lib().ispa_ls_state_reset(ctypes.byref(state), _stream(stream)), "ispa_ls_state_reset")


def ispa_ls_accumulate_workspace_size(dim: int, T: int) -> int:
    return lib().ispa_ls_accumulate_workspace_size(dim, T)


def ispa_ls_accumulate(state: LSState, a_loc, a_full, T: int, workspace, ws_bytes: int, stream=None) -> None:
    _check(lib().ispa_ls_accumulate(ctypes.byref(state), _ptr(a_loc), _ptr(a_full), T, _ptr(workspace),
                                    ws_bytes, _stream(stream)), "ispa_ls_accumulate")


def ispa_ls_accumulate_ex(state: LSState, a_loc, a_full, T: int, flags: int, workspace, ws_bytes: int,
                          stream=None) -> None:
    _check(lib().ispa_ls_accumulate_ex(ctypes.byref(state), _ptr(a_loc), _ptr(a_full), T, flags, _ptr(workspace),
                                       ws_bytes, _stream(stream)), "ispa_ls_accumulate_ex")


def ispa_ls_solve_workspace_size(dim: int, d_out: int) -> int:
    return lib().ispa_ls_solve_workspace_size(dim, d_out)


def ispa_ls_solve(state: LSState, W, d_out: int, lam: float, dW, workspace, ws_bytes: int,
                  stream=None) -> float:
    eps = c_double(0.0)
    _check(lib().ispa_ls_solve(ctypes.byref(state), _ptr(W), d_out, lam, _ptr(dW), ctypes.byref(eps),
                               _ptr(workspace), ws_bytes, _stream(stream)), "ispa_ls_solve")
    return eps.value


# ---------------------------------------------------------------- W8A8 projection
def ispa_quantize_rows_e4m3(x, rows: int, cols: int, q, scale, stream=None) -> None:
    _check(lib().ispa_quantize_rows_e4m3(_ptr(x), rows, cols, _ptr(q), _ptr(scale), _stream(stream)),
           "ispa_quantize_rows_e4m3")


def ispa_quantize_weight_e4m3(W, dW, D: int, D_out: int, q_t, scale, stream=None) -> None:
    _check(lib().ispa_quantize_weight_e4m3(_ptr(W), _ptr(dW), D, D_out, _ptr(q_t), _ptr(scale), _stream(stream)),
           "ispa_quantize_weight_e4m3")


def ispa_linear_w8a8(a_q, a_scale, w_q, w_scale, T: int, D: int, D_out: int, out, stream=None) -> None:
    _check(lib().ispa_linear_w8a8(_ptr(a_q), _ptr(a_scale), _ptr(w_q), _ptr(w_scale), T, D, D_out, _ptr(out),
                                  _stream(stream)), "ispa_linear_w8a8")


# ---------------------------------------------------------------- 8-bit Q K^T attention
def ispa_quantize_heads_e4m3(x, n: int, H: int, d: int, q, scale, stream=None) -> None:
    _check(lib().ispa_quantize_heads_e4m3(_ptr(x), n, H, d, _ptr(q), _ptr(scale), _stream(stream)),
           "ispa_quantize_heads_e4m3")


def ispa_kv_append_qk8(ring: KVRing, k_new, v_new, n_frames: int, k_scale, stream=None) -> None:
    _check(lib().ispa_kv_append_qk8(ctypes.byref(ring), _ptr(k_new), _ptr(v_new), n_frames, _ptr(k_scale),
                                    _stream(stream)), "ispa_kv_append_qk8")


def ispa_attn_full_qk8(ring: KVRing, k_ring_scale, q8, q_scale, k8_cur, k_cur_scale, v_cur, n_q: int,
                       scale: float, out, lse=None, stream=None) -> None:
    _check(lib().ispa_attn_full_qk8(ctypes.byref(ring), _ptr(k_ring_scale), _ptr(q8), _ptr(q_scale), _ptr(k8_cur),
                                    _ptr(k_cur_scale), _ptr(v_cur), n_q, scale, _ptr(out), _ptr(lse),
                                    _stream(stream)), "ispa_attn_full_qk8")


def ispa_attn_local_qk8(ring: KVRing, k_ring_scale, win: Window, q8, q_scale, k8_cur, k_cur_scale, v_cur,
                        n_q: int, scale: float, out, lse=None, stream=None) -> None:
    _check(lib().ispa_attn_local_qk8(ctypes.byref(ring), _ptr(k_ring_scale), win, _ptr(q8), _ptr(q_scale),
                                     _ptr(k8_cur), _ptr(k_cur_scale), _ptr(v_cur), n_q, scale, _ptr(out),
                                     _ptr(lse), _stream(stream)), "ispa_attn_local_qk8")


def ispa_quantize_q_e4m3(x, n: int, H: int, d: int, q, scale, stream=None) -> None:
    _check(lib().ispa_quantize_q_e4m3(_ptr(x), n, H, d, _ptr(q), _ptr(scale), _stream(stream)),
           "ispa_quantize_q_e4m3")


def ispa_quantize_k_e4m3(x, n: int, H: int, d: int, scale, q, stream=None) -> None:
    _check(lib().ispa_quantize_k_e4m3(_ptr(x), n, H, d, _ptr(scale), _ptr(q), _stream(stream)),
           "ispa_quantize_k_e4m3")


def ispa_ring_vt_stride(ring: KVRing) -> int:
    return lib().ispa_ring_vt_stride(ctypes.byref(ring))


def ispa_quantize_vt_e4m3(x, n: int, H: int, d: int, scale, qt, ld: int, stream=None) -> None:
    _check(lib().ispa_quantize_vt_e4m3(_ptr(x), n, H, d, _ptr(scale), _ptr(qt), ld, _stream(stream)),
           "ispa_quantize_vt_e4m3")


def ispa_kv_append_kv8(ring: KVRing, k_new, v_new, n_frames: int, k_scale, v_scale, stream=None) -> None:
    _check(lib().ispa_kv_append_kv8(ctypes.byref(ring), _ptr(k_new), _ptr(v_new), n_frames, _ptr(k_scale),
                                    _ptr(v_scale), _stream(stream)), "ispa_kv_append_kv8")


def ispa_attn_full_kv8(ring: KVRing, k_ring_scale, v_scale, q8, q_scale, k8_cur, k_cur_scale, vt8_cur, vt_ld: int,
                       n_q: int, scale: float, out, lse=None, stream=None) -> None:
    _check(lib().ispa_attn_full_kv8(ctypes.byref(ring), _ptr(k_ring_scale), _ptr(v_scale), _ptr(q8), _ptr(q_scale),
                                    _ptr(k8_cur), _ptr(k_cur_scale), _ptr(vt8_cur), vt_ld, n_q, scale, _ptr(out),
                                    _ptr(lse), _stream(stream)), "ispa_attn_full_kv8")


def ispa_attn_local_kv8(ring: KVRing, k_ring_scale, v_scale, win: Window, q8, q_scale, k8_cur, k_cur_scale, vt8_cur,
                        vt_ld: int, n_q: int, scale: float, out, lse=None, stream=None) -> None:
    _check(lib().ispa_attn_local_kv8(ctypes.byref(ring), _ptr(k_ring_scale), _ptr(v_scale), win, _ptr(q8),
                                     _ptr(q_scale), _ptr(k8_cur), _ptr(k_cur_scale), _ptr(vt8_cur), vt_ld, n_q, scale,
                                     _ptr(out), _ptr(lse), _stream(stream)), "ispa_attn_local_kv8")


def ispa_attn_dual_kv8(ring: KVRing, k_ring_scale, v_scale, win: Window, q8, q_scale, k8_cur, k_cur_scale, vt8_cur,
                       vt_ld: int, n_q: int, scale: float, a_full, a_loc, disc, disc_sq_sum, lse_full=None,
                       lse_loc=None, workspace=None, ws_bytes: int = 0, stream=None) -> None:
    _check(lib().ispa_attn_dual_kv8(ctypes.byref(ring), _ptr(k_ring_scale), _ptr(v_scale), win, _ptr(q8),
                                    _ptr(q_scale), _ptr(k8_cur), _ptr(k_cur_scale), _ptr(vt8_cur), vt_ld, n_q, scale,
                                    _ptr(a_full), _ptr(a_loc), _ptr(disc), _ptr(disc_sq_sum), _ptr(lse_full),
                                    _ptr(lse_loc), _ptr(workspace), ws_bytes, _stream(stream)), "ispa_attn_dual_kv8")


def ispa_attn_dual_qk8(ring: KVRing, k_ring_scale, win: Window, q8, q_scale, k8_cur, k_cur_scale, v_cur, n_q: int,
                       scale: float, a_full, a_loc, disc, disc_sq_sum, lse_full=None, lse_loc=None, workspace=None,
                       ws_bytes: int = 0, stream=None) -> None:
    _check(lib().ispa_attn_dual_qk8(ctypes.byref(ring), _ptr(k_ring_scale), win, _ptr(q8), _ptr(q_scale),
                                    _ptr(k8_cur), _ptr(k_cur_scale), _ptr(v_cur), n_q, scale, _ptr(a_full),
                                    _ptr(a_loc), _ptr(disc), _ptr(disc_sq_sum), _ptr(lse_full), _ptr(lse_loc),
                                    _ptr(workspace), ws_bytes, _stream(stream)), "ispa_attn_dual_qk8")

