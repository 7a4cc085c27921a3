"""ispa_attn_dual_static (no workspace, no allocation) against ispa_attn_dual.

The static entry point serves callers that cannot allocate device memory when
they run the warmup pass (a streaming loop with memory fixed at start-up, a
plug-in without an allocator).  It must return what the workspace entry point
returns, call after call, although every call reuses the same library-owned
scratch array.  This file is collected last on purpose.
"""
import ctypes

import numpy as np
import pytest

torch = pytest.importorskip("torch")

from gpu_helpers import Step, assert_close_attn  # noqa: E402
from paper_2607_00712_gb300 import abi  # noqa: E402
from paper_2607_00712_gb300.device import Window, to_f32  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2607_00712_gb300.build import build_library
    build_library()
    abi.lib()


def _outputs(st):
    D = st.H * st.d
    bf = torch.bfloat16
    return dict(a_full=torch.empty(st.n_q, D, dtype=bf, device="cuda"),
                a_loc=torch.empty(st.n_q, D, dtype=bf, device="cuda"),
                disc=torch.empty(st.n_q, dtype=torch.float32, device="cuda"),
                dsum=torch.zeros(1, dtype=torch.float32, device="cuda"),
                lf=torch.empty(st.H, st.n_q, dtype=torch.float32, device="cuda"),
                ll=torch.empty(st.H, st.n_q, dtype=torch.float32, device="cuda"))


def _with_workspace(st, win):
    o = _outputs(st)
    wsb = abi.ispa_attn_dual_workspace_size(st.H, st.n_q)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    abi.ispa_attn_dual(st.ring.c, Window(*win), st.q, st.kc, st.vc, st.n_q, 0.0, o["a_full"], o["a_loc"],
                       o["disc"], o["dsum"], o["lf"], o["ll"], ws, wsb)
    torch.cuda.synchronize()
    return o


def _static(st, win):
    o = _outputs(st)
    abi.ispa_attn_dual_static(st.ring.c, Window(*win), st.q, st.kc, st.vc, st.n_q, 0.0, o["a_full"], o["a_loc"],
                              o["disc"], o["dsum"], o["lf"], o["ll"])
    torch.cuda.synchronize()
    return o


def _same(got, ref):
    for k in ("a_full", "a_loc"):
        assert_close_attn(to_f32(got[k]), to_f32(ref[k]), k)
    assert np.allclose(to_f32(got["disc"]), to_f32(ref["disc"]), rtol=1e-5, atol=1e-6)
    assert abs(float(got["dsum"].item()) - float(ref["dsum"].item())) <= 1e-4 * max(1.0, float(ref["dsum"].item()))
    assert np.abs(to_f32(got["lf"]) - to_f32(ref["lf"])).max() < 2e-3
    assert np.abs(to_f32(got["ll"]) - to_f32(ref["ll"])).max() < 2e-3


def test_static_scratch_matches_workspace_entry_point_two_calls_in_a_row():
    # two different problems back to back: the second call must not see the first one's scratch
    st1 = Step(21, P=100, H=3, d=128, n_past=9, n_chunk_frames=3, capacity=7)
    st2 = Step(22, P=64, H=2, d=64, n_past=5, n_chunk_frames=2, capacity=5)
    ref1 = _with_workspace(st1, (0, 2))
    ref2 = _with_workspace(st2, (0, 3))
    got1 = _static(st1, (0, 2))
    got2 = _static(st2, (0, 3))
    _same(got1, ref1)
    _same(got2, ref2)
    assert abi.ispa_last_device_error()[0] == abi.ISPA_OK


def test_static_scratch_rejects_oversize_before_launch():
    # num_heads * n_q above the fixed maximum: clear error, nothing enqueued
    r = abi.KVRing(2, 64, 16, 4, 0, 0, 2, 16, 16)
    n_q = (1 << 20) // 2 + 1
    st = abi.lib().ispa_attn_dual_static(ctypes.byref(r), Window(0, 1), 16, 16, 16, n_q, 0.0, 16, 16, 16, 16,
                                         None, None, None)
    assert st == abi.ISPA_ERR_WORKSPACE


_CONTEXT_CHILD = r"""
import ctypes, sys
sys.path.insert(0, sys.argv[1])
from paper_2607_00712_gb300 import abi
cu = ctypes.CDLL("libcuda.so.1")
assert cu.cuInit(0) == 0
a1, c1, n1 = abi.ispa_debug_static_scratch()          # the primary context, bound by the library
assert a1 != 0
assert abi.ispa_debug_static_scratch() == (a1, c1, n1)  # cached: no second lookup
dev = ctypes.c_int()
assert cu.cuDeviceGet(ctypes.byref(dev), 0) == 0
ctx = ctypes.c_void_p()
if not hasattr(cu, "cuCtxCreate_v2") or cu.cuCtxCreate_v2(ctypes.byref(ctx), 0, dev) != 0:
    print("no-ctx-create")
    sys.exit(0)
try:
    a2, c2, n2 = abi.ispa_debug_static_scratch()       # the caller's own context is current now
    assert c2 != c1 and n2 == n1 + 1, (c1, c2, n1, n2)
    assert abi.ispa_debug_static_scratch() == (a2, c2, n2)
finally:
    assert cu.cuCtxDestroy_v2(ctx) == 0                 # the primary context is current again
a3, c3, n3 = abi.ispa_debug_static_scratch()
assert (a3, c3) == (a1, c1) and n3 == n2, (a1, c1, a3, c3, n2, n3)
print("ok")
"""


def test_static_scratch_address_is_keyed_on_the_current_context():
    # A caller that makes its own CUDA context current must not be handed the scratch address
    # looked up in another context (a kernel given it would fault).  In a child process that
    # uses only the driver API and the library (no kernel is launched): the primary context's
    # address is looked up once and reused; a context the caller creates gets a lookup of its
    # own; once that context is destroyed the primary context's cached entry is used again.
    # A primary context re-created by cudaDeviceReset carries a new process-unique id too, so
    # it takes the same path as the created context here.
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    r = subprocess.run([sys.executable, "-c", _CONTEXT_CHILD, root], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stdout + r.stderr
    if "no-ctx-create" in r.stdout:
        pytest.skip("the driver offers no cuCtxCreate_v2")
    assert r.stdout.strip().endswith("ok"), r.stdout + r.stderr
