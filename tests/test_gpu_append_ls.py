"""GPU parity: KV append (exact), LS accumulation (<= 1e-3 relative), LS solve, timeout path."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import keysets as ks  # noqa: E402
from oracle import ls as ols  # noqa: E402
from paper_2607_00712_gb300 import abi, synth  # noqa: E402
from paper_2607_00712_gb300.device import LS, Ring, bf16_tensor, to_f32  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2607_00712_gb300.build import build_library
    build_library()
    abi.lib()


@pytest.mark.parametrize("H,d,P,cap,n_sink,group", [(2, 64, 16, 5, 0, 2), (3, 128, 40, 7, 1, 3),
                                                    (2, 128, 1560, 4, 0, 3), (4, 64, 24, 6, 2, 1)])
def test_append_matches_slot_map(H, d, P, cap, n_sink, group):
    ring = Ring(H, d, P, cap, n_sink)
    expect_k = np.zeros((H, cap * P, d), np.float32)
    expect_v = np.zeros((H, cap * P, d), np.float32)
    rng = np.random.default_rng(H * 1000 + d)
    n_total = 3 * cap + 1
    f = 0
    while f < n_total:
        n = min(group, n_total - f)
        k = synth.bf16_round(rng.standard_normal((n * P, H, d), dtype=np.float32))
        v = synth.bf16_round(rng.standard_normal((n * P, H, d), dtype=np.float32))
        abi.ispa_kv_append(ring.c, bf16_tensor(k), bf16_tensor(v), n)
        for i in range(n):
            s = ks.ring_slot(f + i, cap, n_sink)
            expect_k[:, s * P:(s + 1) * P] = k[i * P:(i + 1) * P].transpose(1, 0, 2)
            expect_v[:, s * P:(s + 1) * P] = v[i * P:(i + 1) * P].transpose(1, 0, 2)
        f += n
        torch.cuda.synchronize()
        assert ring.frames_written == f
        assert np.array_equal(to_f32(ring.k), expect_k)
        assert np.array_equal(to_f32(ring.v), expect_v)


def test_append_layers_one_launch():
    H, d, P, cap = 2, 128, 30, 6
    rings = (abi.KVRing * 3)()
    keep = []
    for l in range(3):
        r = Ring(H, d, P, cap, 0)
        keep.append(r)
        rings[l] = r.c
    ks_ = [bf16_tensor(synth.bf16_round(np.full((2 * P, H, d), l + 1, np.float32))) for l in range(3)]
    vs_ = [bf16_tensor(synth.bf16_round(np.full((2 * P, H, d), -(l + 1), np.float32))) for l in range(3)]
    abi.ispa_kv_append_layers(rings, ks_, vs_, 2)
    torch.cuda.synchronize()
    for l in range(3):
        assert rings[l].frames_written == 2
        k = to_f32(keep[l].k)
        assert np.all(k[:, :2 * P] == l + 1) and np.all(k[:, 2 * P:] == 0)
        assert np.all(to_f32(keep[l].v)[:, :2 * P] == -(l + 1))


def _gpu_accumulate(D, batches):
    st = LS(D)
    for a_loc, a_full in batches:
        T = a_loc.shape[0]
        wsb = abi.ispa_ls_accumulate_workspace_size(D, T)
        ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
        abi.ispa_ls_accumulate(st.c, bf16_tensor(a_loc), bf16_tensor(a_full), T, ws, wsb)
    torch.cuda.synchronize()
    return st


def _upper_tiles_rel_err(got, want, sym, bn):
    """Frobenius-relative error over the tiles the kernel maintains."""
    D = want.shape[0]
    mask = np.ones_like(want, dtype=bool)
    if sym:
        for i in range(D):
            mask[i, : (i // 128 * 128) // bn * bn] = False
    diff = (got - want)[mask]
    return np.linalg.norm(diff) / np.linalg.norm(want[mask])


@pytest.mark.parametrize("D,T", [(128, 128), (256, 300), (384, 1000), (512, 4680)])
def test_ls_accumulate_matches_oracle(D, T):
    a_loc, a_full = synth.make_activations(10 + D, T, D)
    st = _gpu_accumulate(D, [(a_loc, a_full)])
    ref = ols.ls_accumulate(ols.ls_state(D), a_loc, a_full)
    G, X, S = st.blocks()
    bn = 256 if D % 256 == 0 else 128
    assert _upper_tiles_rel_err(G, ref["G"], True, bn) <= 1e-3
    assert np.linalg.norm(X - ref["X"]) / np.linalg.norm(ref["X"]) <= 1e-3
    assert _upper_tiles_rel_err(S, ref["S"], True, bn) <= 1e-3
    assert st.c.n_tokens == T


def test_ls_accumulate_over_steps():
    # 8 warmup steps of 300 tokens each add up to one accumulation over 2400 tokens
    D = 256
    batches = [synth.make_activations(100 + i, 300, D) for i in range(8)]
    st = _gpu_accumulate(D, batches)
    ref = ols.ls_state(D)
    for a, f in batches:
        ols.ls_accumulate(ref, a, f)
    G, X, S = st.blocks()
    assert np.linalg.norm(X - ref["X"]) / np.linalg.norm(ref["X"]) <= 1e-3
    assert _upper_tiles_rel_err(G, ref["G"], True, 256) <= 1e-3
    assert _upper_tiles_rel_err(S, ref["S"], True, 256) <= 1e-3


def _solve_gpu(st, W, lam):
    D, Do = W.shape
    wsb = abi.ispa_ls_solve_workspace_size(D, Do)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    dW = torch.empty(D, Do, dtype=torch.float32, device="cuda")
    eps = abi.ispa_ls_solve(st.c, torch.from_numpy(W).cuda(), Do, lam, dW, ws, wsb)
    return to_f32(dW).astype(np.float64), eps


@pytest.mark.parametrize("D,Do,T", [(128, 128, 640), (256, 192, 2000)])
def test_ls_solve_planted(D, Do, T):
    # Exactly realisable instance built in fp64, then rounded to bf16 for both paths.
    r = np.random.default_rng(D)
    A = r.standard_normal((T, D))
    W = (r.standard_normal((D, Do)) / np.sqrt(D) + np.eye(D, Do)).astype(np.float32)
    dW_star = r.standard_normal((D, Do)) * 0.05
    delta = A @ dW_star @ np.linalg.pinv(W.astype(np.float64))
    a_loc = synth.bf16_round(A.astype(np.float32))
    a_full = synth.bf16_round((A + delta).astype(np.float32))
    st = _gpu_accumulate(D, [(a_loc, a_full)])
    ref = ols.ls_accumulate(ols.ls_state(D), a_loc, a_full)
    lam = 1e-3
    dW_ref, eps_ref = ols.ls_solve(ref["G"], ref["X"], ref["S"], W, lam)
    dW, eps = _solve_gpu(st, W, lam)
    assert np.linalg.norm(dW - dW_ref) / np.linalg.norm(dW_ref) <= 1e-3
    scale = float(np.sum(W.astype(np.float64) * (ref["S"] @ W)))   # tr(W^T S W)
    assert abs(eps - eps_ref) <= 1e-3 * scale
    # normal equations with the oracle's sums
    res = (ref["G"] + lam * np.eye(D)) @ dW - ref["X"] @ W
    assert np.linalg.norm(res) / np.linalg.norm(ref["X"] @ W) <= 1e-3
    # the planted modulation is recovered up to the bf16 rounding of the inputs
    assert np.linalg.norm(dW - dW_star) / np.linalg.norm(dW_star) <= 5e-2


def test_ls_solve_not_spd():
    st = LS(128)                       # G = 0, lambda = 0: the first pivot is 0
    W = np.eye(128, dtype=np.float32)
    with pytest.raises(abi.IspaError) as e:
        _solve_gpu(st, W, 0.0)
    assert e.value.status == abi.ISPA_ERR_NOT_SPD


def test_bounded_wait_reports_timeout():
    abi.ispa_last_device_error()       # clear
    abi.ispa_debug_wait_probe(2_000_000)   # 2 ms on a barrier nothing arrives at
    torch.cuda.synchronize()
    st, code = abi.ispa_last_device_error()
    assert st == abi.ISPA_ERR_TIMEOUT and code == 1
    st, code = abi.ispa_last_device_error()
    assert st == abi.ISPA_OK and code == 0
    # the context is still usable
    x = torch.ones(4, device="cuda")
    assert float(x.sum()) == 4.0


def test_append_sixteen_frames_the_largest_single_append():
    H, d, P, cap = 2, 64, 24, 20
    ring = Ring(H, d, P, cap, 1)
    rng = np.random.default_rng(16)
    k = synth.bf16_round(rng.standard_normal((16 * P, H, d), dtype=np.float32))
    v = synth.bf16_round(rng.standard_normal((16 * P, H, d), dtype=np.float32))
    ring.c.frames_written = 7                      # the 16 frames wrap around the non-sink slots
    abi.ispa_kv_append(ring.c, bf16_tensor(k), bf16_tensor(v), 16)
    torch.cuda.synchronize()
    assert ring.frames_written == 23
    kk, vv = to_f32(ring.k), to_f32(ring.v)
    for i in range(16):
        s = ks.ring_slot(7 + i, cap, 1)
        assert np.array_equal(kk[:, s * P:(s + 1) * P], k[i * P:(i + 1) * P].transpose(1, 0, 2))
        assert np.array_equal(vv[:, s * P:(s + 1) * P], v[i * P:(i + 1) * P].transpose(1, 0, 2))
