"""The whole ISPA flow through the C-ABI, on a small multi-layer synthetic rollout:

  warmup (Sec. 3.1 phase 1): every layer runs the dual pass per chunk step, accumulates the
      normal-equation sums (Eq. 5) and appends the chunk;
  transition (Sec. 3.2-3.3): every layer solves for dW and eps (Eq. 5-6), the k lowest-eps
      layers become L-layers, get W + dW (weight injection) and keep only their window
      (eviction into a small ring);
  inference: an L-layer's next chunk attends to the compacted ring.

Properties checked, beyond the per-component parity tests: eps is the residual of Eq. 4,
||A_loc (W + dW) - A_full W||_F^2 over the warmup tokens (plus the ridge term), so the
absorbed weight makes the local outputs reproduce the full-cache projection better than W
alone; the chosen layers are the ones with the smallest eps; the compacted ring gives the same
L-layer attention as the full ring restricted to the window.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from gpu_helpers import assert_close_attn  # noqa: E402
from paper_2607_00712_gb300 import abi, synth  # noqa: E402
from paper_2607_00712_gb300.device import LS, Ring, Window, bf16_tensor, to_f32  # noqa: E402

pytestmark = pytest.mark.gpu
P, H, d, CHUNK, CAP, WARM_STEPS, N_LAYERS, K_L = 64, 2, 128, 2, 12, 3, 4, 2
D = H * d
LAM = 1e-3


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2607_00712_gb300.build import build_library
    build_library()
    abi.lib()


def _chunk(seed):
    s = synth.make_step(seed, 0, P, H, d, n_chunk_frames=CHUNK)
    return bf16_tensor(s.q), bf16_tensor(s.k_cur), bf16_tensor(s.v_cur)


def test_warmup_transition_inference():
    win = Window(0, 2)
    n = CHUNK * P
    rings, states, a_locs, a_fulls = [], [], [[] for _ in range(N_LAYERS)], [[] for _ in range(N_LAYERS)]
    for layer in range(N_LAYERS):
        r = Ring(H, d, P, CAP, 0)
        for f0 in range(0, 4, CHUNK):                       # some history before the warmup
            _, k, v = _chunk(10_000 + 100 * layer + f0)
            abi.ispa_kv_append(r.c, k, v, CHUNK)
        rings.append(r)
        states.append(LS(D))
    wsb = abi.ispa_attn_dual_workspace_size(H, n)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    lwsb = abi.ispa_ls_accumulate_workspace_size(D, n)
    lws = torch.empty(lwsb, dtype=torch.uint8, device="cuda")
    disc = torch.empty(n, dtype=torch.float32, device="cuda")
    dsum = torch.zeros(1, dtype=torch.float32, device="cuda")
    # ---------------------------------------------------------------- warmup
    for step in range(WARM_STEPS):
        for layer in range(N_LAYERS):
            q, kc, vc = _chunk(20_000 + 100 * layer + step)
            a_full = torch.empty(n, D, dtype=torch.bfloat16, device="cuda")
            a_loc = torch.empty_like(a_full)
            abi.ispa_attn_dual(rings[layer].c, win, q, kc, vc, n, 0.0, a_full, a_loc, disc, dsum, None, None,
                               ws, wsb)
            abi.ispa_ls_accumulate(states[layer].c, a_loc, a_full, n, lws, lwsb)
            abi.ispa_kv_append(rings[layer].c, kc, vc, CHUNK)
            a_locs[layer].append(a_loc)
            a_fulls[layer].append(a_full)
    torch.cuda.synchronize()
    # ---------------------------------------------------------------- transition
    Ws = [torch.from_numpy(synth.make_weight(300 + layer, D, D)).cuda() for layer in range(N_LAYERS)]
    swsb = abi.ispa_ls_solve_workspace_size(D, D)
    sws = torch.empty(swsb, dtype=torch.uint8, device="cuda")
    eps, dWs = [], []
    for layer in range(N_LAYERS):
        dW = torch.empty(D, D, dtype=torch.float32, device="cuda")
        eps.append(abi.ispa_ls_solve(states[layer].c, Ws[layer], D, LAM, dW, sws, swsb))
        dWs.append(dW)
        # eps is the ridge objective of Eq. 4-5 at its minimiser, on the warmup tokens
        A = np.concatenate([to_f32(t) for t in a_locs[layer]]).astype(np.float64)
        F = np.concatenate([to_f32(t) for t in a_fulls[layer]]).astype(np.float64)
        W = Ws[layer].cpu().numpy().astype(np.float64)
        dw = dW.cpu().numpy().astype(np.float64)
        resid = np.sum((A @ (W + dw) - F @ W) ** 2)
        assert abs(eps[-1] - resid) <= 1e-3 * resid + 1e-6, (layer, eps[-1], resid)
        # the absorbed weight reproduces the full-cache projection better than W alone
        assert resid + LAM * np.sum(dw ** 2) <= np.sum((A @ W - F @ W) ** 2) * (1 + 1e-9)
    is_l = abi.ispa_select_layers(eps, K_L)
    assert sum(is_l) == K_L
    chosen = [i for i in range(N_LAYERS) if is_l[i]]
    assert max(eps[i] for i in chosen) <= min(eps[i] for i in range(N_LAYERS) if not is_l[i])
    for layer in chosen:
        W_before = Ws[layer].cpu().numpy()
        abi.ispa_apply_absorption(Ws[layer], dWs[layer], D, D)
        torch.cuda.synchronize()
        assert np.array_equal(Ws[layer].cpu().numpy(), W_before + dWs[layer].cpu().numpy())
    # ---------------------------------------------------------------- inference
    for layer in chosen:
        small = Ring(H, d, P, win.n_sink_frames + win.n_recent_frames, win.n_sink_frames)
        abi.ispa_ring_compact(rings[layer].c, win, small.c)
        q, kc, vc = _chunk(30_000 + layer)
        out_small = torch.empty(n, D, dtype=torch.bfloat16, device="cuda")
        out_big = torch.empty_like(out_small)
        abi.ispa_attn_local(small.c, win, q, kc, vc, n, 0.0, out_small)
        abi.ispa_attn_local(rings[layer].c, win, q, kc, vc, n, 0.0, out_big)
        torch.cuda.synchronize()
        got, want = to_f32(out_small), to_f32(out_big)
        assert_close_attn(got, want, f"layer {layer}: compacted ring vs full ring")
    st, code = abi.ispa_last_device_error()
    assert st == abi.ISPA_OK, code
