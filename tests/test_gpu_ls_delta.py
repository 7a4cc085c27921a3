"""GPU parity: the warmup dual pass that also writes Delta = A_full - A_loc as a bf16 hi / lo
pair, and the least-squares sums (Sec. 3.2, Eq. 5) taken from that pair.

* ispa_attn_dual_delta: a_full, a_loc and disc bit-identical to ispa_attn_dual's on the same
  inputs (the same attention launch; the pair comes from the launch that also reduces the
  discrepancy partials), the running sum of disc^2 equal to fp32 rounding, and the pair exactly the
  round-to-nearest-even split hi = bf16(Delta), lo = bf16(Delta - hi) of the difference of the
  stored outputs, Delta taken in fp32 (exact for bf16 operands one exponent range apart);
* ispa_ls_accumulate_delta: on seeded activations split on the host, G, X and S within 1e-3
  Frobenius-relative of the oracle's fp64 sums, nothing written outside the maintained
  tiles, and within fp32 reduction-order noise of ispa_ls_accumulate on (A_loc, A_full);
* the chain dual_delta -> ls_accumulate_delta at the 1.3B-shaped warmup step equals the
  two-input chain dual -> ls_accumulate to the same noise.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from gpu_helpers import Step  # noqa: E402
from oracle import ls as ols  # noqa: E402
from paper_2607_00712_gb300 import abi, synth  # noqa: E402
from paper_2607_00712_gb300.device import LS, Window, bf16_tensor, to_f32  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2607_00712_gb300.build import build_library
    build_library()
    abi.lib()


def _split_host(a_loc: np.ndarray, a_full: np.ndarray):
    """hi = RNE bf16 of Delta (fp32), lo = RNE bf16 of (Delta - hi), with torch's CPU conversions."""
    d = a_full.astype(np.float32) - a_loc.astype(np.float32)
    hi = torch.from_numpy(d).to(torch.bfloat16)
    lo = torch.from_numpy(d - hi.float().numpy()).to(torch.bfloat16)
    return hi, lo


def _bits(t):
    return t.contiguous().view(torch.int16).cpu().numpy()


def _dual(st: Step, win, delta: bool):
    D = st.H * st.d
    bf = torch.bfloat16
    a_full = torch.empty(st.n_q, D, dtype=bf, device="cuda")
    a_loc = torch.empty(st.n_q, D, dtype=bf, device="cuda")
    disc = torch.empty(st.n_q, dtype=torch.float32, device="cuda")
    dsum = torch.zeros(1, dtype=torch.float32, device="cuda")
    wsb = abi.ispa_attn_dual_workspace_size(st.H, st.n_q)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    out = dict(a_full=a_full, a_loc=a_loc, disc=disc, dsum=dsum)
    if delta:
        hi = torch.full((st.n_q, D), float("nan"), dtype=bf, device="cuda")
        lo = torch.full((st.n_q, D), float("nan"), dtype=bf, device="cuda")
        abi.ispa_attn_dual_delta(st.ring.c, Window(*win), st.q, st.kc, st.vc, st.n_q, 0.0, 0, a_full, a_loc, hi, lo,
                                 disc, dsum, None, None, ws, wsb)
        out.update(hi=hi, lo=lo)
    else:
        abi.ispa_attn_dual(st.ring.c, Window(*win), st.q, st.kc, st.vc, st.n_q, 0.0, a_full, a_loc, disc, dsum,
                           None, None, ws, wsb)
    torch.cuda.synchronize()
    return out


@pytest.mark.parametrize("shape", [
    dict(seed=0, P=64, H=2, d=64, n_past=4, n_chunk_frames=2, capacity=4, win=(0, 2)),
    dict(seed=1, P=100, H=3, d=128, n_past=12, n_chunk_frames=3, capacity=7, n_sink_pinned=1, win=(1, 2)),
    dict(seed=5, P=64, H=2, d=128, n_past=0, n_chunk_frames=2, capacity=4, win=(0, 2)),   # no history: Delta = 0
    dict(seed=62, P=1560, H=12, d=128, n_past=18, n_chunk_frames=3, capacity=18, win=(0, 6)),
], ids=["tiny", "ragged_wrapped", "no_history", "step_1.3b"])
def test_dual_delta_outputs_and_pair(shape):
    shape = dict(shape)
    win = shape.pop("win")
    seed = shape.pop("seed")
    st = Step(seed, **shape)
    ref = _dual(st, win, False)
    got = _dual(st, win, True)
    for k in ("a_full", "a_loc"):
        assert np.array_equal(_bits(got[k]), _bits(ref[k])), k
    assert np.array_equal(got["disc"].cpu().numpy(), ref["disc"].cpu().numpy())
    d1, d2 = float(got["dsum"].item()), float(ref["dsum"].item())
    assert abs(d1 - d2) <= 1e-5 * abs(d2) + 1e-30
    hi, lo = _split_host(to_f32(got["a_loc"]), to_f32(got["a_full"]))
    assert np.array_equal(_bits(got["hi"]), _bits(hi)), "hi"
    assert np.array_equal(_bits(got["lo"]), _bits(lo)), "lo"
    if len(st.resident) == 0:
        assert not np.any(to_f32(got["hi"])) and not np.any(to_f32(got["lo"]))
    assert abi.ispa_last_device_error()[0] == abi.ISPA_OK


def _maintained_mask(D):
    t = np.arange(D) // 128
    keep = t[None, :] >= t[:, None]
    if D % 256 == 0:
        keep |= (t[:, None] % 2 == 1) & (t[None, :] == t[:, None] - 1)
    return keep


def _rel(a, b):
    return np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300)


@pytest.mark.parametrize("D,Ts", [(128, [100]), (384, [64, 1999]), (512, [4680]), (1536, [4680, 37]),
                                  (2048, [640])], ids=str)
def test_ls_accumulate_delta_against_oracle(D, Ts):
    st, st2 = LS(D), LS(D)
    ref = ols.ls_state(D)
    for i, T in enumerate(Ts):
        a_loc, a_full = synth.make_activations(8100 + 13 * D + 5 * i + T, T, D)
        hi, lo = _split_host(a_loc, a_full)
        abi.ispa_ls_accumulate_delta(st.c, bf16_tensor(a_loc), hi.cuda(), lo.cuda(), T)
        wsb = abi.ispa_ls_accumulate_workspace_size(D, T)
        ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
        abi.ispa_ls_accumulate(st2.c, bf16_tensor(a_loc), bf16_tensor(a_full), T, ws, wsb)
        ols.ls_accumulate(ref, a_loc, a_full)
    torch.cuda.synchronize()
    assert st.c.n_tokens == sum(Ts)
    full = st.gram.view(2 * D, 2 * D).double().cpu().numpy()
    full2 = st2.gram.view(2 * D, 2 * D).double().cpu().numpy()
    G, X, S, low = full[:D, :D], full[:D, D:], full[D:, D:], full[D:, :D]
    keep = _maintained_mask(D)
    for name, got, want in (("G", G, ref["G"]), ("S", S, ref["S"])):
        assert _rel(got[keep], want[keep]) <= 1e-3, name
        assert np.all(got[~keep] == 0.0), name
    assert _rel(X, ref["X"]) <= 1e-3
    assert np.all(low == 0.0)
    # the same products as the two-input call: only the order of fp32 partial-sum additions differs
    assert _rel(full, full2) <= 1e-6


def test_dual_delta_chain_equals_two_input_chain_at_the_step_shape():
    st = Step(63, P=1560, H=12, d=128, n_past=18, n_chunk_frames=3, capacity=18)
    D, T = st.H * st.d, st.n_q
    ref = _dual(st, (0, 6), False)
    got = _dual(st, (0, 6), True)
    ls1, ls2 = LS(D), LS(D)
    abi.ispa_ls_accumulate_delta(ls1.c, got["a_loc"], got["hi"], got["lo"], T)
    wsb = abi.ispa_ls_accumulate_workspace_size(D, T)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    abi.ispa_ls_accumulate(ls2.c, ref["a_loc"], ref["a_full"], T, ws, wsb)
    torch.cuda.synchronize()
    for (n1, b1), b2 in zip(zip("GXS", ls1.blocks()), ls2.blocks()):
        assert _rel(b1, b2) <= 1e-6, n1
    assert abi.ispa_last_device_error()[0] == abi.ISPA_OK


def test_dual_delta_frame_causal_matches_dual_ex():
    # the option bits pass through: frame-causal chunk in both outputs, the pair from them
    st = Step(64, P=96, H=2, d=128, n_past=5, n_chunk_frames=3, capacity=8)
    D = st.H * st.d
    bf = torch.bfloat16
    outs = {}
    for name in ("ex", "delta"):
        a_full = torch.empty(st.n_q, D, dtype=bf, device="cuda")
        a_loc = torch.empty(st.n_q, D, dtype=bf, device="cuda")
        disc = torch.empty(st.n_q, dtype=torch.float32, device="cuda")
        dsum = torch.zeros(1, dtype=torch.float32, device="cuda")
        wsb = abi.ispa_attn_dual_workspace_size(st.H, st.n_q)
        ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
        if name == "ex":
            abi.ispa_attn_dual_ex(st.ring.c, Window(0, 2), st.q, st.kc, st.vc, st.n_q, 0.0, abi.ISPA_ATTN_FRAME_CAUSAL,
                                  a_full, a_loc, disc, dsum, None, None, ws, wsb)
            outs[name] = (a_full, a_loc, disc)
        else:
            hi = torch.empty(st.n_q, D, dtype=bf, device="cuda")
            lo = torch.empty(st.n_q, D, dtype=bf, device="cuda")
            abi.ispa_attn_dual_delta(st.ring.c, Window(0, 2), st.q, st.kc, st.vc, st.n_q, 0.0,
                                     abi.ISPA_ATTN_FRAME_CAUSAL, a_full, a_loc, hi, lo, disc, dsum, None, None, ws, wsb)
            outs[name] = (a_full, a_loc, disc, hi, lo)
    torch.cuda.synchronize()
    for a, b in zip(outs["ex"], outs["delta"][:3]):
        assert np.array_equal(a.cpu().view(torch.int32 if a.dtype == torch.float32 else torch.int16).numpy(),
                              b.cpu().view(torch.int32 if b.dtype == torch.float32 else torch.int16).numpy())
    hi, lo = _split_host(to_f32(outs["delta"][1]), to_f32(outs["delta"][0]))
    assert np.array_equal(_bits(outs["delta"][3]), _bits(hi)) and np.array_equal(_bits(outs["delta"][4]), _bits(lo))


@pytest.mark.parametrize("D", [384, 1536])
def test_back_to_back_accumulates_in_both_forms(D):
    # Six accumulate calls on one stream with no host synchronisation, alternating the two-input
    # and the pre-split form: each Gram launch starts under the end of the kernel before it and
    # must see the state the previous Gram launch wrote.
    st = LS(D)
    ref = ols.ls_state(D)
    bufs = []
    for i in range(6):
        T = [700, 64, 1313, 5, 2048, 999][i]
        a_loc, a_full = synth.make_activations(9100 + 17 * i + D, T, D)
        ols.ls_accumulate(ref, a_loc, a_full)
        a_d, f_d = bf16_tensor(a_loc), bf16_tensor(a_full)
        if i % 2:
            hi, lo = _split_host(a_loc, a_full)
            hi, lo = hi.cuda(), lo.cuda()
            bufs.append((a_d, hi, lo))
            abi.ispa_ls_accumulate_delta(st.c, a_d, hi, lo, T)
        else:
            wsb = abi.ispa_ls_accumulate_workspace_size(D, T)
            ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
            bufs.append((a_d, f_d, ws))
            abi.ispa_ls_accumulate(st.c, a_d, f_d, T, ws, wsb)
    torch.cuda.synchronize()
    assert abi.ispa_last_device_error()[0] == abi.ISPA_OK
    full = st.gram.view(2 * D, 2 * D).double().cpu().numpy()
    G, X, S = full[:D, :D], full[:D, D:], full[D:, D:]
    keep = _maintained_mask(D)
    assert _rel(G[keep], ref["G"][keep]) <= 1e-3
    assert _rel(S[keep], ref["S"][keep]) <= 1e-3
    assert _rel(X, ref["X"]) <= 1e-3
