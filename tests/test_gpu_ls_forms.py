"""GPU parity: the two operand forms of the least-squares sums (Sec. 3.2, Eq. 5).

* scaled (ispa_ls_accumulate): A_loc and Delta as fp16 times per-call powers of two;
* exact (ispa_ls_accumulate_ex with ISPA_LS_EXACT_DELTA): Delta as a bf16 hi / lo pair.

Both are compared with the oracle's fp64 sums (<= 1e-3 Frobenius-relative per maintained
block, nothing written outside it) on seeded activations, and with each other where the scaled
form is exact by construction.  The scale choice is exercised at the ends of the range (huge,
tiny, all-zero Delta, a few large outliers, calls of very different magnitude into one state),
and back-to-back calls on one stream check the ordering of the programmatically dependent
launches (amax -> convert -> Gram -> next call's Gram).
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import ls as ols  # noqa: E402
from paper_2607_00712_gb300 import abi, synth  # noqa: E402
from paper_2607_00712_gb300.device import LS, bf16_tensor  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2607_00712_gb300.build import build_library
    build_library()
    abi.lib()


def _bf16(x):
    return torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(torch.bfloat16).float().numpy()


def _accumulate(st, a_loc, a_full, exact):
    T, D = a_loc.shape
    wsb = abi.ispa_ls_accumulate_workspace_size(D, T)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    a, f = bf16_tensor(a_loc), bf16_tensor(a_full)
    if exact:
        abi.ispa_ls_accumulate_ex(st.c, a, f, T, abi.ISPA_LS_EXACT_DELTA, ws, wsb)
    else:
        abi.ispa_ls_accumulate(st.c, a, f, T, ws, wsb)
    return (a, f, ws)   # keep the buffers alive until the stream has used them


def _maintained_mask(D):
    t = np.arange(D) // 128
    keep = t[None, :] >= t[:, None]
    if D % 256 == 0:
        keep |= (t[:, None] % 2 == 1) & (t[None, :] == t[:, None] - 1)
    return keep


def _rel(a, b):
    return np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300)


def _check(st, ref, tol=1e-3):
    D = st.c.dim
    full = st.gram.view(2 * D, 2 * D).double().cpu().numpy()
    G, X, S, low = full[:D, :D], full[:D, D:], full[D:, D:], full[D:, :D]
    keep = _maintained_mask(D)
    errs = {}
    for name, got, want in (("G", G, ref["G"]), ("S", S, ref["S"])):
        assert np.all(got[~keep] == 0.0), f"{name}: a tile outside the maintained set was written"
        errs[name] = _rel(got[keep], want[keep]) if np.any(want[keep]) else np.abs(got[keep]).max()
    errs["X"] = _rel(X, ref["X"]) if np.any(ref["X"]) else np.abs(X).max()
    assert np.all(low == 0.0), "the lower-left block was written"
    for k, v in errs.items():
        assert v <= tol, (k, v)
    return full


@pytest.mark.parametrize("exact", [False, True], ids=["scaled", "exact"])
@pytest.mark.parametrize("D,Ts", [(128, [100]), (256, [1, 3]), (384, [64, 1999]), (512, [4680]),
                                  (1536, [4680, 37]), (2048, [640])], ids=str)
def test_both_forms_against_oracle(D, Ts, exact):
    st = LS(D)
    ref = ols.ls_state(D)
    keep = []
    for i, T in enumerate(Ts):
        a_loc, a_full = synth.make_activations(8100 + 13 * D + 5 * i + T, T, D)
        keep.append(_accumulate(st, a_loc, a_full, exact))
        ols.ls_accumulate(ref, a_loc, a_full)
    torch.cuda.synchronize()
    assert abi.ispa_last_device_error()[0] == abi.ISPA_OK
    assert st.c.n_tokens == sum(Ts)
    _check(st, ref)


def test_scaled_form_is_exact_when_delta_fits_fp16():
    # A_loc and A_full multiples of 2^-6 below 4 in magnitude (8 significant bits at most, so
    # bf16 holds them), Delta with at most 4: every value survives the fp16 conversion at the
    # chosen scale, so the scaled form runs the same products as the exact one (which has
    # lo = 0 here); the two states differ by fp32 summation order only
    D, T = 512, 3000
    rng = np.random.default_rng(4)
    a_loc = rng.integers(-200, 201, size=(T, D)).astype(np.float32) * np.float32(2.0 ** -6)
    q = rng.integers(-15, 16, size=(T, D)).astype(np.float32) * np.float32(2.0 ** -6)
    a_full = a_loc + q
    assert np.array_equal(_bf16(a_full), a_full)
    s1, s2 = LS(D), LS(D)
    keep = [_accumulate(s1, a_loc, a_full, False), _accumulate(s2, a_loc, a_full, True)]
    torch.cuda.synchronize()
    f1 = s1.gram.view(2 * D, 2 * D).double().cpu().numpy()
    f2 = s2.gram.view(2 * D, 2 * D).double().cpu().numpy()
    assert _rel(f1, f2) <= 1e-6
    del keep


@pytest.mark.parametrize("case", ["huge", "tiny", "zero_delta", "outliers", "mixed_calls"])
def test_scaled_form_range(case):
    D, T = 768, 2100
    rng = np.random.default_rng({"huge": 1, "tiny": 2, "zero_delta": 3, "outliers": 4, "mixed_calls": 5}[case])
    st = LS(D)
    ref = ols.ls_state(D)
    calls = []
    base = rng.standard_normal((T, D)).astype(np.float32)
    noise = 0.5 * rng.standard_normal((T, D)).astype(np.float32)
    if case == "huge":        # |A| ~ 2^20, |Delta| ~ 2^19: beyond fp16 without the scale
        calls.append((_bf16(base * 2.0 ** 20), _bf16((base + noise) * 2.0 ** 20)))
    elif case == "tiny":      # |A| ~ 2^-40, |Delta| ~ 2^-41: below fp16's normal range without it
        calls.append((_bf16(base * 2.0 ** -40), _bf16((base + noise) * 2.0 ** -40)))
    elif case == "zero_delta":
        a = _bf16(base)
        calls.append((a, a.copy()))
    elif case == "outliers":  # 50 Delta values a thousand times the rest set the scale
        f = (base + noise).reshape(-1)
        f[rng.choice(f.size, 50, replace=False)] *= 1000.0
        calls.append((_bf16(base), _bf16(f.reshape(T, D))))
    else:                     # each call its own scale, into one state
        calls.append((_bf16(base * 2.0 ** 12), _bf16((base + noise) * 2.0 ** 12)))
        b2 = rng.standard_normal((T, D)).astype(np.float32)
        calls.append((_bf16(b2 * 2.0 ** -12), _bf16((b2 + noise) * 2.0 ** -12)))
    keep = []
    for a_loc, a_full in calls:
        keep.append(_accumulate(st, a_loc, a_full, False))
        ols.ls_accumulate(ref, a_loc, a_full)
    torch.cuda.synchronize()
    assert abi.ispa_last_device_error()[0] == abi.ISPA_OK
    full = _check(st, ref)
    if case == "zero_delta":
        assert np.all(full[:D, D:] == 0.0) and np.all(full[D:, D:] == 0.0)


@pytest.mark.parametrize("D", [384, 1536])
def test_back_to_back_accumulates_in_both_forms(D):
    # Six accumulate calls on one stream with no host synchronisation, alternating the forms:
    # each Gram launch starts under the end of the kernel before it and must see the state the
    # previous Gram launch wrote.
    st = LS(D)
    ref = ols.ls_state(D)
    keep = []
    for i in range(6):
        T = [700, 64, 1313, 5, 2048, 999][i]
        a_loc, a_full = synth.make_activations(9100 + 17 * i + D, T, D)
        ols.ls_accumulate(ref, a_loc, a_full)
        keep.append(_accumulate(st, a_loc, a_full, exact=bool(i % 2)))
    torch.cuda.synchronize()
    assert abi.ispa_last_device_error()[0] == abi.ISPA_OK
    _check(st, ref)


def test_many_short_calls_alternating_forms():
    # 40 calls of 1 to 130 tokens (ragged 64-token blocks, single-block and single-token calls),
    # alternating the two forms, all on one stream before one synchronisation
    D = 256
    rng = np.random.default_rng(77)
    st = LS(D)
    ref = ols.ls_state(D)
    keep = []
    total = 0
    for i in range(40):
        T = int(rng.integers(1, 131))
        a_loc, a_full = synth.make_activations(9300 + i, T, D)
        ols.ls_accumulate(ref, a_loc, a_full)
        keep.append(_accumulate(st, a_loc, a_full, exact=bool(i % 2)))
        total += T
    torch.cuda.synchronize()
    assert abi.ispa_last_device_error()[0] == abi.ISPA_OK
    assert st.c.n_tokens == total
    _check(st, ref)
