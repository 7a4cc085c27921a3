"""Seeded fuzz of the LS accumulation (Sec. 3.2, Eq. 5) through the C-ABI.

Both operand forms (scaled fp16, the default, and the exact bf16 hi / lo pair), random hidden
sizes (both Gram kernels: 256 x 256 tiles when the size is a multiple of 256,
128 x 128 tiles otherwise), random token counts (ragged last 64-token block), one to three
accumulate calls into the same state, and shapes whose tile counts exceed the grid so that the
lockstep-wave phase of the wide kernel runs, not only its stream-K tail.  Every maintained
tile is compared with the oracle's fp64 sums (<= 1e-3 Frobenius-relative per block), and the
parts of the state the kernels must not write stay exactly zero.
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


def _cases():
    rng = np.random.default_rng(2024)
    out = [(2048, [64]), (3072, [64]), (4096, [100]), (2048, [64, 37])]   # full waves present
    for _ in range(10):
        D = int(rng.choice([128, 256, 384, 512, 640, 768, 1024]))
        n_calls = int(rng.integers(1, 4))
        out.append((D, [int(rng.integers(1, 2000)) for _ in range(n_calls)]))
    return out


def _maintained_mask(D):
    """Tiles of a symmetric block the kernels keep: every 128 x 128 tile on or above the
    diagonal, plus the tiles (2k+1, 2k) when D is a multiple of 256."""
    t = np.arange(D) // 128
    keep = t[None, :] >= t[:, None]
    if D % 256 == 0:
        keep |= (t[:, None] % 2 == 1) & (t[None, :] == t[:, None] - 1)
    return keep


@pytest.mark.parametrize("exact", [False, True], ids=["scaled", "exact"])
@pytest.mark.parametrize("D,Ts", _cases(), ids=lambda v: str(v))
def test_ls_accumulate_fuzz(D, Ts, exact):
    st = LS(D)
    ref = ols.ls_state(D)
    for i, T in enumerate(Ts):
        a_loc, a_full = synth.make_activations(7000 + 31 * D + 7 * i + T, T, D)
        wsb = abi.ispa_ls_accumulate_workspace_size(D, T)
        ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
        abi.ispa_ls_accumulate_ex(st.c, bf16_tensor(a_loc), bf16_tensor(a_full), T,
                                  abi.ISPA_LS_EXACT_DELTA if exact else 0, ws, wsb)
        ols.ls_accumulate(ref, a_loc, a_full)
    torch.cuda.synchronize()
    assert st.c.n_tokens == sum(Ts)
    full = st.gram.view(2 * D, 2 * D).double().cpu().numpy()
    G, X, S, low = full[:D, :D], full[:D, D:], full[D:, D:], full[D:, :D]
    keep = _maintained_mask(D)
    for name, got, want in (("G", G, ref["G"]), ("S", S, ref["S"])):
        rel = np.linalg.norm((got - want)[keep]) / np.linalg.norm(want[keep])
        assert rel <= 1e-3, (name, rel)
        assert np.all(got[~keep] == 0.0), f"{name}: a tile outside the maintained set was written"
    rel = np.linalg.norm(X - ref["X"]) / np.linalg.norm(ref["X"])
    assert rel <= 1e-3, ("X", rel)
    assert np.all(low == 0.0), "the lower-left block was written"
