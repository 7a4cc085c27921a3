"""CPU check of the discrepancy bound the GPU dual-pass tests use (tests/gpu_helpers.py).

The dual pass stores A_full and A_loc in bf16 and takes disc_t = ||A_full,t - A_loc,t||_2
(Sec. 3.1's output discrepancy, reading: L2 norm over all H*d features) on the stored
values in fp32.  Here that computation is simulated from the oracle's exact outputs
(bf16 rounding, fp32 sums) and must pass the bound; discrepancies with a planted mistake
(a dropped head, a sum instead of a difference, the square not rooted, one token's value
swapped with its neighbour's) must fail it.
"""
import numpy as np
import pytest

from gpu_helpers import assert_disc_close
from oracle import attention as at
from paper_2607_00712_gb300 import synth


def _case(seed=3):
    s = synth.make_step(seed, 4, 48, 3, 64, 2)
    r = at.attn_dual(s.q, s.k_hist, s.v_hist, s.k_cur, s.v_cur, 48, 0, 1)
    return r


def _stored(r):
    """What the device stores and computes: bf16 outputs, fp32 differences and sums."""
    n = r["a_full"].shape[0]
    gf = synth.bf16_round(r["a_full"].astype(np.float32))
    gl = synth.bf16_round(r["a_loc"].astype(np.float32))
    d = (gf - gl).astype(np.float32).reshape(n, -1)
    disc = np.sqrt((d * d).sum(axis=1, dtype=np.float32))
    return gf, gl, disc


def test_simulated_device_discrepancy_passes():
    r = _case()
    gf, gl, disc = _stored(r)
    assert_disc_close(gf, gl, disc, r, "simulated", float((disc.astype(np.float64) ** 2).sum()))


@pytest.mark.parametrize("mistake", ["drop_head", "sum", "unrooted", "swapped_token"])
def test_planted_mistakes_fail(mistake):
    r = _case()
    gf, gl, disc = _stored(r)
    n = gf.shape[0]
    if mistake == "drop_head":
        d = (gf - gl)[:, 1:, :].reshape(n, -1)
        bad = np.sqrt((d * d).sum(axis=1))
    elif mistake == "sum":
        d = (gf + gl).reshape(n, -1)
        bad = np.sqrt((d * d).sum(axis=1))
    elif mistake == "unrooted":
        bad = disc * disc
    else:
        bad = disc.copy()
        bad[[0, 1]] = bad[[1, 0]]
    with pytest.raises(AssertionError):
        assert_disc_close(gf, gl, bad, r, mistake)
