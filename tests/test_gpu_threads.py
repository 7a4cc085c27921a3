"""Entry points called from several host threads at once, each with its own rings, LS state
and stream (the threading convention of include/ispa.h): every thread's attention outputs equal,
bit for bit, those of the same calls made one after another on one thread, and the sums that
use atomics agree to rounding.  (ctypes releases the GIL during each call, so the C entry points
really run concurrently: tensor-map encoding, launch set-up and the kernels' one-time shared-
memory settings.)"""
import threading

import numpy as np
import pytest

torch = pytest.importorskip("torch")

from paper_2607_00712_gb300 import abi, synth  # noqa: E402
from paper_2607_00712_gb300.device import LS, Ring, Window, bf16_tensor  # noqa: E402

pytestmark = pytest.mark.gpu
N_THREADS, ROUNDS = 4, 6


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2607_00712_gb300.build import build_library
    build_library()
    abi.lib()


class Job:
    """One thread's buffers: a ring with history, a chunk, outputs, an LS state, a stream."""

    def __init__(self, seed):
        P, H, d, F, L = 96, 2, 128, 6, 2
        s = synth.make_step(seed, F, P, H, d, n_chunk_frames=L)
        self.ring = Ring(H, d, P, F, 0)
        abi.ispa_kv_append(self.ring.c, bf16_tensor(s.k_hist[: 3 * P]), bf16_tensor(s.v_hist[: 3 * P]), 3)
        abi.ispa_kv_append(self.ring.c, bf16_tensor(s.k_hist[3 * P:]), bf16_tensor(s.v_hist[3 * P:]), 3)
        self.q, self.kc, self.vc = bf16_tensor(s.q), bf16_tensor(s.k_cur), bf16_tensor(s.v_cur)
        self.nq, self.D = s.q.shape[0], H * d
        mk = lambda: torch.empty(self.nq, self.D, dtype=torch.bfloat16, device="cuda")  # noqa: E731
        self.out_full, self.out_loc, self.a_full, self.a_loc = mk(), mk(), mk(), mk()
        self.disc = torch.empty(self.nq, dtype=torch.float32, device="cuda")
        self.dsum = torch.zeros(1, dtype=torch.float32, device="cuda")
        self.wsb = abi.ispa_attn_dual_workspace_size(H, self.nq)
        self.ws = torch.empty(self.wsb, dtype=torch.uint8, device="cuda")
        self.ls = LS(self.D)
        self.lwsb = abi.ispa_ls_accumulate_workspace_size(self.D, self.nq)
        self.lws = torch.empty(self.lwsb, dtype=torch.uint8, device="cuda")
        self.win = Window(0, 2)
        self.stream = torch.cuda.Stream()
        torch.cuda.synchronize()

    def run(self, rounds):
        for _ in range(rounds):
            abi.ispa_attn_full(self.ring.c, self.q, self.kc, self.vc, self.nq, 0.0, self.out_full, None, self.stream)
            abi.ispa_attn_local(self.ring.c, self.win, self.q, self.kc, self.vc, self.nq, 0.0, self.out_loc, None,
                                self.stream)
            abi.ispa_attn_dual(self.ring.c, self.win, self.q, self.kc, self.vc, self.nq, 0.0, self.a_full,
                               self.a_loc, self.disc, self.dsum, None, None, self.ws, self.wsb, self.stream)
            abi.ispa_ls_accumulate(self.ls.c, self.a_loc, self.a_full, self.nq, self.lws, self.lwsb, self.stream)
        self.stream.synchronize()

    def results(self):
        return [t.view(torch.int16).cpu().numpy() if t.dtype == torch.bfloat16 else t.cpu().numpy()
                for t in (self.out_full, self.out_loc, self.a_full, self.a_loc, self.disc, self.dsum,
                          self.ls.gram)]


def test_concurrent_threads_match_serial_calls():
    jobs = [Job(900 + i) for i in range(N_THREADS)]
    errors = []

    def work(j):
        try:
            j.run(ROUNDS)
        except Exception as e:  # noqa: BLE001 -- reported below
            errors.append(e)

    threads = [threading.Thread(target=work, args=(j,)) for j in jobs]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    assert not errors, errors
    st, code = abi.ispa_last_device_error()
    assert st == abi.ISPA_OK, code
    for i, j in enumerate(jobs):
        ref = Job(900 + i)
        ref.run(ROUNDS)
        got, want = j.results(), ref.results()
        for a, b in zip(got[:5], want[:5]):
            assert np.array_equal(a, b), i
        # sums over identical rounds: the atomics' order may differ, the values must agree
        np.testing.assert_allclose(got[5], want[5], rtol=1e-6)
        np.testing.assert_allclose(got[6], want[6], rtol=1e-5, atol=1e-3)
