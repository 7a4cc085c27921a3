"""fp64 CPU oracle of the ISPA hot path (arxiv 2607.00712).

TEST INFRASTRUCTURE ONLY.  This package is a plain, slow, obviously correct
restatement of what the paper computes, written from the paper and nothing
else.  Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline /
reference legs of ``bench.py`` may import it; the library
(``paper_2607_00712_gb300``) never does, and the oracle imports nothing from
the library.  The two share no code.

Modules
  keysets   -- which past frames form the local / history / full key sets
               (Eq. 7-8), the ring slot of a logical frame, and the KV-cache
               fraction accounting of Tables 1-2.
  attention -- softmax attention over a key set (Eq. 3), the dual warmup
               outputs and their discrepancy, and the LSE fusion (Eq. 9-12).
  ls        -- accumulation of the normal-equation sums, the textbook
               Cholesky solve of Eq. 5 and the feasibility score of Eq. 6.
  quant     -- e4m3 coding from the format definition, per-token / per-channel
               quantisation and the W8A8 linear layer on W + dW (Sec. 4's
               post-training quantisation).

Every function runs in float64.  Pins (what each function is checked
against, independent of itself) live in tests/test_oracle_*.py.
Parity status: every function is pinned; none is "parity unpinned".
"""
