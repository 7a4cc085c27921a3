"""GB300 microbenchmarks behind the attention kernel's design (not part of libispa).

    python -m paper_2607_00712_gb300.microbench [umma_stream] [softmax_loop] [mufu_rate]

Each benchmark is a standalone CUDA program in this directory.  It is compiled with nvcc for
sm_103a into paper_2607_00712_gb300/_build/microbench/ and run on the current GPU, and it prints
its own table:
  umma_stream   cycles per tcgen05 UMMA and MAC/clk/SM for attention issue patterns (one CTA per
                SM, one issuing thread), alone and with bulk copies, TMEM loads or MUFU loops on
                the other warps, with rotating K/V stages, and with commits between groups;
  softmax_loop  cycles per 128-element score row per warp of the softmax's inner loop (TMEM load,
                max, exp2, packed P store), 4 or 8 softmax warps, with or without a UMMA stream;
  mufu_rate     ex2.approx throughput (f32 and packed f16x2) per SM sub-partition.
No argument runs all three.  A benchmark's exit status is nonzero if one of its bounded waits
ran out or CUDA reported an error.
"""
from __future__ import annotations

import os
import subprocess
import sys

from ..build import ARCH, BUILD, CSRC, _nvcc

HERE = os.path.dirname(os.path.abspath(__file__))
NAMES = ("umma_stream", "softmax_loop", "mufu_rate")


def build(name: str) -> str:
    out_dir = os.path.join(BUILD, "microbench")
    os.makedirs(out_dir, exist_ok=True)
    src = os.path.join(HERE, name + ".cu")
    exe = os.path.join(out_dir, name)
    if not os.path.exists(exe) or os.path.getmtime(exe) < max(os.path.getmtime(src),
                                                             os.path.getmtime(os.path.join(CSRC, "ptx.cuh"))):
        cmd = [_nvcc(), *ARCH, "-O3", "-std=c++17", "-I", CSRC, src, "-o", exe]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on {src}:\n{r.stdout}\n{r.stderr}")
    return exe


def main(argv: list[str]) -> int:
    names = argv or list(NAMES)
    bad = [n for n in names if n not in NAMES]
    if bad:
        print(f"unknown benchmark(s) {bad}; choose from {NAMES}", file=sys.stderr)
        return 2
    status = 0
    for n in names:
        print(f"== {n}", flush=True)
        status |= subprocess.run([build(n)]).returncode
    return status


if __name__ == "__main__":
    sys.exit(main(sys.argv[1:]))
