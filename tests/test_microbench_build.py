"""The microbenchmarks under paper_2607_00712_gb300/microbench/ compile for sm_103a (no GPU needed;
running them needs one).  Built in parallel, each into the package's build folder."""
import os
import shutil
from concurrent.futures import ThreadPoolExecutor

import pytest


@pytest.mark.skipif(shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"),
                    reason="nvcc not available")
def test_microbenchmarks_compile():
    from paper_2607_00712_gb300.microbench.__main__ import NAMES, build
    with ThreadPoolExecutor(len(NAMES)) as ex:
        exes = list(ex.map(build, NAMES))
    assert all(os.path.exists(e) for e in exes)
