"""ISPA's hot path on one GB300: libispa (C-ABI over sm_103a CUDA kernels) and its binding.

    from paper_2607_00712_gb300 import abi          # ctypes binding, names = C entry points
    from paper_2607_00712_gb300.device import Ring   # torch-allocated ring buffers

The binding marshals arguments only; every step of the path runs in the
library's kernels (include/ispa.h documents each entry point).
"""
from . import _lib as abi  # noqa: F401
from ._lib import IspaError, KeySets, KVRing, LSState, Window  # noqa: F401

__all__ = ["abi", "IspaError", "KeySets", "KVRing", "LSState", "Window"]
