"""GB300 (sm_103a) CUDA implementation of the TReVS two-stage visual-token pruning path.

The compute path lives in libtrevs.so (C ABI: include/trevs.h); `trevs` is its
thin ctypes binding. Importing this package does not load the library; the
first call does, and fails loudly if the library has not been built.
"""
from . import trevs  # noqa: F401

__all__ = ["trevs"]
