"""GB300 implementation of UNISON's shared live ranking (SPEAR score + TIDE
fill) and its batched trace replay (arXiv 2609.09643).

The compute path is libunison.so (include/unison.h): hand-written CUDA
kernels for sm_103a behind a C ABI.  ``binding`` is a thin ctypes layer over
it; PyTorch is used only for device memory and streams.
"""
from .native import build, LIB  # noqa: F401

__all__ = ["build", "LIB"]
