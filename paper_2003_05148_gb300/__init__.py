"""GB300-native (sm_103a) hot path of Kernel Quantization (arXiv 2003.05148).

The computation lives in libkq.so (CUDA kernels behind the C ABI of
include/kq.h); ``kq`` is its thin ctypes binding and ``build`` compiles it.
"""
from . import build  # noqa: F401
