"""GB300 (sm_103a) implementation of LazyMAR's cached MAR decoding step.

The product is the C-ABI library liblazymar.so (include/lazymar.h, CUDA
sources in csrc/); `lazymar` is its ctypes binding and `build` compiles it.
"""
from . import build  # noqa: F401
from .lazymar import *  # noqa: F401,F403
