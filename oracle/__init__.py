"""CPU oracle for LazyMAR's cached decoding step (test infrastructure only).

Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline / reference
leg may import this package. The CUDA library and its Python binding never do,
and nothing here imports them.
"""
from .lazymar_oracle import *  # noqa: F401,F403
