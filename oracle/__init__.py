"""Float64 CPU oracle of the Sparse Delta Memory hot path (test infrastructure only).

Only tests, ``__graft_entry__.smoke()`` and bench.py's CPU-baseline legs use it;
the CUDA library never does.
"""
from .sdm_oracle import *  # noqa: F401,F403
from . import sdm_oracle  # noqa: F401
