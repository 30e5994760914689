"""CPU oracle for layer-wise KV-cache eviction (test infrastructure only).

Only the test suite, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline
leg may import this package.  It shares no code with the CUDA library.
"""
from .oracle import *  # noqa: F401,F403
