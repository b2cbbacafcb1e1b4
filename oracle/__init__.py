"""Float64 CPU oracle for the eviction-by-design hot path (test infrastructure).

Only the test suite, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` use this package.  It shares no code with the CUDA library and
imports nothing from the product package.
"""
from .ebd_oracle import *  # noqa: F401,F403
