"""CPU oracle for the block-CAT W4A4 linear layer (test infrastructure).

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline leg may import
this package.  It shares no code with the CUDA library in ``paper_2603_04359_gb300``.
Every function is pinned by the tests in ``tests/test_oracle_*.py``; none is "parity unpinned".
"""
from .cat_oracle import *  # noqa: F401,F403
