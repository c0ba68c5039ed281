"""fp64 CPU oracle for GRKV's compression path — test infrastructure only.

Only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  It shares no code with the CUDA library.
"""
from .grkv_oracle import *  # noqa: F401,F403
from .grkv_oracle import __all__  # noqa: F401
