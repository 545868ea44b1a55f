"""fp64 CPU oracle for the LAMB / LARS optimizer step.

TEST INFRASTRUCTURE: only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import it.  Parity of every function here
is pinned by the CPU tests in ``tests/test_oracle_pins.py``.
"""
from .lamb_oracle import *  # noqa: F401,F403
from .lamb_oracle import __all__  # noqa: F401
