"""CPU oracle for the experience path -- TEST INFRASTRUCTURE ONLY.

Only the test-suite, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  The library path never does.

Every function here marshals numpy arrays into the plain-C oracle
(``edp_oracle.c``), except the scheduling model (``sched.py``, plain Python);
the functions that have no pin against an independent result are listed as
"parity unpinned" in their docstrings (none at present).
"""
from .oracle import *  # noqa: F401,F403
