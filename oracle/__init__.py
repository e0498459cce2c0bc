"""fp64 CPU oracle for ISM attention.

TEST INFRASTRUCTURE ONLY: imported by ``tests/``, ``__graft_entry__.smoke()``
and the CPU-baseline / reference leg of ``bench.py``, never by the library.
"""
from .ism_oracle import *  # noqa: F401,F403
