"""CPU oracle for the pruned prefill (test infrastructure only).

Imported by the test suite, ``__graft_entry__.smoke()`` and the CPU-baseline
leg of ``bench.py``; never by the CUDA library or its binding.
"""
from .zsaa_oracle import *  # noqa: F401,F403
from .zsaa_oracle import OracleConfig  # noqa: F401
