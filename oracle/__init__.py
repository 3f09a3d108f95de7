"""CPU oracle for Residual Fallback Quantization (RFQ).

TEST INFRASTRUCTURE ONLY: tests/, ``__graft_entry__.smoke()`` and the CPU
baseline leg of ``bench.py`` are the only callers.  The product path never
imports this package.
"""
from .oracle import *  # noqa: F401,F403
