"""CPU oracle for the joint evaluator: test infrastructure, not product code.

Only the test suite, ``__graft_entry__.smoke()`` and the benchmark's
CPU-baseline leg may import this package.  The CUDA path never calls it.
"""
from .fe_oracle import *  # noqa: F401,F403
