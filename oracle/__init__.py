"""CPU FP64 oracle for the AF1 binary-factorized linear layer.

Test infrastructure only: imported by tests/, __graft_entry__.smoke() and the
CPU-baseline / reference legs of bench.py, never by the product package.
"""
from .af1_oracle import *  # noqa: F401,F403
from . import af1_oracle  # noqa: F401
