"""CPU oracle of TPP-SD -- test infrastructure only.

Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg may
import this package.  The CUDA library never does.
"""
from .oracle import *  # noqa: F401,F403
