"""CPU oracle of the StepPrune inference path (test infrastructure only).

Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline leg may import
this package.  It shares no code with the CUDA library.
"""
from .stepprune_oracle import *  # noqa: F401,F403
from . import stepprune_oracle as core  # noqa: F401
