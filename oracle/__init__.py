"""CPU fp64 oracle of the CAS-Spec tree step (casspec_oracle) and of the DyTC scheduler
(dytc_oracle) -- TEST INFRASTRUCTURE ONLY.

Imported only by tests/, __graft_entry__.smoke() and bench.py's CPU baseline / reference arm.
The CUDA library never imports, links or runs anything here.
"""
from .casspec_oracle import *  # noqa: F401,F403
