"""CPU oracle for the ACE MoE layer (test infrastructure only).

Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline / reference
leg may import this package. The product path (the CUDA library and its
Python binding) never imports, calls or links anything here, and nothing here
imports the product path.

Parity status of each function is stated in its module's header.
"""
from .ace_oracle import *  # noqa: F401,F403
