"""GB300-native (sm_103a) ACE MoE layer: token-adaptive expert skipping.

The compute path lives in the CUDA library libace.so (csrc/), reached through
the C ABI declared in include/ace.h. `paper_2609_05228_gb300.ace` is the thin
ctypes binding (argument marshalling only). Importing this package does not
load the library; the binding loads it on first use and raises if it is
missing.
"""
__all__ = ["synth", "offline", "ace"]
