"""GB300-native DistillCache budgeted KV-cache eviction decode step.

The compute path is hand-written CUDA for sm_103a behind a C ABI
(``include/distillcache.h``); this package is the thin Python binding over it.
Importing the package loads nothing: the shared library is opened on first use
and its absence is an error (there is no CPU fallback).
"""

__all__ = ["synth"]
