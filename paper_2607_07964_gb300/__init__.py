"""GB300-native (sm_103a) implementation of KronQ's per-layer quantization path.

libkronq.so (csrc/, C ABI in include/kronq.h) holds every kernel; `kronq` is its thin
Python binding and `pipeline` runs one layer through the four stages.
"""
from . import kronq  # noqa: F401

__all__ = ["kronq"]
