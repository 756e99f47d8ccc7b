"""GB300-native decoder for the PIC synthesis g_r (arxiv 2609.09020).

Submodules:
  workloads -- seeded synthetic inputs shaped like the paper's decode workloads
  pic       -- ctypes binding of the C-ABI library ``libpic_gb300.so``
  build     -- compiles that library with nvcc for sm_103a

Importing the package loads nothing; ``pic`` loads the CUDA library on first
use and raises if it is missing (there is no CPU fallback).
"""
__all__ = ["workloads", "pic", "build"]
