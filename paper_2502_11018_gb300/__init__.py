"""GB300-native draft-tree verification pass (GRIFFIN, arXiv 2502.11018).

Submodules:
  gv      ctypes binding of libgv.so (the C ABI in include/gv.h)
  step    VerifyStep: the five calls of one verify step on torch buffers
  inputs  seeded synthetic workloads (no verify arithmetic)
  build   nvcc build of libgv.so for sm_103a
The CUDA library is loaded on first use; nothing here falls back to the CPU.
"""

__all__ = ["gv", "step", "inputs", "build"]
