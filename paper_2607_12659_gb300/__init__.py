"""GB300-native flow-matching denoise of a pi0.5-style action expert.

The computation lives in the CUDA library ``libjpi.so`` (C-ABI in ``include/jpi.h``, kernels in
``csrc/``); ``jpi`` is its ctypes binding. Nothing here computes on the CPU.
"""

__all__ = ["jpi", "build"]
