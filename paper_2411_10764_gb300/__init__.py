"""GB300-native batched candidate screening for ML^2Tuner-style autotuning.

`mlt` is the ctypes binding of the CUDA library libmlt.so (C ABI in
include/mlt.h); `workloads` draws the seeded synthetic screening workloads.
"""
from . import mlt, workloads  # noqa: F401
