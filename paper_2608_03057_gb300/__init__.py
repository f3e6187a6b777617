"""GB300-native masked-W8A8 GEMM library for TASQ (arXiv 2608.03057).

The compute path is the C-ABI shared library built from csrc/ (declared in
include/tasq.h); `tasq` is its thin ctypes binding.  Importing the package does
not load the library: the first call into `tasq` does, and raises if the
library has not been built.
"""
