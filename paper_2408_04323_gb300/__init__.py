"""GB300-native candidate-scoring path of SCOOT (arXiv 2408.04323).

The path itself lives in libscoot.so (CUDA kernels for sm_103a behind the C
ABI of include/scoot.h); `scoot` is its ctypes binding and `pipeline` chains
the calls of one suggestion round.  `build()` compiles the library in-tree.
"""
from ._build import build  # noqa: F401

__all__ = ["build"]
