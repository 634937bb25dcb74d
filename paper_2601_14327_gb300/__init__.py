"""GB300-native (sm_103a) MoE expert-layer hot path with LAEP expert pruning.

The compute lives in the CUDA library libmoe_laep.so (C ABI in
include/moe_laep.h); `_lib` binds it with ctypes and `layer` strings the
calls of one layer step together. Importing this package does not load the
library; the first call does, and raises if it cannot be built or loaded.
"""
__all__ = ["build", "synth"]
