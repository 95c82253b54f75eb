"""GB300-native Hadamard-domain INT8 convolution (HaTQ's DH/WH operator).

The compute path is libhatq.so (CUDA for sm_103a, C ABI in include/hatq.h);
`hatq` is its thin ctypes binding and `chain` sequences prepared layers by a
static DH/WH profile mask.
"""
from . import build, hatq  # noqa: F401

__all__ = ["build", "hatq", "chain"]
