"""GB300-native (sm_103a) Stream-Factorized Attention hot path for Hidden Decoding.

The compute lives in ``libhdsfa.so`` (hand-written CUDA kernels behind a C ABI,
declared in ``include/hdsfa.h``); ``binding`` is a thin ctypes layer over it.
"""
from .inputs import WITHIN, CROSS, LOCAL  # noqa: F401
