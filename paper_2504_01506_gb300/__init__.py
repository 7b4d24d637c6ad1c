"""GB300-native batched embedding key-value store (MLKV's data-parallel hot path).

The compute lives in libmlkv_gb300.so (hand-written CUDA for sm_103a, C ABI in
include/mlkv_gpu.h); this package is its thin binding.
"""
from ._lib import STALENESS_ASYNC, load  # noqa: F401
from .store import EmbeddingStore, MLKVError  # noqa: F401
