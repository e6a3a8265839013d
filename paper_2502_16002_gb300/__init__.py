"""GB300 (sm_103a) KVLink linked prefill: positional re-encoding and concatenation of
precomputed document caches, and the suffix attention of link and question tokens
(arXiv 2502.16002, Sec. 2.2-2.3), behind the C ABI in include/kvlink.h.

Importing this package loads libkvlink.so and fails if it has not been built.
"""
from . import kvlink  # noqa: F401  (loads the CUDA library; no fallback)
from .kvlink import KvlinkError  # noqa: F401

__all__ = ["kvlink", "KvlinkError"]
