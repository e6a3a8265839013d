"""GB300 (sm_103a) KVLink linked prefill: positional re-encoding and concatenation of
precomputed document caches, and the suffix attention of link and question tokens
(arXiv 2502.16002, Sec. 2.2-2.3), behind the C ABI in include/kvlink.h.

`paper_2502_16002_gb300.kvlink` (the binding) and `.runtime` load libkvlink.so
on import and fail if it has not been built (`paper_2502_16002_gb300.build`);
there is no fallback.
"""
__all__ = ["kvlink", "runtime", "build"]
