"""ctypes binding of libkvlink.so (include/kvlink.h), argument marshalling only.

The functions carry the C names.  Device pointers are passed as integers (e.g.
``tensor.data_ptr()``), streams as ``torch.cuda.Stream.cuda_stream`` integers.
Every step of the linked prefill runs in the library's CUDA kernels; there is no
Python or CPU fallback, and importing this module fails if the library has not
been built.
"""
from __future__ import annotations

import ctypes as C
import os

import numpy as np

# the in-tree build; KVLINK_LIBRARY may name another build of the same library
_LIB_PATH = os.environ.get("KVLINK_LIBRARY") or os.path.join(os.path.dirname(os.path.abspath(__file__)),
                                                              "libkvlink.so")

KVLINK_OK = 0
KVLINK_EINVAL = -1
KVLINK_EBOUNDS = -2
KVLINK_ECAPACITY = -3
KVLINK_EUNSUPPORTED = -4
KVLINK_ECUDA = -5
KVLINK_EDEVICE = -6

KVLINK_SEG_PREFIX, KVLINK_SEG_DOC, KVLINK_SEG_LINK, KVLINK_SEG_QUESTION = 0, 1, 2, 3
KVLINK_LAYOUT_INTERLEAVED, KVLINK_LAYOUT_LINKS_AT_END = 0, 1
KVLINK_SRC_POOL, KVLINK_SRC_FRESH = 0, 1
KVLINK_GROUP_FRESH = 1 << 30
KVLINK_STATUS_WAIT_TIMEOUT, KVLINK_STATUS_COPY_TIMEOUT = 0x41, 0x21
KVLINK_STATUS_BAD_INDEX_ATTN, KVLINK_STATUS_BAD_INDEX_COPY = 0x42, 0x22


class kvlink_batch_desc_t(C.Structure):
    _fields_ = [
        ("batch", C.c_int32), ("n_link", C.c_int32), ("h_q", C.c_int32), ("h_kv", C.c_int32),
        ("head_dim", C.c_int32),
        ("pool_docs", C.c_int32),
        ("pool_len", C.POINTER(C.c_int32)),
        ("pool_start", C.POINTER(C.c_int64)),
        ("pool_rows", C.c_int64),
        ("pool_block_size", C.c_int32),
        ("pool_block_table", C.POINTER(C.c_int32)),
        ("pool_block_table_len", C.c_int64),
        ("prefix_doc", C.POINTER(C.c_int32)),
        ("n_docs", C.POINTER(C.c_int32)),
        ("doc_ids", C.POINTER(C.c_int32)),
        ("q_len", C.POINTER(C.c_int32)),
        ("num_sms", C.c_int32),
        ("layout", C.c_int32),
    ]


class kvlink_segment_t(C.Structure):
    _fields_ = [
        ("query", C.c_int32), ("kind", C.c_int32), ("src", C.c_int32), ("len", C.c_int32),
        ("dst", C.c_int64), ("pos", C.c_int32), ("table", C.c_int32),
    ]


SEGMENT_DTYPE = np.dtype([("query", "<i4"), ("kind", "<i4"), ("src", "<i4"), ("len", "<i4"),
                          ("dst", "<i8"), ("pos", "<i4"), ("table", "<i4")])
SOURCE_DTYPE = np.dtype([("kind", "<i4"), ("row", "<i4"), ("slot", "<i4"), ("table", "<i4")])


class kvlink_plan_info_t(C.Structure):
    _fields_ = [
        ("batch", C.c_int32), ("h_q", C.c_int32), ("h_kv", C.c_int32), ("head_dim", C.c_int32),
        ("n_link", C.c_int32),
        ("n_segments", C.c_int32), ("n_rope_rows", C.c_int32), ("n_fresh", C.c_int32),
        ("ctx_rows", C.c_int64), ("cached_tokens", C.c_int64),
        ("n_copy_chunks", C.c_int32), ("n_attn_items", C.c_int32), ("n_attn_splits", C.c_int32),
        ("num_sms", C.c_int32),
        ("device_bytes", C.c_size_t), ("workspace_bytes", C.c_size_t),
        ("attn_pairs", C.c_int64), ("n_attn_ctas", C.c_int32),
    ]


def _load():
    if not os.path.exists(_LIB_PATH):
        raise ImportError(f"{_LIB_PATH} is missing: build it with __graft_entry__.build() "
                          "(the linked prefill has no fallback)")
    lib = C.CDLL(_LIB_PATH)
    P, V = C.c_void_p, C.c_void_p
    sig = {
        "kvlink_version": (C.c_int, []),
        "kvlink_strerror": (C.c_char_p, [C.c_int]),
        "kvlink_last_cuda_error": (C.c_char_p, []),
        "kvlink_plan_create": (C.c_int, [C.POINTER(kvlink_batch_desc_t), C.POINTER(P)]),
        "kvlink_plan_destroy": (None, [P]),
        "kvlink_plan_get_info": (C.c_int, [P, C.POINTER(kvlink_plan_info_t)]),
        "kvlink_plan_get_segments": (C.c_int, [P, V, C.c_int32]),
        "kvlink_plan_get_offsets": (C.c_int, [P, V, V]),
        "kvlink_plan_get_fresh_positions": (C.c_int, [P, V, C.c_int32]),
        "kvlink_plan_get_sources": (C.c_int, [P, V, C.c_int64]),
        "kvlink_plan_get_attention_items": (C.c_int, [P, V, C.c_int32]),
        "kvlink_plan_get_value_groups": (C.c_int, [P, V, V, C.c_int64]),
        "kvlink_plan_upload": (C.c_int, [P, C.c_double, V, C.c_size_t, V]),
        "kvlink_reencode_concat": (C.c_int, [P, V, V, V, V, V]),
        "kvlink_suffix_attention": (C.c_int, [P, V, V, V, V, V, V, V, C.c_size_t, V]),
        "kvlink_suffix_attention_pool_values": (C.c_int, [P, V, V, V, V, V, V, V, C.c_size_t, V]),
        "kvlink_suffix_attention_simt": (C.c_int, [P, V, V, V, V, V, V, V]),
        "kvlink_suffix_attention_noalloc": (C.c_int, [P, V, V, V, V, V, V, V]),
        "kvlink_rope_fresh": (C.c_int, [P, V, V, V]),
        "kvlink_linked_prefill": (C.c_int, [P, V, V, V, V, V, V, V, V, V, C.c_size_t, V]),
        "kvlink_linked_prefill_fused": (C.c_int, [P, V, V, V, V, V, V, V, V, V, C.c_size_t, V]),
        "kvlink_linked_prefill_layers": (C.c_int, [P, C.c_int32, V, V, V, V, V, V, V, V, V, C.c_size_t, V]),
        "kvlink_reencode_concat_layers": (C.c_int, [P, C.c_int32, V, V, V, V, V]),
        "kvlink_plan_rebuild": (C.c_int, [P, C.POINTER(kvlink_batch_desc_t)]),
        "kvlink_linked_prefill_layers_overlapped": (C.c_int, [P, C.c_int32, V, V, V, V, V, V, V, V, V, C.c_size_t,
                                                              V, V]),
        "kvlink_linked_prefill_layers_host": (C.c_int, [P, C.c_int32] + [V] * 13 + [C.c_size_t, V, V, V, V]),
        "kvlink_reencode_concat_host_pool": (C.c_int, [P, V, V, V, V, V]),
        "kvlink_linked_prefill_layers_host_pool": (C.c_int, [P, C.c_int32] + [V] * 9 + [C.c_size_t, V, V]),
        "kvlink_device_status": (C.c_int, [C.POINTER(C.c_int32)]),
        "kvlink_clear_device_status": (C.c_int, []),
        "kvlink_selftest_wait_timeout": (C.c_int, [C.c_uint32, V]),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    return lib


lib = _load()

DECLARED = [
    "kvlink_plan_create", "kvlink_plan_destroy", "kvlink_plan_get_info", "kvlink_plan_get_segments",
    "kvlink_plan_get_offsets", "kvlink_plan_get_fresh_positions", "kvlink_plan_upload",
    "kvlink_reencode_concat", "kvlink_suffix_attention", "kvlink_suffix_attention_simt",
    "kvlink_linked_prefill",
    "kvlink_device_status", "kvlink_clear_device_status", "kvlink_strerror",
    "kvlink_last_cuda_error", "kvlink_version", "kvlink_suffix_attention_noalloc", "kvlink_rope_fresh",
    "kvlink_plan_get_sources", "kvlink_linked_prefill_fused", "kvlink_linked_prefill_layers",
    "kvlink_reencode_concat_layers", "kvlink_plan_rebuild", "kvlink_linked_prefill_layers_overlapped",
    "kvlink_linked_prefill_layers_host", "kvlink_reencode_concat_host_pool", "kvlink_linked_prefill_layers_host_pool",
    "kvlink_selftest_wait_timeout", "kvlink_suffix_attention_pool_values", "kvlink_plan_get_attention_items",
    "kvlink_plan_get_value_groups",
]

# size of the static scratch used by kvlink_suffix_attention_noalloc (include/kvlink.h)
KVLINK_NOALLOC_MAX_WORKSPACE_BYTES = 8 << 20


class KvlinkError(RuntimeError):
    def __init__(self, code: int, where: str):
        msg = lib.kvlink_strerror(code).decode()
        if code == KVLINK_ECUDA:
            msg += ": " + lib.kvlink_last_cuda_error().decode()
        super().__init__(f"{where}: {msg} ({code})")
        self.code = code


def _check(code: int, where: str) -> None:
    if code != KVLINK_OK:
        raise KvlinkError(code, where)


def _i32(a):
    return np.ascontiguousarray(np.asarray(a, dtype=np.int32))


def _i64(a):
    return np.ascontiguousarray(np.asarray(a, dtype=np.int64))


def _ptr(a, ctype):
    return a.ctypes.data_as(C.POINTER(ctype))


class Plan:
    """Owns a kvlink_plan_t handle (kvlink_plan_destroy on close)."""

    def __init__(self, handle):
        self.handle = handle

    def close(self):
        if self.handle:
            lib.kvlink_plan_destroy(self.handle)
            self.handle = None

    def __del__(self):
        self.close()


def _batch_desc(n_link, h_q, h_kv, head_dim, pool_len, pool_start, pool_rows, prefix_doc, n_docs, doc_ids,
                q_len, pool_block_size, pool_block_table, num_sms, layout):
    """A kvlink_batch_desc_t and the arrays it points into (kept alive by the caller)."""
    arrs = dict(pool_len=_i32(pool_len), pool_start=_i64(pool_start), prefix_doc=_i32(prefix_doc),
                n_docs=_i32(n_docs), doc_ids=_i32(doc_ids), q_len=_i32(q_len))
    bt = _i32(pool_block_table) if pool_block_table is not None else None
    d = kvlink_batch_desc_t()
    d.batch = len(arrs["n_docs"])
    d.n_link, d.h_q, d.h_kv, d.head_dim = int(n_link), int(h_q), int(h_kv), int(head_dim)
    d.pool_docs = len(arrs["pool_len"])
    d.pool_len = _ptr(arrs["pool_len"], C.c_int32)
    d.pool_start = _ptr(arrs["pool_start"], C.c_int64)
    d.pool_rows = int(pool_rows)
    d.pool_block_size = int(pool_block_size)
    d.pool_block_table = _ptr(bt, C.c_int32) if bt is not None else None
    d.pool_block_table_len = len(bt) if bt is not None else 0
    d.prefix_doc = _ptr(arrs["prefix_doc"], C.c_int32)
    d.n_docs = _ptr(arrs["n_docs"], C.c_int32)
    d.doc_ids = _ptr(arrs["doc_ids"], C.c_int32) if len(arrs["doc_ids"]) else None
    d.q_len = _ptr(arrs["q_len"], C.c_int32)
    d.num_sms = int(num_sms)
    d.layout = int(layout)
    return d, (arrs, bt)


def kvlink_plan_create(*, n_link, h_q, h_kv, head_dim, pool_len, pool_start, pool_rows,
                       prefix_doc, n_docs, doc_ids, q_len, pool_block_size=0,
                       pool_block_table=None, num_sms=0, layout=KVLINK_LAYOUT_INTERLEAVED) -> Plan:
    d, keep = _batch_desc(n_link, h_q, h_kv, head_dim, pool_len, pool_start, pool_rows, prefix_doc, n_docs,
                          doc_ids, q_len, pool_block_size, pool_block_table, num_sms, layout)
    h = C.c_void_p()
    _check(lib.kvlink_plan_create(C.byref(d), C.byref(h)), "kvlink_plan_create")
    return Plan(h)


def kvlink_plan_rebuild(plan: Plan, *, n_link, h_q, h_kv, head_dim, pool_len, pool_start, pool_rows,
                        prefix_doc, n_docs, doc_ids, q_len, pool_block_size=0,
                        pool_block_table=None, num_sms=0, layout=KVLINK_LAYOUT_INTERLEAVED) -> None:
    d, keep = _batch_desc(n_link, h_q, h_kv, head_dim, pool_len, pool_start, pool_rows, prefix_doc, n_docs,
                          doc_ids, q_len, pool_block_size, pool_block_table, num_sms, layout)
    _check(lib.kvlink_plan_rebuild(plan.handle, C.byref(d)), "kvlink_plan_rebuild")


def kvlink_plan_get_info(plan: Plan) -> kvlink_plan_info_t:
    info = kvlink_plan_info_t()
    _check(lib.kvlink_plan_get_info(plan.handle, C.byref(info)), "kvlink_plan_get_info")
    return info


def kvlink_plan_get_segments(plan: Plan) -> np.ndarray:
    n = kvlink_plan_get_info(plan).n_segments
    out = np.zeros(n, dtype=SEGMENT_DTYPE)
    _check(lib.kvlink_plan_get_segments(plan.handle, out.ctypes.data, n), "kvlink_plan_get_segments")
    return out


def kvlink_plan_get_offsets(plan: Plan):
    B = kvlink_plan_get_info(plan).batch
    cu_ctx = np.zeros(B + 1, np.int64)
    cu_fresh = np.zeros(B + 1, np.int32)
    _check(lib.kvlink_plan_get_offsets(plan.handle, cu_ctx.ctypes.data, cu_fresh.ctypes.data),
           "kvlink_plan_get_offsets")
    return cu_ctx, cu_fresh


def kvlink_plan_get_fresh_positions(plan: Plan) -> np.ndarray:
    n = kvlink_plan_get_info(plan).n_fresh
    out = np.zeros(n, np.int32)
    _check(lib.kvlink_plan_get_fresh_positions(plan.handle, out.ctypes.data, n),
           "kvlink_plan_get_fresh_positions")
    return out


def kvlink_plan_get_sources(plan: Plan) -> np.ndarray:
    n = kvlink_plan_get_info(plan).ctx_rows
    out = np.zeros(n, dtype=SOURCE_DTYPE)
    _check(lib.kvlink_plan_get_sources(plan.handle, out.ctypes.data, n), "kvlink_plan_get_sources")
    return out


ATTN_ITEM_DTYPE = np.dtype([(n, np.int32) for n in ("query", "kv_head", "tok0", "tok1", "entry0", "entry1",
                                                      "a_tiles", "b_tile0", "slot", "cta")])


def kvlink_plan_get_attention_items(plan: Plan) -> np.ndarray:
    """The persistent attention's work items in run order, with the CTA of each."""
    n = int(kvlink_plan_get_info(plan).n_attn_items)
    out = np.zeros(n, ATTN_ITEM_DTYPE)
    _check(lib.kvlink_plan_get_attention_items(plan.handle, out.ctypes.data, n), "kvlink_plan_get_attention_items")
    return out


def kvlink_plan_get_value_groups(plan: Plan):
    """(grp, cu_grp): the 8-row value groups of every query (entry m of query b at
    cu_grp[b] + m: first source row, with KVLINK_GROUP_FRESH for fresh rows, or -1)."""
    cu_ctx, _ = kvlink_plan_get_offsets(plan)
    n = int(np.sum((np.diff(cu_ctx) + 7) // 8))
    grp = np.zeros(n, np.int32)
    cu = np.zeros(len(cu_ctx), np.int32)
    _check(lib.kvlink_plan_get_value_groups(plan.handle, grp.ctypes.data, cu.ctypes.data, n),
           "kvlink_plan_get_value_groups")
    return grp, cu


def kvlink_plan_upload(plan: Plan, theta: float, d_buf: int, nbytes: int, stream: int = 0) -> None:
    _check(lib.kvlink_plan_upload(plan.handle, float(theta), d_buf, nbytes, stream), "kvlink_plan_upload")


def kvlink_reencode_concat(plan: Plan, pool_k: int, pool_v: int, cache_k: int, cache_v: int,
                           stream: int = 0) -> None:
    _check(lib.kvlink_reencode_concat(plan.handle, pool_k, pool_v, cache_k, cache_v, stream),
           "kvlink_reencode_concat")


def kvlink_suffix_attention(plan: Plan, q: int, k_new, v_new, cache_k: int, cache_v: int, out: int,
                            workspace, workspace_bytes: int, stream: int = 0) -> None:
    _check(lib.kvlink_suffix_attention(plan.handle, q, k_new, v_new, cache_k, cache_v, out, workspace,
                                       workspace_bytes, stream), "kvlink_suffix_attention")


def kvlink_suffix_attention_pool_values(plan: Plan, q: int, k_new, v_new: int, pool_v: int, cache_k: int, out: int,
                                        workspace, workspace_bytes: int, stream: int = 0) -> None:
    """Suffix attention with zero-copy values: value rows read from pool_v and v_new."""
    _check(lib.kvlink_suffix_attention_pool_values(plan.handle, q, k_new, v_new, pool_v, cache_k, out, workspace,
                                                   workspace_bytes, stream), "kvlink_suffix_attention_pool_values")


def kvlink_suffix_attention_simt(plan: Plan, q: int, k_new, v_new, cache_k: int, cache_v: int, out: int,
                                 stream: int = 0) -> None:
    _check(lib.kvlink_suffix_attention_simt(plan.handle, q, k_new, v_new, cache_k, cache_v, out, stream),
           "kvlink_suffix_attention_simt")


def kvlink_suffix_attention_noalloc(plan: Plan, q: int, k_new, v_new, cache_k: int, cache_v: int, out: int,
                                    stream: int = 0) -> None:
    """Suffix attention without a caller workspace: the split-KV scratch is the library's
    static device array (see include/kvlink.h); it allocates nothing."""
    _check(lib.kvlink_suffix_attention_noalloc(plan.handle, q, k_new, v_new, cache_k, cache_v, out, stream),
           "kvlink_suffix_attention_noalloc")


def kvlink_rope_fresh(plan: Plan, q: int, k_new: int, stream: int = 0) -> None:
    _check(lib.kvlink_rope_fresh(plan.handle, q, k_new, stream), "kvlink_rope_fresh")


def kvlink_linked_prefill(plan: Plan, pool_k: int, pool_v: int, q: int, k_new: int, v_new: int,
                          cache_k: int, cache_v: int, out: int, workspace, workspace_bytes: int,
                          stream: int = 0) -> None:
    _check(lib.kvlink_linked_prefill(plan.handle, pool_k, pool_v, q, k_new, v_new, cache_k, cache_v, out,
                                     workspace, workspace_bytes, stream), "kvlink_linked_prefill")


def kvlink_linked_prefill_fused(plan: Plan, pool_k: int, pool_v: int, q: int, k_new: int, v_new: int,
                                cache_k, cache_v, out: int, workspace, workspace_bytes: int,
                                stream: int = 0) -> None:
    _check(lib.kvlink_linked_prefill_fused(plan.handle, pool_k, pool_v, q, k_new, v_new, cache_k, cache_v, out,
                                           workspace, workspace_bytes, stream), "kvlink_linked_prefill_fused")


def _ptr_array(ptrs):
    arr = (C.c_void_p * len(ptrs))(*[int(x) for x in ptrs])
    return arr


def _ptr_arrays(n, seqs, optional=()):
    """HOST arrays of per-layer pointers; a sequence at an index in `optional` may be None
    (passed as a NULL array: e.g. cache_v for zero-copy values)."""
    out = []
    for i, x in enumerate(seqs):
        if x is None and i in optional:
            out.append(None)
            continue
        a = _ptr_array(x)
        if len(a) != n:
            raise ValueError("every per-layer pointer list needs one entry per layer")
        out.append(C.cast(a, C.c_void_p))
    return out


def kvlink_linked_prefill_layers(plan: Plan, pool_k, pool_v, q, k_new, v_new, cache_k, cache_v, out,
                                 workspace, workspace_bytes: int, stream: int = 0) -> None:
    """Every argument but the plan, workspace and stream: a sequence of per-layer device pointers."""
    n = len(pool_k)
    arrs = _ptr_arrays(n, (pool_k, pool_v, q, k_new, v_new, cache_k, cache_v, out), optional=(6,))
    _check(lib.kvlink_linked_prefill_layers(plan.handle, n, *arrs, workspace, workspace_bytes, stream),
           "kvlink_linked_prefill_layers")


def kvlink_linked_prefill_layers_overlapped(plan: Plan, pool_k, pool_v, q, k_new, v_new, cache_k, cache_v, out,
                                            workspace, workspace_bytes: int, stream: int, reencode_stream: int) -> None:
    """As kvlink_linked_prefill_layers, with the re-encode on reencode_stream."""
    n = len(pool_k)
    arrs = _ptr_arrays(n, (pool_k, pool_v, q, k_new, v_new, cache_k, cache_v, out), optional=(6,))
    _check(lib.kvlink_linked_prefill_layers_overlapped(plan.handle, n, *arrs, workspace, workspace_bytes, stream,
                                                       reencode_stream),
           "kvlink_linked_prefill_layers_overlapped")


def kvlink_linked_prefill_layers_host(plan: Plan, pool_k, pool_v, h_q, h_k_new, h_v_new, q, k_new, v_new, cache_k,
                                      cache_v, out, h_out, workspace, workspace_bytes: int, stream: int,
                                      reencode_stream: int, copy_in_stream: int, copy_out_stream: int) -> None:
    """Per-layer pointer sequences (h_*: host, the rest device); see include/kvlink.h."""
    n = len(pool_k)
    seqs = (pool_k, pool_v, h_q, h_k_new, h_v_new, q, k_new, v_new, cache_k, cache_v, out, h_out)
    arrs = _ptr_arrays(n, seqs, optional=(9,))
    _check(lib.kvlink_linked_prefill_layers_host(plan.handle, n, *arrs, workspace,
                                                 workspace_bytes, stream, reencode_stream, copy_in_stream,
                                                 copy_out_stream), "kvlink_linked_prefill_layers_host")


def kvlink_reencode_concat_host_pool(plan: Plan, h_pool_k: int, h_pool_v: int, cache_k: int, cache_v: int,
                                     stream: int = 0) -> None:
    """h_pool_k / h_pool_v: page-locked host memory; cache_k / cache_v: device memory."""
    _check(lib.kvlink_reencode_concat_host_pool(plan.handle, h_pool_k, h_pool_v, cache_k, cache_v, stream),
           "kvlink_reencode_concat_host_pool")


def kvlink_linked_prefill_layers_host_pool(plan: Plan, h_pool_k, h_pool_v, q, k_new, v_new, cache_k, cache_v, out,
                                           workspace, workspace_bytes: int, stream: int, load_stream: int) -> None:
    """Per-layer pointer sequences: h_pool_*: page-locked host memory, the rest device memory."""
    n = len(h_pool_k)
    arrs = [_ptr_array(x) for x in (h_pool_k, h_pool_v, q, k_new, v_new, cache_k, cache_v, out)]
    if any(len(a) != n for a in arrs):
        raise ValueError("every per-layer pointer list needs one entry per layer")
    _check(lib.kvlink_linked_prefill_layers_host_pool(plan.handle, n, *[C.cast(a, C.c_void_p) for a in arrs],
                                                      workspace, workspace_bytes, stream, load_stream),
           "kvlink_linked_prefill_layers_host_pool")


def kvlink_reencode_concat_layers(plan: Plan, pool_k, pool_v, cache_k, cache_v, stream: int = 0) -> None:
    """Every argument but the plan and stream: a sequence of per-layer device pointers."""
    n = len(pool_k)
    arrs = _ptr_arrays(n, (pool_k, pool_v, cache_k, cache_v), optional=(1, 3))
    _check(lib.kvlink_reencode_concat_layers(plan.handle, n, *arrs, stream),
           "kvlink_reencode_concat_layers")


def kvlink_device_status() -> int:
    s = C.c_int32(0)
    _check(lib.kvlink_device_status(C.byref(s)), "kvlink_device_status")
    return int(s.value)


def kvlink_clear_device_status() -> None:
    _check(lib.kvlink_clear_device_status(), "kvlink_clear_device_status")


def kvlink_selftest_wait_timeout(limit_ms: int, stream: int = 0) -> None:
    _check(lib.kvlink_selftest_wait_timeout(int(limit_ms), stream), "kvlink_selftest_wait_timeout")
