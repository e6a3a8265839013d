"""Device-side plumbing around the C ABI: torch owns the buffers, libkvlink does the work.

LinkedPrefill builds and uploads one batch's plan and holds the plan buffer and
the attention workspace; its methods are one ABI call each.
"""
from __future__ import annotations

import numpy as np
import torch

from . import kvlink as K


def bf16_from_bits(u16: np.ndarray, device=None) -> torch.Tensor:
    """bf16 tensor with the given bit patterns (uint16 numpy array)."""
    t = torch.from_numpy(np.ascontiguousarray(u16).view(np.int16)).view(torch.bfloat16)
    return t.to(device) if device is not None else t


def bits_from_bf16(t: torch.Tensor) -> np.ndarray:
    return t.detach().contiguous().cpu().view(torch.int16).numpy().view(np.uint16)


def _ptr(t):
    """Device pointer of a tensor, or None (NULL) for None."""
    return t.data_ptr() if t is not None else None


def _ptr_seqs(seqs):
    """Per-layer pointer lists; a None sequence stays None (a NULL array)."""
    return [None if seq is None else [t.data_ptr() for t in seq] for seq in seqs]


def _stream_handle(stream) -> int:
    if stream is None:
        stream = torch.cuda.current_stream()
    return int(stream.cuda_stream)


class LinkedPrefill:
    """One batch of linked-prefill queries: plan, plan buffer and workspace on a device."""

    def __init__(self, *, n_link, h_q, h_kv, head_dim, theta, pool_len, pool_start, pool_rows,
                 prefix_doc, n_docs, doc_ids, q_len, pool_block_size=0, pool_block_table=None,
                 num_sms=0, layout=K.KVLINK_LAYOUT_INTERLEAVED, device="cuda", stream=None):
        self.device = torch.device(device)
        self.plan = K.kvlink_plan_create(
            n_link=n_link, h_q=h_q, h_kv=h_kv, head_dim=head_dim, pool_len=pool_len,
            pool_start=pool_start, pool_rows=pool_rows, prefix_doc=prefix_doc, n_docs=n_docs,
            doc_ids=doc_ids, q_len=q_len, pool_block_size=pool_block_size,
            pool_block_table=pool_block_table, num_sms=num_sms, layout=layout)
        self.info = K.kvlink_plan_get_info(self.plan)
        self.theta = float(theta)
        self.plan_buf = torch.empty(max(int(self.info.device_bytes), 256), dtype=torch.uint8,
                                    device=self.device)
        self.workspace = torch.empty(max(int(self.info.workspace_bytes), 256), dtype=torch.uint8,
                                     device=self.device)
        K.kvlink_plan_upload(self.plan, self.theta, self.plan_buf.data_ptr(), self.plan_buf.numel(),
                             _stream_handle(stream))

    @classmethod
    def from_batch(cls, batch, device="cuda", num_sms=0, stream=None, layout=K.KVLINK_LAYOUT_INTERLEAVED):
        """From a workloads.Batch-like object (pool metadata and per-query tables)."""
        cfg = batch.cfg
        return cls(n_link=cfg.n_link, h_q=cfg.h_q, h_kv=cfg.h_kv, head_dim=cfg.head_dim,
                   theta=cfg.theta, pool_len=batch.pool_len, pool_start=batch.pool_start,
                   pool_rows=batch.pool_rows, prefix_doc=batch.prefix_doc, n_docs=batch.n_docs,
                   doc_ids=batch.doc_ids, q_len=batch.q_len, pool_block_size=cfg.pool_block_size,
                   pool_block_table=batch.pool_block_table, num_sms=num_sms, layout=layout,
                   device=device, stream=stream)

    def rebuild_from_batch(self, batch, num_sms=0, stream=None, layout=K.KVLINK_LAYOUT_INTERLEAVED):
        """Reuse this object for another batch: the plan is rebuilt in place (its host storage
        reused) and uploaded into the same plan buffer and workspace when they are large
        enough.  The upload is ordered after the work already enqueued on `stream`."""
        cfg = batch.cfg
        K.kvlink_plan_rebuild(self.plan, n_link=cfg.n_link, h_q=cfg.h_q, h_kv=cfg.h_kv, head_dim=cfg.head_dim,
                              pool_len=batch.pool_len, pool_start=batch.pool_start, pool_rows=batch.pool_rows,
                              prefix_doc=batch.prefix_doc, n_docs=batch.n_docs, doc_ids=batch.doc_ids,
                              q_len=batch.q_len, pool_block_size=cfg.pool_block_size,
                              pool_block_table=batch.pool_block_table, num_sms=num_sms, layout=layout)
        self.info = K.kvlink_plan_get_info(self.plan)
        self.theta = float(cfg.theta)
        if int(self.info.device_bytes) > self.plan_buf.numel():
            self.plan_buf = torch.empty(int(self.info.device_bytes), dtype=torch.uint8, device=self.device)
        if int(self.info.workspace_bytes) > self.workspace.numel():
            self.workspace = torch.empty(int(self.info.workspace_bytes), dtype=torch.uint8, device=self.device)
        K.kvlink_plan_upload(self.plan, self.theta, self.plan_buf.data_ptr(), self.plan_buf.numel(),
                             _stream_handle(stream))
        return self

    def sources(self) -> np.ndarray:
        """Per-position sources (kvlink_source_t records) of the plan."""
        return K.kvlink_plan_get_sources(self.plan)

    # shapes of the per-layer tensors
    def cache_shape(self):
        return (int(self.info.ctx_rows), int(self.info.h_kv), int(self.info.head_dim))

    def fresh_shape(self, heads):
        return (int(self.info.n_fresh), int(heads), int(self.info.head_dim))

    def empty_cache(self):
        return (torch.empty(self.cache_shape(), dtype=torch.bfloat16, device=self.device),
                torch.empty(self.cache_shape(), dtype=torch.bfloat16, device=self.device))

    # one ABI call each
    def reencode_concat(self, pool_k, pool_v, cache_k, cache_v, stream=None):
        """cache_v None: keys only (zero-copy values; pool_v is then not read)."""
        K.kvlink_reencode_concat(self.plan, pool_k.data_ptr(), _ptr(pool_v), cache_k.data_ptr(),
                                 _ptr(cache_v), _stream_handle(stream))

    def suffix_attention_pool_values(self, q, k_new, v_new, pool_v, cache_k, out, stream=None):
        """Suffix attention with zero-copy values: value rows read from pool_v and v_new
        (k_new None: the fresh keys are already in cache_k)."""
        K.kvlink_suffix_attention_pool_values(self.plan, q.data_ptr(), _ptr(k_new), v_new.data_ptr(),
                                              pool_v.data_ptr(), cache_k.data_ptr(), out.data_ptr(),
                                              self.workspace.data_ptr(), self.workspace.numel(),
                                              _stream_handle(stream))

    def suffix_attention(self, q, k_new, v_new, cache_k, cache_v, out, stream=None):
        K.kvlink_suffix_attention(self.plan, q.data_ptr(),
                                  k_new.data_ptr() if k_new is not None else None,
                                  v_new.data_ptr() if v_new is not None else None,
                                  cache_k.data_ptr(), cache_v.data_ptr(), out.data_ptr(),
                                  self.workspace.data_ptr(), self.workspace.numel(),
                                  _stream_handle(stream))

    def rope_fresh(self, q, k_new, stream=None):
        K.kvlink_rope_fresh(self.plan, q.data_ptr(), k_new.data_ptr(), _stream_handle(stream))

    def suffix_attention_simt(self, q, k_new, v_new, cache_k, cache_v, out, stream=None):
        K.kvlink_suffix_attention_simt(self.plan, q.data_ptr(),
                                       k_new.data_ptr() if k_new is not None else None,
                                       v_new.data_ptr() if v_new is not None else None,
                                       cache_k.data_ptr(), cache_v.data_ptr(), out.data_ptr(),
                                       _stream_handle(stream))

    def linked_prefill(self, pool_k, pool_v, q, k_new, v_new, cache_k, cache_v, out, stream=None):
        K.kvlink_linked_prefill(self.plan, pool_k.data_ptr(), pool_v.data_ptr(), q.data_ptr(),
                                k_new.data_ptr(), v_new.data_ptr(), cache_k.data_ptr(),
                                _ptr(cache_v), out.data_ptr(), self.workspace.data_ptr(),
                                self.workspace.numel(), _stream_handle(stream))

    def linked_prefill_fused(self, pool_k, pool_v, q, k_new, v_new, cache_k, cache_v, out, stream=None):
        """One kernel: attention over pool/fresh rows, linked cache written as a side output
        (cache_k / cache_v may be None: that half is not written)."""
        K.kvlink_linked_prefill_fused(self.plan, pool_k.data_ptr(), pool_v.data_ptr(), q.data_ptr(),
                                      k_new.data_ptr(), v_new.data_ptr(),
                                      cache_k.data_ptr() if cache_k is not None else None,
                                      cache_v.data_ptr() if cache_v is not None else None, out.data_ptr(),
                                      self.workspace.data_ptr(), self.workspace.numel(), _stream_handle(stream))

    def linked_prefill_layers(self, pool_k, pool_v, q, k_new, v_new, cache_k, cache_v, out, stream=None):
        """All layers in one ABI call (sequences of per-layer tensors; cache_v None: zero-copy values)."""
        ptrs = _ptr_seqs((pool_k, pool_v, q, k_new, v_new, cache_k, cache_v, out))
        K.kvlink_linked_prefill_layers(self.plan, *ptrs, self.workspace.data_ptr(), self.workspace.numel(),
                                       _stream_handle(stream))

    def linked_prefill_layers_overlapped(self, pool_k, pool_v, q, k_new, v_new, cache_k, cache_v, out,
                                         stream=None, reencode_stream=None):
        """All layers in one ABI call, the re-encode on a second stream (created if not given)."""
        if reencode_stream is None:
            reencode_stream = self._reencode_stream()
        ptrs = _ptr_seqs((pool_k, pool_v, q, k_new, v_new, cache_k, cache_v, out))
        K.kvlink_linked_prefill_layers_overlapped(self.plan, *ptrs, self.workspace.data_ptr(), self.workspace.numel(),
                                                  _stream_handle(stream), _stream_handle(reencode_stream))

    def _reencode_stream(self):
        if getattr(self, "_re_stream", None) is None:
            self._re_stream = torch.cuda.Stream(self.device)
        return self._re_stream

    def reencode_concat_host_pool(self, h_pool_k, h_pool_v, cache_k, cache_v, stream=None):
        """One layer's re-encode + concat with its pool in pinned host memory."""
        for t in (h_pool_k, h_pool_v):
            if not t.is_pinned():
                raise ValueError("the host pool must be pinned")
        K.kvlink_reencode_concat_host_pool(self.plan, h_pool_k.data_ptr(), h_pool_v.data_ptr(), cache_k.data_ptr(),
                                           cache_v.data_ptr(), _stream_handle(stream))

    def linked_prefill_layers_host_pool(self, h_pool_k, h_pool_v, q, k_new, v_new, cache_k, cache_v, out,
                                        stream=None, load_stream=None):
        """All layers in one ABI call with every layer's pool in pinned host memory (sequences of
        per-layer tensors); the loading and re-encode run on load_stream (created if not given)."""
        if load_stream is None:
            load_stream = self._reencode_stream()
        ptrs = [[t.data_ptr() for t in seq] for seq in (h_pool_k, h_pool_v, q, k_new, v_new, cache_k, cache_v, out)]
        K.kvlink_linked_prefill_layers_host_pool(self.plan, *ptrs, self.workspace.data_ptr(), self.workspace.numel(),
                                                 _stream_handle(stream), _stream_handle(load_stream))

    def reencode_concat_layers(self, pool_k, pool_v, cache_k, cache_v, stream=None):
        """The document caches of all layers in one launch (sequences of per-layer tensors)."""
        ptrs = _ptr_seqs((pool_k, pool_v, cache_k, cache_v))
        K.kvlink_reencode_concat_layers(self.plan, *ptrs, _stream_handle(stream))

    def linked_prefill_layers_from_host(self, pool_k, pool_v, h_q, h_k_new, h_v_new, q, k_new, v_new,
                                        cache_k, cache_v, out, h_out, streams=None, wait=True):
        """Every layer of the linked prefill with the fresh rows and outputs in host memory, in
        one kvlink_linked_prefill_layers_host call.

        h_q, h_k_new, h_v_new, h_out: pinned host tensors [L, n_fresh, heads, D]; the rest
        device tensors, one per layer (or [L, ...]).  Per layer the fresh rows are copied in on
        an input stream, the document caches re-encoded on a fourth stream, the placement and
        attention run on the compute stream, and the output is copied back on an output
        stream.  streams: optional (input, compute, output) torch.cuda.Stream triple.

        wait=False returns once everything is enqueued, so that the host can prepare the next
        batch (rebuild_from_batch on the compute stream) while this one runs; successive calls
        on this object chain through events the plan keeps.
        """
        if streams is None:
            streams = (torch.cuda.Stream(self.device), torch.cuda.current_stream(self.device),
                       torch.cuda.Stream(self.device))
        s_in, s_c, s_out = streams
        for seq in (h_q, h_k_new, h_v_new, h_out):
            if not all(t.is_pinned() for t in seq):
                raise ValueError("host tensors must be pinned")
        ptrs = _ptr_seqs((pool_k, pool_v, h_q, h_k_new, h_v_new, q, k_new, v_new, cache_k, cache_v, out, h_out))
        K.kvlink_linked_prefill_layers_host(self.plan, *ptrs, self.workspace.data_ptr(), self.workspace.numel(),
                                            _stream_handle(s_c), _stream_handle(self._reencode_stream()),
                                            _stream_handle(s_in), _stream_handle(s_out))
        if wait:
            s_out.synchronize()
