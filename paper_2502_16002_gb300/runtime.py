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
        K.kvlink_reencode_concat(self.plan, pool_k.data_ptr(), pool_v.data_ptr(), cache_k.data_ptr(),
                                 cache_v.data_ptr(), _stream_handle(stream))

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
                                cache_v.data_ptr(), out.data_ptr(), self.workspace.data_ptr(),
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
        """All layers in one ABI call (sequences of per-layer tensors)."""
        ptrs = [[t.data_ptr() for t in seq] for seq in (pool_k, pool_v, q, k_new, v_new, cache_k, cache_v, out)]
        K.kvlink_linked_prefill_layers(self.plan, *ptrs, self.workspace.data_ptr(), self.workspace.numel(),
                                       _stream_handle(stream))

    def linked_prefill_layers_overlapped(self, pool_k, pool_v, q, k_new, v_new, cache_k, cache_v, out,
                                         stream=None, reencode_stream=None):
        """All layers in one ABI call, the re-encode on a second stream (created if not given)."""
        if reencode_stream is None:
            reencode_stream = self._reencode_stream()
        ptrs = [[t.data_ptr() for t in seq] for seq in (pool_k, pool_v, q, k_new, v_new, cache_k, cache_v, out)]
        K.kvlink_linked_prefill_layers_overlapped(self.plan, *ptrs, self.workspace.data_ptr(), self.workspace.numel(),
                                                  _stream_handle(stream), _stream_handle(reencode_stream))

    def _reencode_stream(self):
        if getattr(self, "_re_stream", None) is None:
            self._re_stream = torch.cuda.Stream(self.device)
        return self._re_stream

    def reencode_concat_layers(self, pool_k, pool_v, cache_k, cache_v, stream=None):
        """The document caches of all layers in one launch (sequences of per-layer tensors)."""
        ptrs = [[t.data_ptr() for t in seq] for seq in (pool_k, pool_v, cache_k, cache_v)]
        K.kvlink_reencode_concat_layers(self.plan, *ptrs, _stream_handle(stream))

    def linked_prefill_layers_from_host(self, pool_k, pool_v, h_q, h_k_new, h_v_new, q, k_new, v_new,
                                        cache_k, cache_v, out, h_out, streams=None, wait=True):
        """Every layer of the linked prefill with the fresh rows in host memory.

        The document caches of every layer are re-encoded on a fourth stream, as in
        kvlink_linked_prefill_layers_overlapped.  Per layer l: h_q[l], h_k_new[l], h_v_new[l]
        (pinned host tensors) are copied to q[l], k_new[l], v_new[l] on an input stream; the
        fresh-row placement and the suffix attention run on the compute stream once they have
        landed and layer l's caches are in place; out[l] is copied to h_out[l] (pinned) on an
        output stream once it is written.  The copies of one layer thus overlap the kernels of
        the layers around it.  Returns after the last output has arrived.

        streams: optional (input, compute, output) torch.cuda.Stream triple.
        wait=False returns once everything is enqueued, so that the host can prepare the
        next batch (e.g. rebuild_from_batch on the compute stream) while this one runs.
        Calls on the same object then chain through per-layer events: a layer's inputs are
        overwritten only after the previous call's kernels of that layer have read them, and
        its output only after the previous call's copy of it to the host.
        """
        if streams is None:
            streams = (torch.cuda.Stream(self.device), torch.cuda.current_stream(self.device),
                       torch.cuda.Stream(self.device))
        s_in, s_c, s_out = streams
        s_re = self._reencode_stream()
        n = len(pool_k)
        prev = getattr(self, "_host_chain", None)
        if prev is not None and len(prev[0]) != n:
            prev = None
        # the document caches of every layer on the re-encode stream (after the work already on
        # the compute stream, e.g. the plan upload); a layer's cache is rewritten only after the
        # previous call's attention of that layer has read it
        ev0 = torch.cuda.Event()
        ev0.record(s_c)
        s_re.wait_event(ev0)
        ev_re = []
        for l in range(n):
            if prev is not None:
                s_re.wait_event(prev[0][l])
            K.kvlink_reencode_concat(self.plan, pool_k[l].data_ptr(), pool_v[l].data_ptr(), cache_k[l].data_ptr(),
                                     cache_v[l].data_ptr(), _stream_handle(s_re))
            e = torch.cuda.Event()
            e.record(s_re)
            ev_re.append(e)
        done_c, done_o = [], []
        for l in range(n):
            ev_in = torch.cuda.Event()
            with torch.cuda.stream(s_in):
                if prev is not None:
                    s_in.wait_event(prev[0][l])      # the previous call's layer l read q, k_new, v_new
                q[l].copy_(h_q[l], non_blocking=True)
                k_new[l].copy_(h_k_new[l], non_blocking=True)
                v_new[l].copy_(h_v_new[l], non_blocking=True)
                ev_in.record(s_in)
            s_c.wait_event(ev_in)
            s_c.wait_event(ev_re[l])
            if prev is not None:
                s_c.wait_event(prev[1][l])           # the previous call's out[l] reached the host
            self.suffix_attention(q[l], k_new[l], v_new[l], cache_k[l], cache_v[l], out[l], stream=s_c)
            ev_out = torch.cuda.Event()
            ev_out.record(s_c)
            s_out.wait_event(ev_out)
            with torch.cuda.stream(s_out):
                h_out[l].copy_(out[l], non_blocking=True)
                ev_d2h = torch.cuda.Event()
                ev_d2h.record(s_out)
            done_c.append(ev_out)
            done_o.append(ev_d2h)
        self._host_chain = (done_c, done_o)
        if wait:
            s_out.synchronize()
