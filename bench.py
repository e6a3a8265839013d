#!/usr/bin/env python3
"""Linked-prefill benchmark (KVLink, arXiv 2502.16002) on GB300.

One step = the whole linked prefill of one batch, over every layer, through
kvlink_linked_prefill_layers_overlapped: the retrieved documents' cached K/V of every
layer re-encoded + concatenated on a second stream, and per layer, once its caches are
in place, the fresh link/question K/V placed and the suffix attention run.

Default workload: Llama-3.1-8B shape (32 layers, 32 query / 8 KV heads, head dim
128), batch 8, each query 20 of 200 pooled 256-token documents drawn by Zipf(1.1),
5 link tokens per document, 32-token prefix, 64 question tokens (5316 context
tokens per query).  Inputs are synthetic N(0,1) bf16, resident in HBM; every layer
has its own pool, cache and fresh tensors, so each step streams well over L2.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--config 3] [--impl ours|reference]
                  [--path two-kernel|two-kernel-serial|one-kernel|one-kernel-k-only] [--layout interleaved|links_at_end]

--path selects the library entry point: kvlink_linked_prefill_layers_overlapped (the
default, above), two-kernel-serial (kvlink_linked_prefill_layers: per layer one launch
that re-encodes and places the fresh rows, then the attention, on one stream), or
kvlink_linked_prefill_fused per layer (one kernel per layer; -k-only leaves the values
in the pool).
--layout selects the physical order of the linked cache.

Prints one JSON line (rank 0).  --impl reference times the fp64 CPU oracle on the
host cores on a bounded sample of the same workload.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import workloads as W  # noqa: E402
from paper_2502_16002_gb300.clocks import ClockSampler  # noqa: E402

METRIC = "linked-prefill us/query (all layers, 8B-shape)"
UNIT = "us/query"

# dram__bytes_read.sum + dram__bytes_write.sum per launch, from one ncu capture of the
# kernel on the workload, keyed by (kernel, workload).  Each figure carries the hash of the
# sources that built the captured kernel (and planned its launch): when they change, the
# figure no longer describes the kernel being timed and the line reports traffic null.
KERNEL_SOURCES = {
    "attention": ["kvlink_attention_tc.cu", "kvlink_attention_common.cuh", "kvlink_sm100.cuh",
                  "kvlink_internal.h", "kvlink_plan.cpp"],
    "reencode": ["kvlink_reencode.cu", "kvlink_rope.cuh", "kvlink_sm100.cuh", "kvlink_internal.h",
                 "kvlink_plan.cpp"],
}
# Captures: `ncu --set full` of one launch per kernel, on runs of this script with one or two
# layers (each launch does a layer's full work); the zero-copy kernels on workload 3 only.
NCU_TRAFFIC = {
    ("attention", 3): (237_865_728 + 7_885_824, "cee90bd7320fd08e"),
    ("attention", 4): (264_504_832 + 6_526_976, "cee90bd7320fd08e"),
    ("attention", 5): (873_054_720 + 56_700_672, "cee90bd7320fd08e"),
    ("reencode", 3): (102_522_112 + 113_229_568, "a171595bc7e10bc7"),
    ("attention_pool_values", 3): (174_782_720 + 6_285_056, "cee90bd7320fd08e"),
    ("reencode_keys", 3): (40_695_552 + 25_574_400, "a171595bc7e10bc7"),
}
KERNEL_SOURCES["attention_pool_values"] = KERNEL_SOURCES["attention"]
KERNEL_SOURCES["reencode_keys"] = KERNEL_SOURCES["reencode"]


def source_hash(kernel: str) -> str:
    """sha256 (first 16 hex digits) over the sources of one kernel."""
    import hashlib
    h = hashlib.sha256()
    for f in KERNEL_SOURCES[kernel]:
        with open(os.path.join(ROOT, "paper_2502_16002_gb300", "csrc", f), "rb") as fh:
            h.update(f.encode() + b"\0" + fh.read())
    return h.hexdigest()[:16]


def ncu_traffic(kernel: str, workload: int):
    """Measured DRAM bytes per launch when the capture matches the current sources, else None."""
    rec = NCU_TRAFFIC.get((kernel, workload))
    return rec[0] if rec and rec[1] == source_hash(kernel) else None


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as fh:
            d = json.load(fh)
        return {"hbm_gbs": float(d["hbm_gbs"]), "bf16_tflops": float(d["bf16_tflops"]),
                "bf16_tflops_sustained": float(d.get("bf16_tflops_sustained", d["bf16_tflops"])),
                "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
            "source": "fallback"}


def _cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


# ------------------------------------------------------------------ algorithmic counts

def algorithmic_counts(batch, info):
    """Bytes and flops one layer's kernels must move / compute (per launch)."""
    cfg = batch.cfg
    row_bytes = cfg.h_kv * cfg.head_dim * 2            # one token's K (or V) of one layer
    cached = int(info.cached_tokens)
    # unique pool tokens read (documents repeated across the batch are read once)
    used = set(int(d) for d in batch.doc_ids)
    used |= set(int(p) for p in batch.prefix_doc if p >= 0)
    unique_tokens = int(sum(int(batch.pool_len[d]) for d in used))
    fresh = int(info.n_fresh)
    # kvlink_reencode_concat: read each used pool token's K and V once, write K and V of
    # every cached slot (prefix + documents) of the linked cache
    reencode_bytes = 2 * row_bytes * unique_tokens + 2 * row_bytes * cached
    reencode_bytes_naive = 2 * row_bytes * 2 * cached
    attn_flops = 4 * cfg.h_q * cfg.head_dim * int(info.attn_pairs)
    attn_bytes = 2 * row_bytes * int(info.ctx_rows) + 2 * fresh * cfg.h_q * cfg.head_dim * 2
    return dict(reencode_bytes=reencode_bytes, reencode_bytes_naive=reencode_bytes_naive,
                attn_flops=attn_flops, attn_bytes=attn_bytes, unique_pool_tokens=unique_tokens)


# ------------------------------------------------------------------ multi-rank bookkeeping

def max_over_ranks(x: float, world: int, device=None) -> float:
    """The largest value of x over all ranks (timing only: no data-path collective)."""
    if world == 1:
        return float(x)
    import torch
    import torch.distributed as dist

    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_us_per_query(ms_per_step: float, batch_per_rank: int, world: int) -> float:
    """Every rank serves its own batch in parallel: queries of all ranks over the slowest rank's time."""
    return ms_per_step * 1e3 / (batch_per_rank * world)


def rank_batch_seed(rank: int) -> int:
    """Each rank draws an independent batch (weak scaling: fixed work per GPU)."""
    return rank


# ------------------------------------------------------------------ our arm

class Workload:
    """One workload resident on the device: its plan, every layer's pool, fresh rows, linked
    cache and output, and the library calls of one step."""

    def __init__(self, args, cfg_index, rank, dev):
        import torch

        from paper_2502_16002_gb300 import kvlink as K
        from paper_2502_16002_gb300.runtime import LinkedPrefill

        self.K = K
        self.dev = dev
        self.cfg = cfg = W.get_config(cfg_index)
        self.batch = W.draw_batch(cfg, seed=rank_batch_seed(rank))   # every rank serves its own batch
        self.L = L = args.layers or cfg.layers
        self.path, self.layout = args.path, args.layout
        layout = {"interleaved": K.KVLINK_LAYOUT_INTERLEAVED, "links_at_end": K.KVLINK_LAYOUT_LINKS_AT_END}
        self.lp = LinkedPrefill.from_batch(self.batch, device=dev, layout=layout[args.layout])
        self.info = info = self.lp.info
        ctx, T = int(info.ctx_rows), int(info.n_fresh)
        H, Hq, D = cfg.h_kv, cfg.h_q, cfg.head_dim
        pool_shape = ((self.batch.pool_rows // cfg.pool_block_size, cfg.pool_block_size, H, D)
                      if cfg.pool_block_size else (self.batch.pool_rows, H, D))
        base = 1_000_000 * (rank + 1) + 100_000 * cfg_index
        self.pool_k = [W.normal_bf16_torch(pool_shape, base + 10 * l + 1, dev) for l in range(L)]
        self.pool_v = [W.normal_bf16_torch(pool_shape, base + 10 * l + 2, dev) for l in range(L)]
        self.q = W.normal_bf16_torch((L, T, Hq, D), base + 3, dev)
        self.kn = W.normal_bf16_torch((L, T, H, D), base + 4, dev)
        self.vn = W.normal_bf16_torch((L, T, H, D), base + 5, dev)
        self.ck = torch.empty((L, ctx, H, D), dtype=torch.bfloat16, device=dev)
        self.cv = torch.empty_like(self.ck)
        self.out = torch.empty((L, T, Hq, D), dtype=torch.bfloat16, device=dev)
        self.stream = torch.cuda.current_stream(dev)
        self.sh = int(self.stream.cuda_stream)
        self.ws, self.wsb = self.lp.workspace.data_ptr(), self.lp.workspace.numel()
        self.plan = self.lp.plan
        self.one_kernel = args.path.startswith("one-kernel")
        self.ptrs = [[t.data_ptr() for t in seq]
                     for seq in (self.pool_k, self.pool_v, self.q, self.kn, self.vn, self.ck, self.cv, self.out)]
        self.re_stream = torch.cuda.Stream(dev)
        self.re_sh = int(self.re_stream.cuda_stream)
        self.layer_ptrs = [[t.data_ptr() for t in seq] for seq in (self.pool_k, self.pool_v, self.ck, self.cv)]

    def layer_call(self, l):
        K = self.K
        if self.one_kernel:
            K.kvlink_linked_prefill_fused(self.plan, self.pool_k[l].data_ptr(), self.pool_v[l].data_ptr(),
                                          self.q[l].data_ptr(), self.kn[l].data_ptr(), self.vn[l].data_ptr(),
                                          self.ck[l].data_ptr(),
                                          None if self.path == "one-kernel-k-only" else self.cv[l].data_ptr(),
                                          self.out[l].data_ptr(), self.ws, self.wsb, self.sh)
        else:
            K.kvlink_linked_prefill(self.plan, self.pool_k[l].data_ptr(), self.pool_v[l].data_ptr(),
                                    self.q[l].data_ptr(), self.kn[l].data_ptr(), self.vn[l].data_ptr(),
                                    self.ck[l].data_ptr(), self.cv[l].data_ptr(), self.out[l].data_ptr(),
                                    self.ws, self.wsb, self.sh)

    def step(self):
        K = self.K
        if self.one_kernel:
            for l in range(self.L):
                self.layer_call(l)
        elif self.path == "two-kernel-serial":
            K.kvlink_linked_prefill_layers(self.plan, *self.ptrs, self.ws, self.wsb, self.sh)
        else:
            K.kvlink_linked_prefill_layers_overlapped(self.plan, *self.ptrs, self.ws, self.wsb, self.sh, self.re_sh)

    def launches_per_step(self):
        # the persistent attention merges cut KV ranges itself; the one-kernel path needs the
        # merge kernel after it
        n_merge = 1 if self.one_kernel and self.info.n_attn_splits > 0 else 0
        per_layer = 1 if self.one_kernel else 2 if self.path == "two-kernel-serial" else 3
        return self.L * (per_layer + n_merge)

    def timed_steps(self, n, world, clock_ms, local_rank, step=None, per_step=False):
        """ms per step over n steps, CUDA events on the launching stream, barrier and synchronize
        on both sides, max over ranks; with the clocks sampled during the timed region.  With
        per_step, an event is also recorded between steps and the third value is this rank's
        per-step distribution (ms: mean, p50, p99, min, max)."""
        import torch
        step = step or self.step
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        mid = [torch.cuda.Event(enable_timing=True) for _ in range(n - 1)] if per_step else []
        with ClockSampler(local_rank, clock_ms) as clk:
            barrier(world)
            torch.cuda.synchronize(self.dev)
            clk.start()
            e0.record(self.stream)
            for i in range(n):
                step()
                if per_step and i < n - 1:
                    mid[i].record(self.stream)
            e1.record(self.stream)
            torch.cuda.synchronize(self.dev)
            clk.stop()
            barrier(world)
        assert self.K.kvlink_device_status() == 0
        ms = max_over_ranks(e0.elapsed_time(e1), world, self.dev) / n
        if not per_step:
            return ms, clk.summary()
        marks = [e0] + mid + [e1]
        d = np.array([a.elapsed_time(b_) for a, b_ in zip(marks[:-1], marks[1:])])
        dist = {"mean": round(float(d.mean()), 4), "p50": round(float(np.median(d)), 4),
                "p99": round(float(np.percentile(d, 99)), 4), "min": round(float(d.min()), 4),
                "max": round(float(d.max()), 4)}
        return ms, clk.summary(), dist

    def kernel_pass(self, k_steps):
        """The step's kernels timed one launch at a time with events around each call: per layer
        the re-encode of its document caches, then the attention kernel alone (the fresh rows
        already in the cache); and every layer's re-encode in one launch, for comparison.
        Returns seconds per launch (re-encode, attention, all-layer re-encode)."""
        import torch
        K, dev, stream, sh, L = self.K, self.dev, self.stream, self.sh, self.L

        def timed(fn, n):
            evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n)]
            torch.cuda.synchronize(dev)
            for j, (a, b_) in enumerate(evs):
                a.record(stream)
                fn(j)
                b_.record(stream)
            torch.cuda.synchronize(dev)
            return float(np.mean([a.elapsed_time(b_) for a, b_ in evs])) * 1e-3

        if self.one_kernel:      # the whole layer is one kernel: timed as the "attention" launch
            return float("nan"), timed(lambda j: self.layer_call(j % L), k_steps * L), float("nan")
        ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(L * k_steps)]
        torch.cuda.synchronize(dev)
        for j, (a, b_, c) in enumerate(ev):
            l = j % L
            a.record(stream)
            K.kvlink_reencode_concat(self.plan, self.pool_k[l].data_ptr(), self.pool_v[l].data_ptr(),
                                     self.ck[l].data_ptr(), self.cv[l].data_ptr(), sh)
            b_.record(stream)
            K.kvlink_suffix_attention(self.plan, self.q[l].data_ptr(), None, None, self.ck[l].data_ptr(),
                                      self.cv[l].data_ptr(), self.out[l].data_ptr(), self.ws, self.wsb, sh)
            c.record(stream)
        torch.cuda.synchronize(dev)
        t_re = float(np.mean([a.elapsed_time(b_) for a, b_, _ in ev])) * 1e-3
        t_at = float(np.mean([b_.elapsed_time(c) for _, b_, c in ev])) * 1e-3
        t_re_all = timed(lambda j: K.kvlink_reencode_concat_layers(self.plan, *self.layer_ptrs, sh), k_steps)
        # the attention launches back to back over the layers (one event pair around all of them)
        n_b2b = k_steps * L
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize(dev)
        e0.record(stream)
        for j in range(n_b2b):
            l = j % L
            K.kvlink_suffix_attention(self.plan, self.q[l].data_ptr(), None, None, self.ck[l].data_ptr(),
                                      self.cv[l].data_ptr(), self.out[l].data_ptr(), self.ws, self.wsb, sh)
        e1.record(stream)
        torch.cuda.synchronize(dev)
        self.t_at_b2b = e0.elapsed_time(e1) * 1e-3 / n_b2b
        assert K.kvlink_device_status() == 0
        return t_re, t_at, t_re_all

    def roofline(self, t_re, t_at, t_re_all, peaks):
        """Per-kernel figures and the roofline entry of the dominant kernel.  Both kernels are
        timed alone, launch by launch, so the attention's fraction is of the burst bf16 peak
        (the sustained fraction is reported beside it)."""
        cnt = algorithmic_counts(self.batch, self.info)
        at_tfs = cnt["attn_flops"] / t_at / 1e12
        at_frac = at_tfs / peaks["bf16_tflops"]
        default_path = not self.one_kernel and self.layout == "interleaved"
        b2b = getattr(self, "t_at_b2b", None)
        attn_entry = {"us_per_launch": round(t_at * 1e6, 2), "TFLOP_per_s": round(at_tfs, 2),
                      "frac_bf16_burst": round(at_frac, 4),
                      "us_per_launch_back_to_back": round(b2b * 1e6, 2) if b2b else None,
                      "frac_bf16_burst_back_to_back": round(cnt["attn_flops"] / b2b / 1e12 / peaks["bf16_tflops"], 4)
                      if b2b else None,
                      "frac_bf16_sustained": round(at_tfs / peaks["bf16_tflops_sustained"], 4),
                      "algorithmic_flops": cnt["attn_flops"],
                      "hbm_bound_us": round(cnt["attn_bytes"] / peaks["hbm_gbs"] / 1e3, 2),
                      "traffic": ncu_traffic("attention", self.cfg.index) if default_path else None}
        if self.one_kernel:
            kernels = {"linked_prefill_fused": attn_entry}
            re_gbs = float("nan")
        else:
            re_gbs = cnt["reencode_bytes"] / t_re / 1e9
            re_all_gbs = self.L * cnt["reencode_bytes"] / t_re_all / 1e9
            kernels = {"reencode_concat": {"us_per_launch": round(t_re * 1e6, 2), "GB_per_s": round(re_gbs, 1),
                                           "frac_hbm": round(re_gbs / peaks["hbm_gbs"], 4),
                                           "frac_8TBs": round(re_gbs / 8000.0, 4),
                                           "algorithmic_bytes": cnt["reencode_bytes"],
                                           "bytes_per_query_doc_count": cnt["reencode_bytes_naive"],
                                           "traffic": ncu_traffic("reencode", self.cfg.index) if default_path
                                           else None},
                       "reencode_concat_all_layers": {"us_per_launch": round(t_re_all * 1e6, 2), "layers": self.L,
                                                      "GB_per_s": round(re_all_gbs, 1),
                                                      "frac_hbm": round(re_all_gbs / peaks["hbm_gbs"], 4),
                                                      "note": "every layer in one launch; not on the step's path"},
                       "suffix_attention": attn_entry}
        if self.one_kernel or t_at >= t_re:
            name = ("kvlink linked_prefill_fused (one kernel)" if self.one_kernel else
                    "kvlink suffix attention" + ("" if self.layout == "interleaved" else " (rows gathered)"))
            roof = {"kernel": name, "bound": "tensor", "achieved": round(at_tfs, 2), "peak": peaks["bf16_tflops"],
                    "unit": "TFLOP/s", "frac": round(at_frac, 4), "traffic": attn_entry["traffic"],
                    "peak_kind": f"bf16 dense burst ({peaks['source']}): the kernel is timed alone, launch by launch",
                    "algorithmic_unit": "4 * h_q * head_dim flops per unmasked (fresh row, key) pair",
                    "algorithmic_per_launch": cnt["attn_flops"]}
        else:
            roof = {"kernel": "kvlink reencode_concat", "bound": "hbm", "achieved": round(re_gbs, 1),
                    "peak": peaks["hbm_gbs"], "unit": "GB/s", "frac": round(re_gbs / peaks["hbm_gbs"], 4),
                    "traffic": kernels["reencode_concat"]["traffic"], "peak_kind": f"HBM copy ({peaks['source']})",
                    "algorithmic_unit": "unique pool K+V rows read + linked-cache K+V rows written",
                    "algorithmic_per_launch": cnt["reencode_bytes"]}
        return roof, kernels

    def host_pool_leg(self, args, world, local_rank):
        """The same step with every layer's document cache pool in page-locked host memory
        (kvlink_linked_prefill_layers_host_pool: each layer's documents read over the host link
        by the re-encode, on the load stream, while earlier layers' attention runs), and one
        layer's host-pool re-encode timed alone."""
        import torch
        K = self.K
        h_k = [torch.empty(t.shape, dtype=t.dtype, pin_memory=True) for t in self.pool_k]
        h_v = [torch.empty(t.shape, dtype=t.dtype, pin_memory=True) for t in self.pool_v]
        for h, d in zip(h_k + h_v, self.pool_k + self.pool_v):
            h.copy_(d)
        ptrs = [[t.data_ptr() for t in seq] for seq in (h_k, h_v, self.q, self.kn, self.vn, self.ck, self.cv, self.out)]

        def step():
            K.kvlink_linked_prefill_layers_host_pool(self.plan, *ptrs, self.ws, self.wsb, self.sh, self.re_sh)

        for _ in range(args.warmup):
            step()
        torch.cuda.synchronize(self.dev)
        ms, clocks = self.timed_steps(args.steps, world, args.clock_ms, local_rank, step)
        n = min(args.steps, 5) * self.L
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n)]
        for j, (a, b_) in enumerate(evs):
            l = j % self.L
            a.record(self.stream)
            K.kvlink_reencode_concat_host_pool(self.plan, h_k[l].data_ptr(), h_v[l].data_ptr(), self.ck[l].data_ptr(),
                                               self.cv[l].data_ptr(), self.sh)
            b_.record(self.stream)
        torch.cuda.synchronize(self.dev)
        assert K.kvlink_device_status() == 0
        t = float(np.mean([a.elapsed_time(b_) for a, b_ in evs])) * 1e-3
        cnt = algorithmic_counts(self.batch, self.info)
        read = cnt["reencode_bytes"] - 2 * self.cfg.h_kv * self.cfg.head_dim * 2 * int(self.info.cached_tokens)
        return {"value": round(whole_job_us_per_query(ms, self.cfg.batch, world), 3), "unit": UNIT,
                "ms_per_step": round(ms, 4), "steps": args.steps, "clocks": clocks,
                "reencode_host_pool_us_per_launch": round(t * 1e6, 2),
                "host_read_GB_per_s": round(read / t / 1e9, 1),
                "device_write_GB_per_s": round((cnt["reencode_bytes"] - read) / t / 1e9, 1),
                "host_bytes_read_per_layer": int(read),
                "note": "every layer's document pool in pinned host memory, read over NVLink-C2C by the "
                        "re-encode (kvlink_linked_prefill_layers_host_pool); fresh rows resident in HBM"}

    def zero_copy_leg(self, args, world, local_rank):
        """The same step with zero-copy values (cache_v NULL): the re-encode writes keys only and
        the attention reads every value row where it is (pool rows, v_new); and the two kernels
        of one layer timed alone, launch by launch."""
        import torch
        K, sh = self.K, self.sh
        ptrs = list(self.ptrs)
        ptrs[6] = None

        def step():
            K.kvlink_linked_prefill_layers_overlapped(self.plan, *ptrs, self.ws, self.wsb, sh, self.re_sh)

        for _ in range(args.warmup):
            step()
        torch.cuda.synchronize(self.dev)
        ms, clocks = self.timed_steps(args.steps, world, args.clock_ms, local_rank, step)
        n = min(args.steps, 20) * self.L
        ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(n)]
        torch.cuda.synchronize(self.dev)
        for j, (a, b_, c) in enumerate(ev):
            l = j % self.L
            a.record(self.stream)
            K.kvlink_reencode_concat(self.plan, self.pool_k[l].data_ptr(), None, self.ck[l].data_ptr(), None, sh)
            b_.record(self.stream)
            K.kvlink_suffix_attention_pool_values(self.plan, self.q[l].data_ptr(), None, self.vn[l].data_ptr(),
                                                  self.pool_v[l].data_ptr(), self.ck[l].data_ptr(),
                                                  self.out[l].data_ptr(), self.ws, self.wsb, sh)
            c.record(self.stream)
        torch.cuda.synchronize(self.dev)
        assert K.kvlink_device_status() == 0
        t_re = float(np.mean([a.elapsed_time(b_) for a, b_, _ in ev])) * 1e-3
        t_at = float(np.mean([b_.elapsed_time(c) for _, b_, c in ev])) * 1e-3
        cnt = algorithmic_counts(self.batch, self.info)
        peaks = _peaks()
        re_bytes = cnt["reencode_bytes"] // 2          # keys only: half of the K+V figure
        at_tfs = cnt["attn_flops"] / t_at / 1e12
        return {"value": round(whole_job_us_per_query(ms, self.cfg.batch, world), 3), "unit": UNIT,
                "ms_per_step": round(ms, 4), "steps": args.steps, "clocks": clocks,
                "reencode_keys_us_per_launch": round(t_re * 1e6, 2),
                "reencode_keys_GB_per_s": round(re_bytes / t_re / 1e9, 1),
                "reencode_keys_frac_hbm": round(re_bytes / t_re / 1e9 / peaks["hbm_gbs"], 4),
                "reencode_keys_algorithmic_bytes": int(re_bytes),
                "attention_pool_values_us_per_launch": round(t_at * 1e6, 2),
                "attention_pool_values_TFLOP_per_s": round(at_tfs, 2),
                "attention_pool_values_frac_bf16_burst": round(at_tfs / peaks["bf16_tflops"], 4),
                "reencode_keys_traffic": ncu_traffic("reencode_keys", self.cfg.index) if self.layout == "interleaved" else None,
                "attention_pool_values_traffic": ncu_traffic("attention_pool_values", self.cfg.index) if self.layout == "interleaved" else None,
                "launches_per_step": 3 * self.L,
                "note": "kvlink_linked_prefill_layers_overlapped with cache_v NULL: keys re-encoded into "
                        "the linked cache, values read by the attention from the pool and v_new (no "
                        "value copy); the line's value keeps the linked value cache"}

    def config(self, world):
        cfg, info = self.cfg, self.info
        return {"workload": cfg.name, "index": cfg.index, "batch_per_gpu": cfg.batch, "layers": self.L,
                "h_q": cfg.h_q,
                "h_kv": cfg.h_kv, "head_dim": cfg.head_dim, "docs_per_query": cfg.docs_per_query,
                "n_link": cfg.n_link, "ctx_tokens_per_query": int(info.ctx_rows) // cfg.batch,
                "fresh_rows": int(info.n_fresh), "pool": "paged, 16-token blocks" if cfg.pool_block_size else
                "contiguous", "parallelism": f"replicas x{world} (independent batches)", "path": self.path,
                "layout": self.layout,
                "l2": "inputs larger than L2: each layer has its own pool "
                      f"({self.pool_k[0].numel() * 4 / 1e6:.0f} MB K+V) and cache "
                      f"({self.ck[0].numel() * 4 / 1e6:.0f} MB K+V)"}


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def run_e2e(wl, args, world):
    """The same metric through the public API with host buffers (kvlink_linked_prefill_layers_host)."""
    import torch

    from paper_2502_16002_gb300.runtime import LinkedPrefill
    dev, stream, batch, cfg = wl.dev, wl.stream, wl.batch, wl.cfg
    h_q = torch.empty(wl.q.shape, dtype=wl.q.dtype, pin_memory=True)
    h_kn = torch.empty(wl.kn.shape, dtype=wl.kn.dtype, pin_memory=True)
    h_vn = torch.empty(wl.vn.shape, dtype=wl.vn.dtype, pin_memory=True)
    h_out = torch.empty(wl.out.shape, dtype=wl.out.dtype, pin_memory=True)
    h_q.copy_(wl.q)
    h_kn.copy_(wl.kn)
    h_vn.copy_(wl.vn)
    e2e_steps = max(1, min(args.steps, 10))
    streams = (torch.cuda.Stream(dev), stream, torch.cuda.Stream(dev))
    p_e2e = LinkedPrefill.from_batch(batch, device=dev, stream=stream)

    def e2e_step():
        # a new batch: the plan rebuilt on the host and uploaded (ordered after the previous
        # batch's kernels), then every layer with its fresh rows copied in from pinned host
        # memory and its output copied back to pinned host memory, pipelined per layer; the
        # host prepares the next batch while this one runs
        p_e2e.rebuild_from_batch(batch, stream=stream)
        p_e2e.linked_prefill_layers_from_host(wl.pool_k, wl.pool_v, h_q, h_kn, h_vn, wl.q, wl.kn, wl.vn, wl.ck,
                                              wl.cv, wl.out, h_out, streams=streams, wait=False)

    e2e_step()
    torch.cuda.synchronize(dev)
    barrier(world)
    torch.cuda.synchronize(dev)
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        e2e_step()
    torch.cuda.synchronize(dev)          # every step's output is on the host
    t1 = time.perf_counter()
    barrier(world)
    e2e_ms = max_over_ranks((t1 - t0) * 1e3, world, dev) / e2e_steps
    h2d = (h_q.numel() + h_kn.numel() + h_vn.numel()) * 2 + int(wl.info.device_bytes)
    return {"value": round(whole_job_us_per_query(e2e_ms, cfg.batch, world), 3), "unit": UNIT,
            "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(h_out.numel() * 2),
            "steps": e2e_steps,
            "note": "per step: host plan rebuild + table upload, then kvlink_linked_prefill_layers_host: "
                    "per layer fresh q/k/v H2D from pinned memory, document re-encode on its own "
                    "stream, placement + attention, output D2H to pinned memory (four streams); steps "
                    "pipelined (the host prepares the next batch while one runs), wall clock from the "
                    "first step's start to the last output on the host; document pool resident in HBM"}


def run_ours(args, rank, world, local_rank, cfg_index, main=True):
    """One workload: the timed K steps (the line's value), the per-kernel pass and roofline,
    and for the main workload also a sustained run of at least a second with its clocks and
    the end-to-end leg."""
    import torch

    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    wl = Workload(args, cfg_index, rank, dev)
    for _ in range(args.warmup):
        wl.step()
    torch.cuda.synchronize(dev)
    assert wl.K.kvlink_device_status() == 0

    # ---- timed region: the production path, exactly K steps
    ms_per_step, clocks = wl.timed_steps(args.steps, world, args.clock_ms, local_rank)
    value = whole_job_us_per_query(ms_per_step, wl.cfg.batch, world)

    # ---- the same step for at least a second, so that the clock record has many samples
    sustained = None
    if main and not args.no_sustained:
        n = int(min(5000, max(args.steps, math.ceil(1.2e3 / max(ms_per_step, 1e-3)))))
        ms_s, clk_s, dist = wl.timed_steps(n, world, args.clock_ms, local_rank, per_step=True)
        sustained = {"steps": n, "ms_per_step": round(ms_s, 4),
                     "value": round(whole_job_us_per_query(ms_s, wl.cfg.batch, world), 3), "unit": UNIT,
                     "timed_s": round(n * ms_s / 1e3, 3), "clocks": clk_s,
                     "step_ms_distribution": dist}

    t_re, t_at, t_re_all = wl.kernel_pass(min(args.steps, 20) if main else min(args.steps, 5))
    roof, kernels = wl.roofline(t_re, t_at, t_re_all, _peaks())

    zero_copy = None
    if not args.no_zero_copy and not wl.one_kernel:
        zero_copy = wl.zero_copy_leg(args, world, local_rank)

    e2e = host_pool = None
    if main and not args.no_e2e and not wl.one_kernel and args.layout == "interleaved":
        e2e = run_e2e(wl, args, world)
    if main and not args.no_host_pool and not wl.one_kernel and args.layout == "interleaved":
        host_pool = wl.host_pool_leg(args, world, local_rank)

    res = {
        "metric": METRIC, "value": round(value, 3), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_per_step, 4),
        "higher_is_better": False, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic N(0,1) bf16, seeded; document pool resident in HBM",
        "config": wl.config(world),
        "roofline": roof,
        "kernels": kernels,
        "per_rank_us_per_query": round(ms_per_step * 1e3 / wl.cfg.batch, 3),
        "gpu_launches": int(args.steps * wl.launches_per_step()),
        "clocks": clocks,
        "zero_copy_values": zero_copy,
    }
    if main:
        res["sustained"] = sustained
        res["e2e"] = e2e
        res["host_pool"] = host_pool
    del wl
    torch.cuda.synchronize(dev)
    torch.cuda.empty_cache()
    return res


# ------------------------------------------------------------------ CPU oracle (baseline)

def oracle_sample(cfg, n_layers=None, max_seconds=20.0):
    """Time the fp64 oracle on (query, layer) samples of the workload.

    Layers are taken in the order 0, L-1, L/2, ...; within a layer every query is run
    until max_seconds of oracle time have been spent.  Returns (us per query over all
    layers, seconds spent, description)."""
    import oracle

    batch = W.draw_batch(cfg)
    layers = [0, cfg.layers - 1, cfg.layers // 2, cfg.layers // 4][: (n_layers or 4)]
    layers = list(dict.fromkeys(layers))
    times, done, spent = [], [], 0.0
    for layer in layers:
        pk, pv = W.pool_kv(batch, layer)
        q, kn, vn = W.fresh_qkv(batch, layer)
        for b in range(cfg.batch):
            t0 = time.perf_counter()
            oracle.oracle_query_layer(batch, b, pk, pv, q, kn, vn)
            dt = time.perf_counter() - t0
            times.append(dt)
            done.append((b, layer))
            spent += dt
            if spent > max_seconds:
                break
        if spent > max_seconds:
            break
    per_query_layer = float(np.mean(times))
    desc = (f"{len(done)} (query, layer) samples over layers {sorted(set(l for _, l in done))} of "
            f"{cfg.name}: full re-encode/concat of the query's cache and attention of all its fresh "
            f"rows and heads in fp64 (numpy, BLAS threads); value = mean per (query, layer) x "
            f"{cfg.layers} layers")
    return per_query_layer * cfg.layers * 1e6, spent, desc


def run_reference(args):
    cfg = W.get_config(args.config)
    for _ in range(args.warmup):
        oracle_sample(cfg, n_layers=1, max_seconds=0.0)
    vals = []
    t_all = 0.0
    for _ in range(args.steps):
        v, s, desc = oracle_sample(cfg, n_layers=1, max_seconds=0.0)
        vals.append(v)
        t_all += s
    value = float(np.mean(vals))
    cores = _cores()
    return {"metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": 1, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": round(t_all / max(1, args.steps) * 1e3, 2),
            "higher_is_better": False, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic N(0,1) bf16, seeded", "impl": "reference",
            "config": {"workload": cfg.name, "batch_per_gpu": cfg.batch, "layers": cfg.layers},
            "cpu_baseline": {"value": round(value, 1), "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": "each step: " + desc},
            "e2e": {"value": round(value, 1), "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=300)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--config", type=int, default=3)
    ap.add_argument("--layers", type=int, default=0,
                    help="layers per step (default: the workload's); fewer only for small profiling runs")
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--path", choices=["two-kernel", "two-kernel-serial", "one-kernel", "one-kernel-k-only"],
                    default="two-kernel")
    ap.add_argument("--layout", choices=["interleaved", "links_at_end"], default="interleaved")
    ap.add_argument("--extra-configs", type=int, nargs="*", default=None,
                    help="further workloads timed after the main one and reported under 'workloads' "
                         "(default: 4 and 5 when the main workload is 3)")
    ap.add_argument("--clock-ms", type=int, default=50, help="nvidia-smi sampling interval")
    ap.add_argument("--no-host-pool", action="store_true",
                    help="skip the leg with the document pool in pinned host memory")
    ap.add_argument("--no-zero-copy", action="store_true",
                    help="skip the leg with zero-copy values (cache_v NULL)")
    ap.add_argument("--no-sustained", action="store_true",
                    help="skip the run of at least a second that gives the clock record many samples")
    args = ap.parse_args()
    if args.extra_configs is None:
        args.extra_configs = [4, 5] if args.config == 3 and not args.layers else []
    if args.warmup < 3 and args.impl == "ours":
        print("warning: fewer than 3 warm-up steps", file=sys.stderr)

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        if rank == 0:
            print(json.dumps(run_reference(args)), flush=True)
        return

    if world > 1:
        import torch
        import torch.distributed as dist
        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    res = run_ours(args, rank, world, local_rank, args.config)
    extra = {}
    for c in args.extra_configs:
        r = run_ours(args, rank, world, local_rank, c, main=False)
        extra[r["config"]["workload"]] = {k: r[k] for k in ("value", "unit", "ms_per_step", "steps", "config",
                                                             "roofline", "kernels", "clocks", "gpu_launches",
                                                             "zero_copy_values")}
    if extra:
        res["workloads"] = extra
    if rank == 0:
        if not args.no_cpu_baseline and world == 1:
            def baseline(cfg_index, seconds):
                v, spent, desc = oracle_sample(W.get_config(cfg_index), max_seconds=seconds)
                return {"value": round(v, 1), "unit": UNIT, "cores": _cores(), "kind": "oracle",
                        "sample": desc, "seconds": round(spent, 1)}
            res["cpu_baseline"] = baseline(args.config, 20.0)
            for name, r in extra.items():
                r["cpu_baseline"] = baseline(r["config"]["index"], 8.0)
        print(json.dumps(res), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
