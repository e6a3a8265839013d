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
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import workloads as W  # noqa: E402

METRIC = "linked-prefill us/query (all layers, 8B-shape)"
UNIT = "us/query"

# dram__bytes_read.sum + dram__bytes_write.sum per launch from the committed ncu
# summaries under profiles/, keyed by (kernel, workload); None until captured for
# the current kernel version.
NCU_TRAFFIC = {
    ("attention", 3): 259171328,   # profiles/attention_tc_llama8b_b8_zipf.md
    ("reencode", 3): 214893056,    # profiles/reencode_llama8b_b8_zipf.md (cached rows)
}


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


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 200 ms in a background reader.

    Each line is stamped when it arrives; summary() keeps the samples that fall inside
    the window marked with start() / stop()."""

    Q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []
        self.t0 = self.t1 = None

    def __enter__(self):
        import threading
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (FileNotFoundError, OSError):
            self.proc = None
            return self

        def reader():
            for line in self.proc.stdout:
                self.lines.append((time.time(), line))

        self.thread = threading.Thread(target=reader, daemon=True)
        self.thread.start()
        time.sleep(0.5)  # let the first samples arrive before the timed region
        return self

    def start(self):
        self.t0 = time.time()

    def stop(self):
        self.t1 = time.time()

    def __exit__(self, *a):
        if self.proc is None:
            return
        time.sleep(0.3)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=5)

    def summary(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        sm, mx, reasons, n_all = [], None, set(), 0
        for t, line in self.lines:
            f = [x.strip() for x in line.split(",")]
            if len(f) < 8:
                continue
            n_all += 1
            if self.t0 is not None and not (self.t0 - 0.2 <= t <= self.t1 + 0.2):
                continue
            try:
                sm.append(float(f[0]))
                mx = float(f[1])
            except ValueError:
                continue
            for n, v in zip(names, f[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": mx, "reasons": sorted(reasons), "samples": 0,
                    "samples_total": n_all}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


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

def run_ours(args, rank, world, local_rank):
    import torch

    from paper_2502_16002_gb300 import kvlink as K
    from paper_2502_16002_gb300.runtime import LinkedPrefill

    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    cfg = W.get_config(args.config)
    batch = W.draw_batch(cfg, seed=rank_batch_seed(rank))   # every rank serves its own batch
    L = args.layers or cfg.layers
    layout = {"interleaved": K.KVLINK_LAYOUT_INTERLEAVED, "links_at_end": K.KVLINK_LAYOUT_LINKS_AT_END}[args.layout]
    lp = LinkedPrefill.from_batch(batch, device=dev, layout=layout)
    info = lp.info
    ctx, T = int(info.ctx_rows), int(info.n_fresh)
    H, Hq, D = cfg.h_kv, cfg.h_q, cfg.head_dim
    pool_shape = ((batch.pool_rows // cfg.pool_block_size, cfg.pool_block_size, H, D)
                  if cfg.pool_block_size else (batch.pool_rows, H, D))
    base = 1_000_000 * (rank + 1)
    pool_k = [W.normal_bf16_torch(pool_shape, base + 10 * l + 1, dev) for l in range(L)]
    pool_v = [W.normal_bf16_torch(pool_shape, base + 10 * l + 2, dev) for l in range(L)]
    q = W.normal_bf16_torch((L, T, Hq, D), base + 3, dev)
    kn = W.normal_bf16_torch((L, T, H, D), base + 4, dev)
    vn = W.normal_bf16_torch((L, T, H, D), base + 5, dev)
    ck = torch.empty((L, ctx, H, D), dtype=torch.bfloat16, device=dev)
    cv = torch.empty_like(ck)
    out = torch.empty((L, T, Hq, D), dtype=torch.bfloat16, device=dev)
    stream = torch.cuda.current_stream(dev)
    sh = int(stream.cuda_stream)
    ws, wsb = lp.workspace.data_ptr(), lp.workspace.numel()
    plan = lp.plan

    one_kernel = args.path.startswith("one-kernel")

    def layer_call(l):
        if one_kernel:
            K.kvlink_linked_prefill_fused(plan, pool_k[l].data_ptr(), pool_v[l].data_ptr(), q[l].data_ptr(),
                                          kn[l].data_ptr(), vn[l].data_ptr(), ck[l].data_ptr(),
                                          None if args.path == "one-kernel-k-only" else cv[l].data_ptr(),
                                          out[l].data_ptr(), ws, wsb, sh)
        else:
            K.kvlink_linked_prefill(plan, pool_k[l].data_ptr(), pool_v[l].data_ptr(), q[l].data_ptr(),
                                    kn[l].data_ptr(), vn[l].data_ptr(), ck[l].data_ptr(), cv[l].data_ptr(),
                                    out[l].data_ptr(), ws, wsb, sh)

    ptrs = [[t.data_ptr() for t in seq] for seq in (pool_k, pool_v, q, kn, vn, ck, cv, out)]
    re_stream = torch.cuda.Stream(dev)
    re_sh = int(re_stream.cuda_stream)
    layer_ptrs = [[t.data_ptr() for t in seq] for seq in (pool_k, pool_v, ck, cv)]

    def step():
        if one_kernel:
            for l in range(L):
                layer_call(l)
        elif args.path == "two-kernel-serial":
            K.kvlink_linked_prefill_layers(plan, *ptrs, ws, wsb, sh)
        else:
            K.kvlink_linked_prefill_layers_overlapped(plan, *ptrs, ws, wsb, sh, re_sh)

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize(dev)
    assert K.kvlink_device_status() == 0

    # ---- timed region: the production path
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local_rank) as clk:
        barrier()
        torch.cuda.synchronize(dev)
        clk.start()
        e0.record(stream)
        for _ in range(args.steps):
            step()
        e1.record(stream)
        torch.cuda.synchronize(dev)
        clk.stop()
        barrier()
    ms_total = max_over_ranks(e0.elapsed_time(e1), world, dev)
    ms_per_step = ms_total / args.steps
    us_per_query = ms_per_step * 1e3 / cfg.batch      # per rank; ranks run in parallel
    value = whole_job_us_per_query(ms_per_step, cfg.batch, world)
    assert K.kvlink_device_status() == 0

    # ---- per-kernel pass: same work through the separate calls, events around each
    k_steps = min(args.steps, 20)

    def timed(fn, n):
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n)]
        torch.cuda.synchronize(dev)
        for j, (a, b_) in enumerate(evs):
            a.record(stream)
            fn(j)
            b_.record(stream)
        torch.cuda.synchronize(dev)
        return float(np.mean([a.elapsed_time(b_) for a, b_ in evs])) * 1e-3      # s per call

    t_re = t_re_all = float("nan")
    if one_kernel:      # the whole layer is one kernel: timed as the "attention" launch
        t_at = timed(lambda j: layer_call(j % L), k_steps * L)
    else:
        # per layer, as the step runs them: the re-encode of the layer's document caches,
        # then the attention kernel alone (the fresh rows are already in the cache)
        ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(L * k_steps)]
        torch.cuda.synchronize(dev)
        for j, (a, b_, c) in enumerate(ev):
            l = j % L
            a.record(stream)
            K.kvlink_reencode_concat(plan, pool_k[l].data_ptr(), pool_v[l].data_ptr(), ck[l].data_ptr(),
                                     cv[l].data_ptr(), sh)
            b_.record(stream)
            K.kvlink_suffix_attention(plan, q[l].data_ptr(), None, None, ck[l].data_ptr(), cv[l].data_ptr(),
                                      out[l].data_ptr(), ws, wsb, sh)
            c.record(stream)
        torch.cuda.synchronize(dev)
        t_re = float(np.mean([a.elapsed_time(b_) for a, b_, _ in ev])) * 1e-3   # s per launch
        t_at = float(np.mean([b_.elapsed_time(c) for _, b_, c in ev])) * 1e-3
        # every layer's document caches in one launch, for comparison (not on the step's path)
        t_re_all = timed(lambda j: K.kvlink_reencode_concat_layers(plan, *layer_ptrs, sh), k_steps)
    assert K.kvlink_device_status() == 0

    # ---- end to end through the public API with host buffers
    e2e = None
    if not args.no_e2e and not one_kernel and args.layout == "interleaved":
        h_q = torch.empty(q.shape, dtype=q.dtype, pin_memory=True)
        h_kn = torch.empty(kn.shape, dtype=kn.dtype, pin_memory=True)
        h_vn = torch.empty(vn.shape, dtype=vn.dtype, pin_memory=True)
        h_out = torch.empty(out.shape, dtype=out.dtype, pin_memory=True)
        h_q.copy_(q)
        h_kn.copy_(kn)
        h_vn.copy_(vn)
        e2e_steps = max(1, min(args.steps, 10))

        streams = (torch.cuda.Stream(dev), stream, torch.cuda.Stream(dev))

        p_e2e = LinkedPrefill.from_batch(batch, device=dev, stream=stream)

        def e2e_step():
            # a new batch: the plan rebuilt on the host and uploaded (ordered after the previous
            # batch's kernels), then every layer with its fresh rows copied in from pinned host
            # memory and its output copied back to pinned host memory, pipelined per layer; the
            # host prepares the next batch while this one runs
            p_e2e.rebuild_from_batch(batch, stream=stream)
            p_e2e.linked_prefill_layers_from_host(pool_k, pool_v, h_q, h_kn, h_vn, q, kn, vn, ck, cv, out, h_out,
                                                  streams=streams, wait=False)

        e2e_step()
        torch.cuda.synchronize(dev)
        barrier()
        torch.cuda.synchronize(dev)
        t0 = time.perf_counter()
        for _ in range(e2e_steps):
            e2e_step()
        torch.cuda.synchronize(dev)          # every step's output is on the host
        t1 = time.perf_counter()
        barrier()
        e2e_ms = max_over_ranks((t1 - t0) * 1e3, world, dev) / e2e_steps
        h2d = (h_q.numel() + h_kn.numel() + h_vn.numel()) * 2 + int(info.device_bytes)
        e2e = {"value": round(whole_job_us_per_query(e2e_ms, cfg.batch, world), 3), "unit": UNIT,
               "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(h_out.numel() * 2),
               "steps": e2e_steps,
               "note": "per step: host plan rebuild + table upload, then kvlink_linked_prefill_layers_host: "
                       "per layer fresh q/k/v H2D from pinned memory, document re-encode on its own "
                       "stream, placement + attention, output D2H to pinned memory (four streams); steps "
                       "pipelined (the host prepares the next batch while one runs), wall clock from the "
                       "first step's start to the last output on the host; document pool resident in HBM"}

    peaks = _peaks()
    cnt = algorithmic_counts(batch, info)
    re_gbs = cnt["reencode_bytes"] / t_re / 1e9
    re_all_gbs = L * cnt["reencode_bytes"] / t_re_all / 1e9
    at_tfs = cnt["attn_flops"] / t_at / 1e12
    re_frac = re_gbs / peaks["hbm_gbs"]
    at_frac = at_tfs / peaks["bf16_tflops_sustained"]
    dominant = "attention" if one_kernel or t_at >= t_re else "reencode"
    default_path = not one_kernel and args.layout == "interleaved"
    if dominant == "attention":
        name = ("kvlink linked_prefill_fused (one kernel)" if one_kernel else
                "kvlink suffix attention" + ("" if args.layout == "interleaved" else " (rows gathered)"))
        roof = {"kernel": name, "bound": "tensor", "achieved": round(at_tfs, 2),
                "peak": peaks["bf16_tflops_sustained"], "unit": "TFLOP/s", "frac": round(at_frac, 4),
                "traffic": NCU_TRAFFIC.get(("attention", cfg.index)) if default_path else None,
                "peak_kind": f"bf16 sustained, {peaks['source']}"}
    else:
        roof = {"kernel": "kvlink reencode_concat", "bound": "hbm", "achieved": round(re_gbs, 1),
                "peak": peaks["hbm_gbs"], "unit": "GB/s", "frac": round(re_frac, 4),
                "traffic": NCU_TRAFFIC.get(("reencode", cfg.index)) if default_path else None,
                "peak_kind": f"HBM copy, {peaks['source']}"}
    n_merge = 1 if info.n_attn_splits > 0 else 0
    launches_per_step = L * ((1 if one_kernel else 2 if args.path == "two-kernel-serial" else 3) + n_merge)
    attn_entry = {"us_per_launch": round(t_at * 1e6, 2), "TFLOP_per_s": round(at_tfs, 2),
                  "frac_bf16_sustained": round(at_frac, 4),
                  "frac_bf16_burst": round(at_tfs / peaks["bf16_tflops"], 4),
                  "algorithmic_flops": cnt["attn_flops"],
                  "hbm_bound_us": round(cnt["attn_bytes"] / peaks["hbm_gbs"] / 1e3, 2)}
    if one_kernel:
        kernels = {"linked_prefill_fused": attn_entry}
    else:
        kernels = {"reencode_concat": {"us_per_launch": round(t_re * 1e6, 2), "GB_per_s": round(re_gbs, 1),
                                       "frac_hbm": round(re_frac, 4),
                                       "frac_8TBs": round(re_gbs / 8000.0, 4),
                                       "algorithmic_bytes": cnt["reencode_bytes"],
                                       "bytes_per_query_doc_count": cnt["reencode_bytes_naive"]},
                   "reencode_concat_all_layers": {"us_per_launch": round(t_re_all * 1e6, 2), "layers": L,
                                                  "GB_per_s": round(re_all_gbs, 1),
                                                  "frac_hbm": round(re_all_gbs / peaks["hbm_gbs"], 4),
                                                  "note": "every layer in one launch; not on the step's path"},
                   "suffix_attention": attn_entry}
    res = {
        "metric": METRIC, "value": round(value, 3), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_per_step, 4),
        "higher_is_better": False, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic N(0,1) bf16, seeded; document pool resident in HBM",
        "config": {"workload": cfg.name, "batch_per_gpu": cfg.batch, "layers": L, "h_q": Hq, "h_kv": H,
                   "head_dim": D, "docs_per_query": cfg.docs_per_query, "n_link": cfg.n_link,
                   "ctx_tokens_per_query": ctx // cfg.batch, "fresh_rows": T,
                   "parallelism": f"replicas x{world} (independent batches)",
                   "path": args.path, "layout": args.layout,
                   "l2": "inputs larger than L2: each layer has its own pool "
                         f"({pool_k[0].numel() * 4 / 1e6:.0f} MB K+V) and cache "
                         f"({ck[0].numel() * 4 / 1e6:.0f} MB K+V)"},
        "roofline": roof,
        "kernels": kernels,
        "per_rank_us_per_query": round(us_per_query, 3),
        "gpu_launches": int(args.steps * launches_per_step),
        "clocks": clk.summary(),
        "e2e": e2e,
    }
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
    args = ap.parse_args()
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
    res = run_ours(args, rank, world, local_rank)
    if rank == 0:
        if not args.no_cpu_baseline and world == 1:
            v, spent, desc = oracle_sample(W.get_config(args.config))
            res["cpu_baseline"] = {"value": round(v, 1), "unit": UNIT, "cores": _cores(), "kind": "oracle",
                                   "sample": desc, "seconds": round(spent, 1)}
        print(json.dumps(res), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
