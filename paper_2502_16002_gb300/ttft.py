"""Time to first token: standard full prefill against KVLink's linked prefill on GB300.

The paper measures TTFT with ten retrieved documents of 100-500 tokens (1k-5k context) and
reports an 85-96 % reduction against encoding the whole context (Sec. 3.3).  This module
times one transformer layer of the Llama-3.1-8B shape with random weights in both ways and
scales by the layer count (every layer costs the same):

  standard  all N = sum(doc) + Q context tokens go through the layer: RMSNorm, QKV
            projection, RoPE at positions 0..N-1, causal attention over the N tokens,
            output projection, residual, RMSNorm, SwiGLU MLP, residual;
  linked    only the T = n_docs * K + Q fresh link and question tokens go through the
            layer; the documents' cached K/V are re-encoded and concatenated from the pool
            (kvlink_reencode_concat) and the fresh rows attend over the linked cache under
            KVLink's mask (kvlink_suffix_attention).  With --host-caches the documents'
            caches start in pinned host memory and are copied to the GPU in every layer,
            as in the paper's measurement (caches in CPU memory).

Both arms use the same weights, the same cuBLAS GEMMs (torch.matmul) and the same
elementwise glue (RMSNorm, SiLU, residual adds in torch); RoPE of the fresh rows and all
attention run in this library's kernels.  Each arm's layer is captured in a CUDA graph, so
host launch overhead is out of both measurements.  No accuracy is claimed: the weights are
random.

    python -m paper_2502_16002_gb300.ttft [--lengths 100 200 300 400 500] [--links 1 5]
"""
from __future__ import annotations

import argparse
import json

import numpy as np
import torch

from . import kvlink as K
from .clocks import ClockSampler
from .runtime import LinkedPrefill

HIDDEN, H_Q, H_KV, HEAD_DIM, FFN, LAYERS, THETA = 4096, 32, 8, 128, 14336, 32, 500000.0


class Layer:
    """Random bf16 weights of one Llama-3.1-8B-shaped layer, N(0, 1/fan_in): after the RMSNorm
    the projected q, k and v have unit variance, the value distribution of the workloads."""

    def __init__(self, device, seed=0):
        g = torch.Generator(device=device)
        g.manual_seed(seed)
        def w(o, i):
            return (torch.randn(o, i, generator=g, device=device, dtype=torch.float32) / i ** 0.5).to(torch.bfloat16)
        self.wqkv = w((H_Q + 2 * H_KV) * HEAD_DIM, HIDDEN)
        self.wo = w(HIDDEN, H_Q * HEAD_DIM)
        self.wgu = w(2 * FFN, HIDDEN)
        self.wd = w(HIDDEN, FFN)
        self.n1 = torch.ones(HIDDEN, device=device, dtype=torch.bfloat16)
        self.n2 = torch.ones(HIDDEN, device=device, dtype=torch.bfloat16)


def _rmsnorm(x, w, eps=1e-5):
    xf = x.float()
    return (xf * torch.rsqrt(xf.pow(2).mean(-1, keepdim=True) + eps)).to(x.dtype) * w


def _qkv(layer, x):
    qkv = _rmsnorm(x, layer.n1) @ layer.wqkv.t()
    n = x.shape[0]
    q = qkv[:, : H_Q * HEAD_DIM].reshape(n, H_Q, HEAD_DIM).contiguous()
    k = qkv[:, H_Q * HEAD_DIM: (H_Q + H_KV) * HEAD_DIM].reshape(n, H_KV, HEAD_DIM).contiguous()
    v = qkv[:, (H_Q + H_KV) * HEAD_DIM:].reshape(n, H_KV, HEAD_DIM).contiguous()
    return q, k, v


def _finish(layer, x, attn):
    x = x + attn.reshape(x.shape[0], H_Q * HEAD_DIM) @ layer.wo.t()
    gu = _rmsnorm(x, layer.n2) @ layer.wgu.t()
    h = torch.nn.functional.silu(gu[:, :FFN]) * gu[:, FFN:]
    return x + h @ layer.wd.t()


def _plan(doc_lens, n_link, q_len, device, prefix=0):
    """A one-query plan over a pool holding exactly the given documents."""
    lens = np.asarray(list(doc_lens), np.int32)
    starts = np.concatenate([[0], np.cumsum(lens[:-1])]).astype(np.int64) if len(lens) else np.zeros(0, np.int64)
    pool_len = lens if len(lens) else np.asarray([1], np.int32)
    pool_start = starts if len(lens) else np.zeros(1, np.int64)
    return LinkedPrefill(n_link=n_link, h_q=H_Q, h_kv=H_KV, head_dim=HEAD_DIM, theta=THETA,
                         pool_len=pool_len, pool_start=pool_start, pool_rows=int(pool_len.sum()),
                         prefix_doc=[-1], n_docs=[len(lens)], doc_ids=np.arange(len(lens), dtype=np.int32),
                         q_len=[q_len], device=device)


def _graphed(fn):
    """fn captured in a CUDA graph (launch overhead out of the measurement, for both arms)."""
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):  # warm-up outside capture: kernel attributes, cuBLAS handles
        fn()
        fn()
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        fn()
    return g.replay


CLOCKS = {}     # arm -> clock record of its last timed region (filled by _time)


def _time(fn, warmup=10, iters=40, arm=None, min_seconds=1.0):
    """ms per call from CUDA events around `iters` calls (raised so that the timed region lasts
    at least min_seconds), with the GPU clocks sampled during the timed region."""
    for _ in range(warmup):
        fn()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    e0.record()
    fn()
    e1.record()
    torch.cuda.synchronize()
    iters = max(iters, int(min_seconds * 1e3 / max(e0.elapsed_time(e1), 1e-3)) + 1)
    with ClockSampler(torch.cuda.current_device(), 50) as clk:
        torch.cuda.synchronize()
        clk.start()
        e0.record()
        for _ in range(iters):
            fn()
        e1.record()
        torch.cuda.synchronize()
        clk.stop()
    if arm is not None:
        CLOCKS[arm] = dict(clk.summary(), iters=iters)
    return e0.elapsed_time(e1) / iters


def layer_arms(doc_len, n_docs, n_link, q_len, host_caches, device, layer):
    """The two arms of the comparison on one layer, as callables (standard, linked), and a
    dict in which each run leaves what the library read and wrote: under "standard" the
    zero-document plan, q/k/v after RoPE and the attention output; under "linked" the plan,
    the document pool, q/k/v after RoPE, the linked cache and the attention output."""
    n_ctx = n_docs * doc_len + q_len
    seen = {}
    # ---- standard prefill: every token through the layer, causal attention over all of them
    std = _plan([], 0, n_ctx, device)
    x_std = torch.randn(n_ctx, HIDDEN, device=device, dtype=torch.bfloat16)
    ck_s, cv_s = std.empty_cache()
    out_s = torch.empty(n_ctx, H_Q, HEAD_DIM, device=device, dtype=torch.bfloat16)

    def standard():
        q, k, v = _qkv(layer, x_std)
        std.rope_fresh(q, k)
        std.suffix_attention(q, k, v, ck_s, cv_s, out_s)
        seen["standard"] = dict(plan=std, q=q, k=k, v=v, out=out_s)
        return _finish(layer, x_std, out_s)

    # ---- linked prefill: fresh link/question rows only, documents from the cache pool
    lp = _plan([doc_len] * n_docs, n_link, q_len, device)
    rows = n_docs * doc_len
    pool_k = torch.randn(rows, H_KV, HEAD_DIM, device=device, dtype=torch.bfloat16)
    pool_v = torch.randn(rows, H_KV, HEAD_DIM, device=device, dtype=torch.bfloat16)
    if host_caches:
        h_pool_k = pool_k.cpu().pin_memory()
        h_pool_v = pool_v.cpu().pin_memory()
    T = int(lp.info.n_fresh)
    x_new = torch.randn(T, HIDDEN, device=device, dtype=torch.bfloat16)
    ck, cv = lp.empty_cache()
    out = torch.empty(T, H_Q, HEAD_DIM, device=device, dtype=torch.bfloat16)

    def linked():
        if host_caches:  # the paper's setting: this layer's document caches start in CPU memory
            pool_k.copy_(h_pool_k, non_blocking=True)
            pool_v.copy_(h_pool_v, non_blocking=True)
        q, k, v = _qkv(layer, x_new)
        lp.rope_fresh(q, k)
        lp.linked_prefill(pool_k, pool_v, q, k, v, ck, cv, out)
        seen["linked"] = dict(plan=lp, pool_k=pool_k, pool_v=pool_v, q=q, k=k, v=v, cache_k=ck, cache_v=cv,
                              out=out, doc_len=doc_len, n_docs=n_docs, n_link=n_link, q_len=q_len)
        return _finish(layer, x_new, out)

    return standard, linked, seen, n_ctx, T


def measure(doc_len, n_docs, n_link, q_len, host_caches, device, layer):
    """ms per layer of (standard, linked) for n_docs documents of doc_len tokens."""
    standard, linked, _, n_ctx, T = layer_arms(doc_len, n_docs, n_link, q_len, host_caches, device, layer)
    t_std = _time(_graphed(standard), arm="standard")
    t_lnk = _time(_graphed(linked), arm="linked")
    assert K.kvlink_device_status() == 0
    return t_std, t_lnk, n_ctx, T


def measure_pipelined(doc_len, n_docs, n_link, q_len, device, layer, layers=LAYERS):
    """Whole-model TTFT (ms) of both arms with the linked arm's document caches in pinned host
    memory: every layer's caches are copied to the GPU on a copy stream into one of two device
    slots while the previous layer computes (Sec. 3.3: caches in CPU memory, loading counted
    in TTFT).  Each arm's `layers` layers run as one CUDA graph."""
    n_ctx = n_docs * doc_len + q_len
    std = _plan([], 0, n_ctx, device)
    x_std = torch.randn(n_ctx, HIDDEN, device=device, dtype=torch.bfloat16)
    ck_s, cv_s = std.empty_cache()
    out_s = torch.empty(n_ctx, H_Q, HEAD_DIM, device=device, dtype=torch.bfloat16)

    def standard():
        x = x_std
        for _ in range(layers):
            q, k, v = _qkv(layer, x)
            std.rope_fresh(q, k)
            std.suffix_attention(q, k, v, ck_s, cv_s, out_s)
            x = _finish(layer, x, out_s)
        return x

    lp = _plan([doc_len] * n_docs, n_link, q_len, device)
    rows = n_docs * doc_len
    gen = torch.Generator(device="cpu")
    gen.manual_seed(1)
    h_k = [torch.randn(rows, H_KV, HEAD_DIM, generator=gen).to(torch.bfloat16).pin_memory() for _ in range(layers)]
    h_v = [torch.randn(rows, H_KV, HEAD_DIM, generator=gen).to(torch.bfloat16).pin_memory() for _ in range(layers)]
    slot_k = [torch.empty(rows, H_KV, HEAD_DIM, device=device, dtype=torch.bfloat16) for _ in range(2)]
    slot_v = [torch.empty(rows, H_KV, HEAD_DIM, device=device, dtype=torch.bfloat16) for _ in range(2)]
    T = int(lp.info.n_fresh)
    x_new = torch.randn(T, HIDDEN, device=device, dtype=torch.bfloat16)
    ck, cv = lp.empty_cache()
    out = torch.empty(T, H_Q, HEAD_DIM, device=device, dtype=torch.bfloat16)
    copy_stream = torch.cuda.Stream(device)

    def linked():
        compute = torch.cuda.current_stream(device)
        done = [None, None]
        x = x_new
        for l in range(layers):
            b = l % 2
            copy_stream.wait_stream(compute) if done[b] is None else copy_stream.wait_event(done[b])
            with torch.cuda.stream(copy_stream):
                slot_k[b].copy_(h_k[l], non_blocking=True)
                slot_v[b].copy_(h_v[l], non_blocking=True)
                loaded = torch.cuda.Event()
                loaded.record(copy_stream)
            q, k, v = _qkv(layer, x)
            lp.rope_fresh(q, k)
            compute.wait_event(loaded)
            lp.linked_prefill(slot_k[b], slot_v[b], q, k, v, ck, cv, out)
            x = _finish(layer, x, out)
            done[b] = torch.cuda.Event()
            done[b].record(compute)
        compute.wait_stream(copy_stream)
        return x

    t_std = _time(_graphed(standard), warmup=3, iters=10, arm="standard")
    t_lnk = _time(_graphed(linked), warmup=3, iters=10, arm="linked")
    assert K.kvlink_device_status() == 0
    return t_std, t_lnk, n_ctx, T


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--lengths", type=int, nargs="+", default=[100, 200, 300, 400, 500])
    ap.add_argument("--links", type=int, nargs="+", default=[1, 5])
    ap.add_argument("--docs", type=int, default=10)
    ap.add_argument("--question", type=int, default=32)
    ap.add_argument("--host-caches", action="store_true")
    ap.add_argument("--pipelined", action="store_true",
                    help="whole model, caches in host memory, per-layer loading overlapped with compute")
    args = ap.parse_args()
    dev = torch.device("cuda:0")
    layer = Layer(dev)
    if args.pipelined:
        for n_link in args.links:
            for L in args.lengths:
                t_std, t_lnk, n_ctx, T = measure_pipelined(L, args.docs, n_link, args.question, dev, layer)
                print(json.dumps({
                    "workload": f"{args.docs} docs x {L} tokens, question {args.question}, KVLink{n_link}",
                    "context_tokens": n_ctx, "fresh_tokens": T, "ttft_standard_ms": round(t_std, 3),
                    "ttft_linked_ms": round(t_lnk, 3), "reduction_pct": round(100 * (1 - t_lnk / t_std), 1),
                    "caches": "pinned host memory, per-layer copies overlapped with the previous layer",
                    "layers": LAYERS, "shape": "Llama-3.1-8B, random bf16 weights, whole model in one graph",
                    "clocks": dict(CLOCKS)}), flush=True)
        return
    for n_link in args.links:
        for L in args.lengths:
            t_std, t_lnk, n_ctx, T = measure(L, args.docs, n_link, args.question, args.host_caches, dev, layer)
            print(json.dumps({
                "workload": f"{args.docs} docs x {L} tokens, question {args.question}, KVLink{n_link}",
                "context_tokens": n_ctx, "fresh_tokens": T,
                "ttft_standard_ms": round(t_std * LAYERS, 3), "ttft_linked_ms": round(t_lnk * LAYERS, 3),
                "reduction_pct": round(100 * (1 - t_lnk / t_std), 1),
                "caches": "pinned host memory, copied per layer" if args.host_caches else "resident in HBM",
                "layers": LAYERS, "shape": "Llama-3.1-8B, random bf16 weights", "clocks": dict(CLOCKS)}),
                flush=True)


if __name__ == "__main__":
    main()
