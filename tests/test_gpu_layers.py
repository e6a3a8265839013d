"""GPU check of the all-layers calls.  kvlink_linked_prefill_layers and
kvlink_linked_prefill_layers_overlapped (re-encode on a second stream) must give, for every
layer, exactly (bit for bit) what the per-layer kvlink_linked_prefill gives, and
kvlink_reencode_concat_layers exactly what kvlink_reencode_concat gives per layer,
including across the kernel's per-launch layer limit; one query of the last layer is
also checked against the fp64 oracle.
"""
import numpy as np
import pytest

import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from _gpu_common import check_query  # noqa: E402


@pytest.fixture(scope="module")
def RT():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2502_16002_gb300 import runtime

    return runtime


def _sentinel_cache(lp):
    ck, cv = lp.empty_cache()
    ck.view(torch.int16).fill_(-1)
    cv.view(torch.int16).fill_(-1)
    return ck, cv


@pytest.mark.parametrize("overlapped", [False, True])
@pytest.mark.parametrize("cfg_index,n_layers,layout", [(2, 3, 0), (5, 2, 0), (3, 2, 1)])
def test_all_layers_call_equals_per_layer_calls(RT, cfg_index, n_layers, layout, overlapped):
    from paper_2502_16002_gb300 import kvlink as K
    dev = torch.device("cuda:0")
    batch = W.draw_batch(W.get_config(cfg_index))
    pk, pv, q, kn, vn, raw = [], [], [], [], [], []
    for layer in range(n_layers):
        a, b = W.pool_kv(batch, layer)
        x, y, z = W.fresh_qkv(batch, layer)
        raw.append((a, b, x, y, z))
        for lst, arr in zip((pk, pv, q, kn, vn), (a, b, x, y, z)):
            lst.append(RT.bf16_from_bits(arr, dev))
    lp = RT.LinkedPrefill.from_batch(batch, device=dev, layout=layout)
    caches = [_sentinel_cache(lp) for _ in range(n_layers)]
    outs = [torch.full_like(x, float("nan")) for x in q]
    if overlapped:      # the re-encode on a second stream
        lp.linked_prefill_layers_overlapped(pk, pv, q, kn, vn, [c[0] for c in caches], [c[1] for c in caches], outs)
    else:
        lp.linked_prefill_layers(pk, pv, q, kn, vn, [c[0] for c in caches], [c[1] for c in caches], outs)
    for layer in range(n_layers):
        ck, cv = _sentinel_cache(lp)
        ref = torch.full_like(q[layer], float("nan"))
        lp.linked_prefill(pk[layer], pv[layer], q[layer], kn[layer], vn[layer], ck, cv, ref)
        torch.cuda.synchronize()
        assert torch.equal(outs[layer].view(torch.int16), ref.view(torch.int16)), layer
        assert torch.equal(caches[layer][0].view(torch.int16), ck.view(torch.int16)), layer
        assert torch.equal(caches[layer][1].view(torch.int16), cv.view(torch.int16)), layer
    assert K.kvlink_device_status() == 0
    last = n_layers - 1
    gk, gv = RT.bits_from_bf16(caches[last][0]), RT.bits_from_bf16(caches[last][1])
    gout = outs[last].float().cpu().numpy().astype(np.float64)
    check_query(batch, 0, lp, gk, gv, gout, raw[last], layout=layout)


@pytest.mark.parametrize("cfg_index,n_layers", [(1, 70), (2, 5), (5, 3)])
def test_reencode_layers_call_equals_per_layer_calls(RT, cfg_index, n_layers):
    """70 layers of the two-document workload cross the 64-layers-per-launch limit; the
    paged pool (workload 5) resolves its block tables per unit."""
    from paper_2502_16002_gb300 import kvlink as K
    dev = torch.device("cuda:0")
    batch = W.draw_batch(W.get_config(cfg_index))
    lp = RT.LinkedPrefill.from_batch(batch, device=dev)
    c = batch.cfg
    shape = ((batch.pool_rows // c.pool_block_size, c.pool_block_size, c.h_kv, c.head_dim) if c.pool_block_size
             else (batch.pool_rows, c.h_kv, c.head_dim))
    pk = [W.normal_bf16_torch(shape, 7000 + 2 * l, dev) for l in range(n_layers)]
    pv = [W.normal_bf16_torch(shape, 7001 + 2 * l, dev) for l in range(n_layers)]
    caches = [_sentinel_cache(lp) for _ in range(n_layers)]
    lp.reencode_concat_layers(pk, pv, [c[0] for c in caches], [c[1] for c in caches])
    torch.cuda.synchronize()
    for layer in range(n_layers):
        ck, cv = _sentinel_cache(lp)
        lp.reencode_concat(pk[layer], pv[layer], ck, cv)
        torch.cuda.synchronize()
        assert torch.equal(caches[layer][0].view(torch.int16), ck.view(torch.int16)), layer
        assert torch.equal(caches[layer][1].view(torch.int16), cv.view(torch.int16)), layer
    assert K.kvlink_device_status() == 0


def test_pipelined_host_path_chains_calls(RT):
    """Two batches through linked_prefill_layers_from_host(wait=False) on one object and one
    set of device buffers, the plan rebuilt for the second while the first runs: each call's
    host outputs must equal the per-layer kvlink_linked_prefill of its own inputs, bit for bit
    (the second call overwrites q, k_new, v_new and out only after the first is done with them)."""
    dev = torch.device("cuda:0")
    n_layers = 3
    ba, bb = W.draw_batch(W.get_config(2)), W.draw_batch(W.get_config(2), seed=7)
    lp = RT.LinkedPrefill.from_batch(ba, device=dev)
    T = max(int(lp.info.n_fresh), int(RT.LinkedPrefill.from_batch(bb, device=dev).info.n_fresh))
    cfg = ba.cfg

    def host_inputs(batch):
        xs = [W.fresh_qkv(batch, l) for l in range(n_layers)]
        pad = lambda a: np.pad(a, ((0, T - a.shape[0]),) + ((0, 0),) * (a.ndim - 1))
        return [torch.stack([RT.bf16_from_bits(pad(x[i]), None) for x in xs]).pin_memory() for i in range(3)]

    pools = {id(b): [W.pool_kv(b, l) for l in range(n_layers)] for b in (ba, bb)}
    pk = {k: [RT.bf16_from_bits(p[0], dev) for p in v] for k, v in pools.items()}
    pv = {k: [RT.bf16_from_bits(p[1], dev) for p in v] for k, v in pools.items()}
    hin = {id(b): host_inputs(b) for b in (ba, bb)}
    q = torch.empty((n_layers, T, cfg.h_q, cfg.head_dim), dtype=torch.bfloat16, device=dev)
    kn = torch.empty((n_layers, T, cfg.h_kv, cfg.head_dim), dtype=torch.bfloat16, device=dev)
    vn = torch.empty_like(kn)
    ctx = max(int(lp.info.ctx_rows), int(RT.LinkedPrefill.from_batch(bb, device=dev).info.ctx_rows))
    ck = torch.empty((n_layers, ctx, cfg.h_kv, cfg.head_dim), dtype=torch.bfloat16, device=dev)
    cv = torch.empty_like(ck)
    out = torch.empty_like(q)
    h_out = {id(b): torch.empty(out.shape, dtype=out.dtype, pin_memory=True) for b in (ba, bb)}
    streams = (torch.cuda.Stream(dev), torch.cuda.current_stream(dev), torch.cuda.Stream(dev))
    for b in (ba, bb):
        if b is bb:
            lp.rebuild_from_batch(bb, stream=streams[1])
        h_q, h_kn, h_vn = hin[id(b)]
        lp.linked_prefill_layers_from_host(pk[id(b)], pv[id(b)], h_q, h_kn, h_vn, q, kn, vn, ck, cv, out,
                                           h_out[id(b)], streams=streams, wait=False)
    torch.cuda.synchronize(dev)
    from paper_2502_16002_gb300 import kvlink as K
    assert K.kvlink_device_status() == 0
    for b in (ba, bb):
        ref_lp = RT.LinkedPrefill.from_batch(b, device=dev)
        n = int(ref_lp.info.n_fresh)
        h_q, h_kn, h_vn = hin[id(b)]
        for l in range(n_layers):
            c_k, c_v = ref_lp.empty_cache()
            ref = torch.empty(ref_lp.fresh_shape(cfg.h_q), dtype=torch.bfloat16, device=dev)
            ref_lp.linked_prefill(pk[id(b)][l], pv[id(b)][l], h_q[l, :n].to(dev), h_kn[l, :n].to(dev),
                                  h_vn[l, :n].to(dev), c_k, c_v, ref)
            torch.cuda.synchronize(dev)
            assert torch.equal(h_out[id(b)][l, :n].view(torch.int16), ref.cpu().view(torch.int16)), (l,)


def test_host_path_calls_with_different_layer_counts(RT):
    """Host-path calls of 4, then 2, then 4 layers, enqueued back to back (wait=False) on one
    plan and one set of device buffers, each with its own inputs: a call whose layer count
    differs from the previous one must still rewrite the shared device inputs, caches and
    outputs only after the previous call is done with them.  Every call's host outputs must
    equal per-layer kvlink_linked_prefill of its own inputs, bit for bit; the last layer of
    the last call is also checked against the fp64 oracle."""
    from paper_2502_16002_gb300 import kvlink as K
    dev = torch.device("cuda:0")
    batch = W.draw_batch(W.get_config(2))
    cfg = batch.cfg
    lp = RT.LinkedPrefill.from_batch(batch, device=dev)
    calls = [list(range(0, 4)), list(range(4, 6)), list(range(6, 10))]   # source layer of every slot
    raw = {l: W.pool_kv(batch, l) + W.fresh_qkv(batch, l) for c in calls for l in c}
    T = int(lp.info.n_fresh)
    q = torch.empty((4, T, cfg.h_q, cfg.head_dim), dtype=torch.bfloat16, device=dev)
    kn = torch.empty((4, T, cfg.h_kv, cfg.head_dim), dtype=torch.bfloat16, device=dev)
    vn = torch.empty_like(kn)
    ck = torch.empty((4,) + lp.cache_shape(), dtype=torch.bfloat16, device=dev)
    cv = torch.empty_like(ck)
    out = torch.empty_like(q)
    streams = (torch.cuda.Stream(dev), torch.cuda.current_stream(dev), torch.cuda.Stream(dev))
    results = []
    for c in calls:
        n = len(c)
        pk = [RT.bf16_from_bits(raw[l][0], dev) for l in c]
        pv = [RT.bf16_from_bits(raw[l][1], dev) for l in c]
        h_q, h_kn, h_vn = (torch.stack([RT.bf16_from_bits(raw[l][i], None) for l in c]).pin_memory()
                           for i in (2, 3, 4))
        h_out = torch.empty((n, T, cfg.h_q, cfg.head_dim), dtype=torch.bfloat16, pin_memory=True)
        lp.linked_prefill_layers_from_host(pk, pv, h_q, h_kn, h_vn, q[:n], kn[:n], vn[:n], ck[:n], cv[:n],
                                           out[:n], h_out, streams=streams, wait=False)
        results.append((c, pk, pv, h_q, h_kn, h_vn, h_out))
    torch.cuda.synchronize(dev)
    assert K.kvlink_device_status() == 0
    for c, pk, pv, h_q, h_kn, h_vn, h_out in results:
        for i, l in enumerate(c):
            c_k, c_v = lp.empty_cache()
            ref = torch.empty(lp.fresh_shape(cfg.h_q), dtype=torch.bfloat16, device=dev)
            lp.linked_prefill(pk[i], pv[i], h_q[i].to(dev), h_kn[i].to(dev), h_vn[i].to(dev), c_k, c_v, ref)
            torch.cuda.synchronize(dev)
            assert torch.equal(h_out[i].view(torch.int16), ref.cpu().view(torch.int16)), (c, l)
    c, *_, h_out = results[-1]
    gk, gv = RT.bits_from_bf16(ck[len(c) - 1]), RT.bits_from_bf16(cv[len(c) - 1])
    check_query(batch, 0, lp, gk, gv, h_out[len(c) - 1].float().numpy().astype(np.float64), raw[c[-1]])


@pytest.mark.parametrize("zero_copy", [False, True])
def test_overlapped_call_replays_from_a_cuda_graph(RT, zero_copy):
    """The step's call captured once in a CUDA graph (its second stream and events joined into
    the capture) and replayed: every layer's cache and output equal a direct call's, bit for
    bit, on two replays (the attention's merge counters keep growing across launches)."""
    from paper_2502_16002_gb300 import kvlink as K
    dev = torch.device("cuda:0")
    batch = W.draw_batch(W.get_config(2))       # workload 2 cuts KV ranges: in-kernel merges
    L = 3
    lp = RT.LinkedPrefill.from_batch(batch, device=dev)
    t = {}
    for name, seq in (("pk", []), ("pv", []), ("q", []), ("kn", []), ("vn", [])):
        t[name] = seq
    for layer in range(L):
        a, b = W.pool_kv(batch, layer)
        x, y, z = W.fresh_qkv(batch, layer)
        for name, arr in zip(("pk", "pv", "q", "kn", "vn"), (a, b, x, y, z)):
            t[name].append(RT.bf16_from_bits(arr, dev))

    def buffers():
        caches = [_sentinel_cache(lp) for _ in range(L)]
        outs = [torch.full(lp.fresh_shape(batch.cfg.h_q), float("nan"), dtype=torch.bfloat16, device=dev)
                for _ in range(L)]
        return caches, outs

    ref_c, ref_o = buffers()
    lp.linked_prefill_layers_overlapped(t["pk"], t["pv"], t["q"], t["kn"], t["vn"], [c[0] for c in ref_c],
                                        None if zero_copy else [c[1] for c in ref_c], ref_o)
    torch.cuda.synchronize()
    g_c, g_o = buffers()
    s = torch.cuda.Stream(dev)
    re_s = torch.cuda.Stream(dev)
    s.wait_stream(torch.cuda.current_stream(dev))
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=s):
        lp.linked_prefill_layers_overlapped(t["pk"], t["pv"], t["q"], t["kn"], t["vn"], [c[0] for c in g_c],
                                            None if zero_copy else [c[1] for c in g_c], g_o, stream=s,
                                            reencode_stream=re_s)
    for _ in range(2):
        for c, o in zip(g_c, g_o):
            c[0].view(torch.int16).fill_(-1)
            c[1].view(torch.int16).fill_(-1)
            o.fill_(float("nan"))
        torch.cuda.synchronize()
        graph.replay()
        torch.cuda.synchronize()
        assert K.kvlink_device_status() == 0
        for layer in range(L):
            assert torch.equal(ref_c[layer][0].view(torch.int16), g_c[layer][0].view(torch.int16))
            if not zero_copy:
                assert torch.equal(ref_c[layer][1].view(torch.int16), g_c[layer][1].view(torch.int16))
            assert torch.equal(ref_o[layer].view(torch.int16), g_o[layer].view(torch.int16))
