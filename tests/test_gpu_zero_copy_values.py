"""Zero-copy values on the two-kernel path (cache_v NULL), through the C ABI.

Sec. 2.3 ("inference") concatenates the cached values unchanged, so they need not be
copied: with cache_v NULL the re-encode writes keys only and the persistent attention reads
every value row where it already is (the pool's rows for the prefix and the documents, v_new
for the link and question rows), through the plan's 8-row group table and row-by-row copies
at segment boundaries.  Checks:
  - the keys are within one bf16 ulp of the fp64 oracle (the keys-only re-encode rotates with
    a faster form than the value path, so the two may round a key one ulp apart: within one
    ulp of each other too);
  - the attention over those keys equals, bit for bit, the value-cache attention
    (kvlink_suffix_attention) run on the same keys with the value cache built by the value
    path: the same tiles and the same order of operations, only the value rows come from
    elsewhere;
  - the output is within the attention tolerance of the fp64 oracle (max |err| <= 1e-2,
    mean |err| <= 1e-3).
"""
import numpy as np
import pytest

import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from _gpu_common import EDGE, LAYOUTS, check_query, custom_batch, ulp_distance  # noqa: E402


@pytest.fixture(scope="module")
def RT():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2502_16002_gb300 import runtime

    return runtime


def _both(RT, batch, layer, layout=0):
    """One layer with the value cache and with zero-copy values.  Returns what
    _gpu_common.check_query takes for the zero-copy run (value bits None)."""
    from paper_2502_16002_gb300 import kvlink as K
    dev = torch.device("cuda:0")
    pk, pv = W.pool_kv(batch, layer)
    q, kn, vn = W.fresh_qkv(batch, layer)
    t = {k: RT.bf16_from_bits(v, dev) for k, v in dict(pk=pk, pv=pv, q=q, kn=kn, vn=vn).items()}
    lp = RT.LinkedPrefill.from_batch(batch, device=dev, layout=layout)
    ck, cv = lp.empty_cache()
    ck.view(torch.int16).fill_(-1)
    cv.view(torch.int16).fill_(-1)
    out = torch.full(lp.fresh_shape(batch.cfg.h_q), float("nan"), dtype=torch.bfloat16, device=dev)
    lp.linked_prefill(t["pk"], t["pv"], t["q"], t["kn"], t["vn"], ck, cv, out)
    zk = torch.empty_like(ck)
    zk.view(torch.int16).fill_(-1)
    zout = torch.full_like(out, float("nan"))
    lp.linked_prefill(t["pk"], t["pv"], t["q"], t["kn"], t["vn"], zk, None, zout)
    # the value-cache attention over the zero-copy keys
    same = torch.full_like(out, float("nan"))
    lp.suffix_attention(t["q"], None, None, zk, cv, same)
    torch.cuda.synchronize(dev)
    assert K.kvlink_device_status() == 0
    gk, gz = RT.bits_from_bf16(ck), RT.bits_from_bf16(zk)
    assert ulp_distance(gk, gz).max() <= 1, "keys more than one ulp from the value path's"
    assert torch.equal(same.view(torch.int16), zout.view(torch.int16)), "attention differs from the value-cache path"
    zo = zout.float().cpu().numpy().astype(np.float64)
    return lp, gz, None, zo, (pk, pv, q, kn, vn)


@pytest.mark.parametrize("layout", sorted(LAYOUTS))
@pytest.mark.parametrize("name", sorted(EDGE))
def test_edge_cases(RT, name, layout):
    batch = custom_batch(50 + sorted(EDGE).index(name), **EDGE[name])
    lp, gk, gv, gout, inp = _both(RT, batch, 0, LAYOUTS[layout])
    for b in range(batch.cfg.batch):
        check_query(batch, b, lp, gk, gv, gout, inp, layout=LAYOUTS[layout])


@pytest.mark.parametrize("cfg_index", [1, 2])
def test_small_workloads_in_full(RT, cfg_index):
    batch = W.draw_batch(W.get_config(cfg_index))
    lp, gk, gv, gout, inp = _both(RT, batch, 0)
    for b in range(batch.cfg.batch):
        check_query(batch, b, lp, gk, gv, gout, inp)


@pytest.mark.parametrize("layout", sorted(LAYOUTS))
def test_llama8b_batch8_zipf(RT, layout):
    batch = W.draw_batch(W.get_config(3))
    lp, gk, gv, gout, inp = _both(RT, batch, 31, LAYOUTS[layout])
    for b in (0, 3, 7):
        check_query(batch, b, lp, gk, gv, gout, inp, layout=LAYOUTS[layout])


def test_llama8b_long_context(RT):
    batch = W.draw_batch(W.get_config(4))
    lp, gk, gv, gout, inp = _both(RT, batch, 0)
    T = int(batch.n_fresh[0])
    rows = [0, 1, 4, 5, 9, 31, 32, 127, 128, 255, 256, 499, 500, 501] + list(range(600, T))
    check_query(batch, 0, lp, gk, gv, gout, inp, rows=rows)


def test_llama8b_paged_serving(RT):
    """Paged pool: 8-row groups that cross a pool block are copied row by row."""
    batch = W.draw_batch(W.get_config(5))
    lp, gk, gv, gout, inp = _both(RT, batch, 0)
    for b in (0, 31, 63):
        check_query(batch, b, lp, gk, gv, gout, inp)


def _layer_tensors(RT, batch, L, dev):
    pk, pv, q, kn, vn = [], [], [], [], []
    for layer in range(L):
        a, b = W.pool_kv(batch, layer)
        x, y, z = W.fresh_qkv(batch, layer)
        pk.append(RT.bf16_from_bits(a, dev))
        pv.append(RT.bf16_from_bits(b, dev))
        q.append(RT.bf16_from_bits(x, dev))
        kn.append(RT.bf16_from_bits(y, dev))
        vn.append(RT.bf16_from_bits(z, dev))
    return pk, pv, q, kn, vn


def test_overlapped_layers(RT):
    """The step's call with cache_v NULL: keys within one ulp of the value-cache call's, and per
    layer the same output bits as the value-cache attention over those keys."""
    batch = W.draw_batch(W.get_config(3))
    dev = torch.device("cuda:0")
    L = 3
    lp = RT.LinkedPrefill.from_batch(batch, device=dev)
    pk, pv, q, kn, vn = _layer_tensors(RT, batch, L, dev)
    runs = []
    for with_v in (True, False):
        caches = [lp.empty_cache() for _ in range(L)]
        out = [torch.empty(lp.fresh_shape(batch.cfg.h_q), dtype=torch.bfloat16, device=dev) for _ in range(L)]
        lp.linked_prefill_layers_overlapped(pk, pv, q, kn, vn, [c[0] for c in caches],
                                            [c[1] for c in caches] if with_v else None, out)
        torch.cuda.synchronize()
        runs.append(([c[0] for c in caches], out))
        if with_v:
            values = [c[1] for c in caches]
    from paper_2502_16002_gb300 import kvlink as K
    assert K.kvlink_device_status() == 0
    for layer in range(L):
        zk, zout = runs[1][0][layer], runs[1][1][layer]
        assert ulp_distance(RT.bits_from_bf16(runs[0][0][layer]), RT.bits_from_bf16(zk)).max() <= 1
        same = torch.full_like(zout, float("nan"))
        lp.suffix_attention(q[layer], None, None, zk, values[layer], same)
        torch.cuda.synchronize()
        assert torch.equal(same.view(torch.int16), zout.view(torch.int16))


def test_suffix_attention_pool_values(RT):
    """kvlink_reencode_concat (keys only) + kvlink_suffix_attention_pool_values equal the
    separate calls with a value cache, with the fresh keys placed by the call or beforehand."""
    batch = W.draw_batch(W.get_config(2))
    dev = torch.device("cuda:0")
    pk, pv, q, kn, vn = [x[0] for x in _layer_tensors(RT, batch, 1, dev)]
    lp = RT.LinkedPrefill.from_batch(batch, device=dev)
    ck, cv = lp.empty_cache()
    ref = torch.empty(lp.fresh_shape(batch.cfg.h_q), dtype=torch.bfloat16, device=dev)
    lp.reencode_concat(pk, pv, ck, cv)
    lp.suffix_attention(q, kn, vn, ck, cv, ref)
    ck2 = torch.empty_like(ck)
    ck2.view(torch.int16).fill_(-1)
    out = torch.full_like(ref, float("nan"))
    lp.reencode_concat(pk, None, ck2, None)
    lp.suffix_attention_pool_values(q, kn, vn, pv, ck2, out)
    # the value-cache attention over the keys-only cache (its fresh rows are placed now)
    ref = torch.full_like(out, float("nan"))
    lp.suffix_attention(q, None, None, ck2, cv, ref)
    torch.cuda.synchronize()
    assert ulp_distance(RT.bits_from_bf16(ck), RT.bits_from_bf16(ck2)).max() <= 1
    assert torch.equal(ref.view(torch.int16), out.view(torch.int16))
    # fresh keys already in the cache: k_new NULL
    out2 = torch.full_like(ref, float("nan"))
    lp.suffix_attention_pool_values(q, None, vn, pv, ck2, out2)
    torch.cuda.synchronize()
    assert torch.equal(ref.view(torch.int16), out2.view(torch.int16))


def test_reencode_layers_keys_only(RT):
    batch = W.draw_batch(W.get_config(2))
    dev = torch.device("cuda:0")
    L = 2
    pk, pv, _, _, _ = _layer_tensors(RT, batch, L, dev)
    lp = RT.LinkedPrefill.from_batch(batch, device=dev)
    full = [lp.empty_cache() for _ in range(L)]
    keys = [lp.empty_cache()[0] for _ in range(L)]
    for c in [f[0] for f in full] + keys:
        c.view(torch.int16).fill_(-1)
    lp.reencode_concat_layers(pk, pv, [f[0] for f in full], [f[1] for f in full])
    lp.reencode_concat_layers(pk, None, keys, None)
    torch.cuda.synchronize()
    for layer in range(L):
        # the keys-only launch rotates with the fast form: within one ulp of the value path's
        assert ulp_distance(RT.bits_from_bf16(full[layer][0]), RT.bits_from_bf16(keys[layer])).max() <= 1


def test_host_path(RT):
    """kvlink_linked_prefill_layers_host with cache_v NULL: per layer, the output on the host
    equals the value-cache attention over the call's keys, with the value cache of the same
    call made with cache_v."""
    batch = W.draw_batch(W.get_config(2))
    dev = torch.device("cuda:0")
    L = 2
    lp = RT.LinkedPrefill.from_batch(batch, device=dev)
    pk, pv, q, kn, vn = _layer_tensors(RT, batch, L, dev)
    qh = [t.cpu().pin_memory() for t in q]
    kh = [t.cpu().pin_memory() for t in kn]
    vh = [t.cpu().pin_memory() for t in vn]
    runs = []
    for with_v in (True, False):
        dq = [torch.empty_like(t) for t in q]
        dk = [torch.empty_like(t) for t in kn]
        dv = [torch.empty_like(t) for t in vn]
        caches = [lp.empty_cache() for _ in range(L)]
        dout = [torch.empty_like(t) for t in q]
        hout = [torch.empty(t.shape, dtype=torch.bfloat16).pin_memory() for t in q]
        lp.linked_prefill_layers_from_host(pk, pv, qh, kh, vh, dq, dk, dv, [c[0] for c in caches],
                                           [c[1] for c in caches] if with_v else None, dout, hout)
        runs.append((caches, hout))
    for layer in range(L):
        zk, hz = runs[1][0][layer][0], runs[1][1][layer]
        same = torch.full_like(q[layer], float("nan"))
        lp.suffix_attention(q[layer], None, None, zk, runs[0][0][layer][1], same)
        torch.cuda.synchronize()
        assert torch.equal(same.cpu().view(torch.int16), hz.view(torch.int16))
