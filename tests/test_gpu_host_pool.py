"""GPU parity of the document cache pool kept in host memory (Sec. 3.3: caches in CPU memory,
loaded for every request).  kvlink_reencode_concat_host_pool reads the pool from page-locked
host memory and must write the same linked cache, bit for bit, as kvlink_reencode_concat from
a device copy of the same pool; kvlink_linked_prefill_layers_host_pool must give the same
caches and outputs as kvlink_linked_prefill_layers_overlapped.  Queries are also checked
against the fp64 oracle.
"""
import numpy as np
import pytest

import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from _gpu_common import EDGE, check_query, custom_batch  # noqa: E402


@pytest.fixture(scope="module")
def RT():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2502_16002_gb300 import runtime

    return runtime


def _batches():
    out = [("llama1b", W.draw_batch(W.get_config(2))), ("paged_serving", W.draw_batch(W.get_config(5)))]
    for name in ("doc_len_1_and_ragged", "multi_query_ragged", "gqa_8_single_kv_head", "no_link_tokens"):
        out.append((name, custom_batch(50 + sorted(EDGE).index(name), **EDGE[name])))
    return out


@pytest.mark.parametrize("name", [n for n, _ in _batches()])
def test_host_pool_reencode_equals_device_pool(RT, name):
    batch = dict(_batches())[name]
    dev = torch.device("cuda:0")
    pk, pv = W.pool_kv(batch, 0)
    q, kn, vn = W.fresh_qkv(batch, 0)
    lp = RT.LinkedPrefill.from_batch(batch, device=dev)
    h_pk, h_pv = RT.bf16_from_bits(pk).pin_memory(), RT.bf16_from_bits(pv).pin_memory()
    ck, cv = lp.empty_cache()
    ck.view(torch.int16).fill_(-1)
    cv.view(torch.int16).fill_(-1)
    lp.reencode_concat_host_pool(h_pk, h_pv, ck, cv)
    rk, rv = lp.empty_cache()
    rk.view(torch.int16).fill_(-1)
    rv.view(torch.int16).fill_(-1)
    lp.reencode_concat(h_pk.to(dev), h_pv.to(dev), rk, rv)
    torch.cuda.synchronize(dev)
    from paper_2502_16002_gb300 import kvlink as K
    assert K.kvlink_device_status() == 0
    assert torch.equal(ck.view(torch.int16), rk.view(torch.int16))
    assert torch.equal(cv.view(torch.int16), rv.view(torch.int16))
    # fresh rows and attention over the cache loaded from host memory, against the oracle
    out = torch.full(lp.fresh_shape(batch.cfg.h_q), float("nan"), dtype=torch.bfloat16, device=dev)
    lp.suffix_attention(RT.bf16_from_bits(q, dev), RT.bf16_from_bits(kn, dev), RT.bf16_from_bits(vn, dev), ck, cv,
                        out)
    torch.cuda.synchronize(dev)
    gout = out.float().cpu().numpy().astype(np.float64)
    for b in sorted({0, batch.cfg.batch - 1}):
        check_query(batch, b, lp, RT.bits_from_bf16(ck), RT.bits_from_bf16(cv), gout, (pk, pv, q, kn, vn))


@pytest.mark.parametrize("cfg_index,n_layers", [(2, 3), (5, 2)])
def test_layers_host_pool_equals_overlapped(RT, cfg_index, n_layers):
    from paper_2502_16002_gb300 import kvlink as K
    dev = torch.device("cuda:0")
    batch = W.draw_batch(W.get_config(cfg_index))
    lp = RT.LinkedPrefill.from_batch(batch, device=dev)
    raw = [W.pool_kv(batch, l) + W.fresh_qkv(batch, l) for l in range(n_layers)]
    h_pk = [RT.bf16_from_bits(r[0]).pin_memory() for r in raw]
    h_pv = [RT.bf16_from_bits(r[1]).pin_memory() for r in raw]
    q, kn, vn = ([RT.bf16_from_bits(r[i], dev) for r in raw] for i in (2, 3, 4))

    def run(host):
        caches = [lp.empty_cache() for _ in range(n_layers)]
        for ck, cv in caches:
            ck.view(torch.int16).fill_(-1)
            cv.view(torch.int16).fill_(-1)
        outs = [torch.full_like(x, float("nan")) for x in q]
        ks, vs = [c[0] for c in caches], [c[1] for c in caches]
        if host:
            lp.linked_prefill_layers_host_pool(h_pk, h_pv, q, kn, vn, ks, vs, outs)
        else:
            lp.linked_prefill_layers_overlapped([t.to(dev) for t in h_pk], [t.to(dev) for t in h_pv], q, kn, vn,
                                                ks, vs, outs)
        torch.cuda.synchronize(dev)
        return ks, vs, outs

    hk, hv, ho = run(True)
    dk, dv, do = run(False)
    assert K.kvlink_device_status() == 0
    for l in range(n_layers):
        assert torch.equal(hk[l].view(torch.int16), dk[l].view(torch.int16)), l
        assert torch.equal(hv[l].view(torch.int16), dv[l].view(torch.int16)), l
        assert torch.equal(ho[l].view(torch.int16), do[l].view(torch.int16)), l
    last = n_layers - 1
    check_query(batch, 0, lp, RT.bits_from_bf16(hk[last]), RT.bits_from_bf16(hv[last]),
                ho[last].float().cpu().numpy().astype(np.float64), raw[last])


def test_host_pool_rejects_pageable_and_device_memory(RT):
    from paper_2502_16002_gb300 import kvlink as K
    dev = torch.device("cuda:0")
    batch = W.draw_batch(W.get_config(1))
    lp = RT.LinkedPrefill.from_batch(batch, device=dev)
    pk, pv = W.pool_kv(batch, 0)
    ck, cv = lp.empty_cache()
    pageable_k, pageable_v = RT.bf16_from_bits(pk), RT.bf16_from_bits(pv)        # not pinned
    on_device = RT.bf16_from_bits(pk, dev)
    for a, b in ((pageable_k, pageable_v), (on_device, on_device)):
        with pytest.raises(K.KvlinkError) as e:
            K.kvlink_reencode_concat_host_pool(lp.plan, a.data_ptr(), b.data_ptr(), ck.data_ptr(), cv.data_ptr(), 0)
        assert e.value.code == K.KVLINK_EINVAL
