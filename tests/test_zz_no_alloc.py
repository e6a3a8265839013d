"""The allocation-free suffix attention (kvlink_suffix_attention_noalloc).

Some callers cannot allocate device memory: a serving loop whose memory budget is
fixed at start-up and may not call cudaMalloc on the request path, or code that
enqueues work where allocation is not permitted.  For them the library keeps the
split-KV scratch in a static device array.  These tests call that entry point
through the C ABI and check it against kvlink_suffix_attention (caller-owned
workspace) on two calls in a row, with different inputs, so that contents left in
the shared array by the first call cannot leak into the second.

This file is collected last so that a run stopping at the first failure has
already run every other test.
"""
import dataclasses

import numpy as np
import pytest

import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def env():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2502_16002_gb300 import kvlink as K
    from paper_2502_16002_gb300 import runtime as RT

    return K, RT


def _inputs(RT, batch, layer, dev):
    pk, pv = W.pool_kv(batch, layer)
    q, kn, vn = W.fresh_qkv(batch, layer)
    return [RT.bf16_from_bits(a, dev) for a in (pk, pv, q, kn, vn)]


def test_noalloc_matches_workspace_entry_point_on_two_calls(env):
    """Same kernels and same plan as kvlink_suffix_attention, so the outputs must be the
    same bits; the second call runs with other inputs over the scratch the first call
    left behind.  One query of each call is also checked against the fp64 oracle."""
    K, RT = env
    from _gpu_common import check_query

    from _gpu_common import EDGE, custom_batch

    dev = torch.device("cuda:0")
    # one 6000-token document and 50 fresh rows: 16 long M-tiles on 152 SMs, so the plan cuts
    # their KV ranges between CTAs and the partials go to the scratch
    name = "long_single_doc_split_kv"
    batch = custom_batch(50 + sorted(EDGE).index(name), **EDGE[name])
    lp = RT.LinkedPrefill.from_batch(batch, device=dev)
    info = lp.info
    assert info.n_attn_splits > 0, "the plan must use scratch for this test to mean anything"
    assert 0 < info.workspace_bytes <= K.KVLINK_NOALLOC_MAX_WORKSPACE_BYTES
    stream = torch.cuda.current_stream(dev)
    sh = int(stream.cuda_stream)
    for layer in (0, 1):                        # two calls in a row, different inputs
        pk, pv, q, kn, vn = _inputs(RT, batch, layer, dev)
        ck, cv = lp.empty_cache()
        lp.reencode_concat(pk, pv, ck, cv)
        ref = torch.full(lp.fresh_shape(batch.cfg.h_q), float("nan"), dtype=torch.bfloat16, device=dev)
        lp.suffix_attention(q, kn, vn, ck, cv, ref)
        got = torch.full_like(ref, float("nan"))
        K.kvlink_suffix_attention_noalloc(lp.plan, q.data_ptr(), kn.data_ptr(), vn.data_ptr(), ck.data_ptr(),
                                          cv.data_ptr(), got.data_ptr(), sh)
        torch.cuda.synchronize(dev)
        assert K.kvlink_device_status() == 0
        a, b = RT.bits_from_bf16(got), RT.bits_from_bf16(ref)
        assert np.all(np.isfinite(got.float().cpu().numpy()))
        assert np.array_equal(a, b), (layer, int((a != b).sum()))
        # the fp64 oracle on the allocation-free call's own output (query 0, every fresh row)
        check_query(batch, 0, lp, RT.bits_from_bf16(ck), RT.bits_from_bf16(cv),
                    got.float().cpu().numpy().astype(np.float64), tuple(W.pool_kv(batch, layer)) +
                    tuple(W.fresh_qkv(batch, layer)))


def test_noalloc_rejects_plans_larger_than_its_scratch(env):
    K, RT = env
    dev = torch.device("cuda:0")
    # 100 documents x 512 tokens and one 32-token question, no link tokens: 8 items for 152
    # SMs, so every KV range is split, into about 10 MB of partials
    base = W.draw_batch(W.get_config(4))
    batch = dataclasses.replace(base, cfg=dataclasses.replace(base.cfg, n_link=0),
                                q_len=np.asarray([32], np.int32))
    lp = RT.LinkedPrefill.from_batch(batch, device=dev, num_sms=152)
    assert lp.info.workspace_bytes > K.KVLINK_NOALLOC_MAX_WORKSPACE_BYTES
    T, Hq, Hkv, D = lp.info.n_fresh, batch.cfg.h_q, batch.cfg.h_kv, batch.cfg.head_dim
    q = torch.zeros((T, Hq, D), dtype=torch.bfloat16, device=dev)
    kn = torch.zeros((T, Hkv, D), dtype=torch.bfloat16, device=dev)
    ck, cv = lp.empty_cache()
    out = torch.zeros_like(q)
    with pytest.raises(K.KvlinkError) as e:
        K.kvlink_suffix_attention_noalloc(lp.plan, q.data_ptr(), kn.data_ptr(), kn.data_ptr(), ck.data_ptr(),
                                          cv.data_ptr(), out.data_ptr(), 0)
    assert e.value.code == K.KVLINK_ECAPACITY
