"""GPU parity of the linked prefill against the fp64 oracle, through the C ABI.

Tolerances: segment tables bit-exact (tests/test_abi_cpu.py); re-encoded keys
within 1 bf16 ulp of the oracle's correctly rounded fp64 rotation; values,
prefix and fresh rows bit-exact; attention output max |err| <= 1e-2 and mean
|err| <= 1e-3 against the fp64 oracle.
"""
import dataclasses

import numpy as np
import pytest

import oracle as O
import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

MAX_ABS, MEAN_ABS = 1e-2, 1e-3


@pytest.fixture(scope="module")
def RT():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2502_16002_gb300 import runtime

    return runtime


def ulp_distance(a: np.ndarray, b: np.ndarray) -> np.ndarray:
    """Distance between bf16 bit patterns in representable steps (+0 and -0 equal)."""
    def ordinal(u):
        u = u.astype(np.int32)
        return np.where(u & 0x8000, -(u & 0x7FFF), u)
    return np.abs(ordinal(a) - ordinal(b))


def run_layer(RT, batch, layer, mode="fused", rows=None):
    """Run one layer on the GPU.  Returns (lp, cache_k bits, cache_v bits, out float64, inputs)."""
    dev = torch.device("cuda:0")
    pk, pv = W.pool_kv(batch, layer)
    q, kn, vn = W.fresh_qkv(batch, layer)
    lp = RT.LinkedPrefill.from_batch(batch, device=dev)
    ck, cv = lp.empty_cache()
    ck.view(torch.int16).fill_(-1)   # NaN sentinel: every slot must be written
    cv.view(torch.int16).fill_(-1)
    out = torch.full(lp.fresh_shape(batch.cfg.h_q), float("nan"), dtype=torch.bfloat16, device=dev)
    t = {k: RT.bf16_from_bits(v, dev) for k, v in dict(pk=pk, pv=pv, q=q, kn=kn, vn=vn).items()}
    if mode == "fused":
        lp.linked_prefill(t["pk"], t["pv"], t["q"], t["kn"], t["vn"], ck, cv, out)
    else:
        lp.reencode_concat(t["pk"], t["pv"], ck, cv)
        lp.suffix_attention(t["q"], t["kn"], t["vn"], ck, cv, out)
    torch.cuda.synchronize(dev)
    from paper_2502_16002_gb300 import kvlink as K
    assert K.kvlink_device_status() == 0
    return (lp, RT.bits_from_bf16(ck), RT.bits_from_bf16(cv), out.float().cpu().numpy().astype(np.float64),
            (pk, pv, q, kn, vn))


def check_query(batch, b, lp, gk, gv, gout, inputs, rows=None, attention=True):
    from paper_2502_16002_gb300 import kvlink as K
    pk, pv, q, kn, vn = inputs
    cu_ctx, cu_fresh = K.kvlink_plan_get_offsets(lp.plan)
    nf = batch.n_fresh
    r0 = int(nf[:b].sum())
    r1 = r0 + int(nf[b])
    assert cu_fresh[b] == r0 and cu_fresh[b + 1] == r1
    cache = O.reencode_concat(pk, pv, batch.pool_start, batch.pool_len, int(batch.prefix_doc[b]),
                              [int(d) for d in batch.docs_of(b)], batch.cfg.n_link, kn[r0:r1], vn[r0:r1],
                              int(batch.q_len[b]), batch.cfg.theta, block_table=batch.pool_block_table,
                              block_size=batch.cfg.pool_block_size)
    c0, c1 = int(cu_ctx[b]), int(cu_ctx[b + 1])
    assert c1 - c0 == cache.layout.total
    k_gpu, v_gpu = gk[c0:c1], gv[c0:c1]
    assert np.array_equal(v_gpu, cache.v_bits), "V concat not bit-exact"
    d = ulp_distance(k_gpu, cache.k_bits)
    assert d.max() <= 1, f"re-encoded K off by {d.max()} ulp"
    not_doc = cache.layout.kind != O.DOC
    assert np.array_equal(k_gpu[not_doc], cache.k_bits[not_doc]), "prefix/fresh K not bit-exact"
    if not attention:
        return None
    sel = np.arange(r1 - r0) if rows is None else np.asarray(rows)
    ref = O.suffix_attention(O.bf16_bits_to_f64(q[r0:r1][sel]), O.bf16_bits_to_f64(cache.k_bits),
                             O.bf16_bits_to_f64(cache.v_bits), cache.layout.fresh_pos[sel])
    got = gout[r0:r1][sel]
    assert np.all(np.isfinite(got))
    err = np.abs(got - ref)
    assert err.max() <= MAX_ABS and err.mean() <= MEAN_ABS, (err.max(), err.mean())
    return err.max(), err.mean()


# ----------------------------------------------------------------- small workloads, in full

@pytest.mark.parametrize("mode", ["fused", "separate"])
def test_tiny_two_documents(RT, mode):
    batch = W.draw_batch(W.get_config(1))
    lp, gk, gv, gout, inp = run_layer(RT, batch, 0, mode)
    check_query(batch, 0, lp, gk, gv, gout, inp)


@pytest.mark.parametrize("layer", [0, 15])
def test_llama1b_ten_documents(RT, layer):
    batch = W.draw_batch(W.get_config(2))
    lp, gk, gv, gout, inp = run_layer(RT, batch, layer)
    check_query(batch, 0, lp, gk, gv, gout, inp)


# ----------------------------------------------------------------- edge cases

def custom_batch(index, *, h_q, h_kv, D, n_link, prefix, doc_lens_per_query, q_lens, theta=500000.0,
                 pool_block_size=0, seed=0):
    """A batch whose pool holds exactly the listed documents (plus one prefix entry)."""
    lens = [L for q in doc_lens_per_query for L in q]
    cfg = W.WorkloadConfig(index=index, name=f"edge{index}", batch=len(q_lens), layers=1, h_q=h_q,
                           h_kv=h_kv, head_dim=D, theta=theta, prefix_len=prefix, n_link=n_link,
                           docs_per_query=0, pool_docs=len(lens), pool_block_size=pool_block_size)
    pool_len = np.asarray(lens + ([prefix] if prefix else []), np.int32)
    ids, off = [], 0
    for q in doc_lens_per_query:
        ids.extend(range(off, off + len(q)))
        off += len(q)
    if pool_block_size:
        nblk = (pool_len.astype(np.int64) + pool_block_size - 1) // pool_block_size
        rng = np.random.default_rng(index)
        bt = rng.permutation(int(nblk.sum())).astype(np.int32)
        pool_start = np.concatenate([[0], np.cumsum(nblk)[:-1]]).astype(np.int64)
        rows = int(nblk.sum()) * pool_block_size
    else:
        bt = None
        pool_start = np.concatenate([[0], np.cumsum(pool_len.astype(np.int64))[:-1]]).astype(np.int64)
        rows = int(pool_len.sum())
    B = len(q_lens)
    return W.Batch(cfg=cfg, seed=seed, pool_len=pool_len, pool_start=pool_start, pool_block_table=bt,
                   pool_rows=rows, prefix_doc=np.full(B, len(lens) if prefix else -1, np.int32),
                   n_docs=np.asarray([len(q) for q in doc_lens_per_query], np.int32),
                   doc_ids=np.asarray(ids, np.int32), q_len=np.asarray(q_lens, np.int32))


EDGE = {
    "doc_len_1_and_ragged": dict(h_q=8, h_kv=2, D=128, n_link=5, prefix=0,
                                 doc_lens_per_query=[[1, 17, 33, 127, 129]], q_lens=[9]),
    "no_link_tokens": dict(h_q=8, h_kv=2, D=64, n_link=0, prefix=3,
                           doc_lens_per_query=[[40, 41, 42]], q_lens=[7]),
    "one_doc_question_len_1": dict(h_q=4, h_kv=4, D=128, n_link=1, prefix=0,
                                   doc_lens_per_query=[[200]], q_lens=[1]),
    "gqa_8_single_kv_head": dict(h_q=8, h_kv=1, D=64, n_link=2, prefix=5,
                                 doc_lens_per_query=[[70, 3]], q_lens=[30]),
    "gqa_16_head_dim_128": dict(h_q=32, h_kv=2, D=128, n_link=5, prefix=0,
                                doc_lens_per_query=[[100, 50]], q_lens=[20]),
    "multi_query_ragged": dict(h_q=32, h_kv=8, D=128, n_link=5, prefix=16,
                               doc_lens_per_query=[[13, 250, 77], [5], [300, 1, 64, 64]],
                               q_lens=[33, 1, 70]),
    "long_single_doc_split_kv": dict(h_q=32, h_kv=8, D=128, n_link=5, prefix=0,
                                     doc_lens_per_query=[[6000, 300]], q_lens=[40]),
    "paged_pool_ragged": dict(h_q=16, h_kv=4, D=128, n_link=5, prefix=0, pool_block_size=16,
                              doc_lens_per_query=[[15, 16, 17, 100], [33]], q_lens=[12, 5]),
}


@pytest.mark.parametrize("name", sorted(EDGE))
@pytest.mark.parametrize("mode", ["fused", "separate"])
def test_edge_cases(RT, name, mode):
    batch = custom_batch(50 + sorted(EDGE).index(name), **EDGE[name])
    lp, gk, gv, gout, inp = run_layer(RT, batch, 0, mode)
    for b in range(batch.cfg.batch):
        check_query(batch, b, lp, gk, gv, gout, inp)


def test_reencode_leaves_fresh_slots_untouched(RT):
    batch = W.draw_batch(W.get_config(1))
    dev = torch.device("cuda:0")
    pk, pv = W.pool_kv(batch, 0)
    lp = RT.LinkedPrefill.from_batch(batch, device=dev)
    ck, cv = lp.empty_cache()
    ck.view(torch.int16).fill_(0x1234)
    cv.view(torch.int16).fill_(0x1234)
    lp.reencode_concat(RT.bf16_from_bits(pk, dev), RT.bf16_from_bits(pv, dev), ck, cv)
    torch.cuda.synchronize()
    lay = O.linked_layout(0, [64, 64], 2, 16)
    fresh = RT.bits_from_bf16(ck)[lay.fresh_pos]
    assert np.all(fresh == 0x1234)
    assert not np.any(RT.bits_from_bf16(ck)[lay.kind == O.DOC] == 0x1234)


# ----------------------------------------------------------------- full-size workloads, sampled

def test_llama8b_batch8_zipf_sampled(RT):
    batch = W.draw_batch(W.get_config(3))
    lp, gk, gv, gout, inp = run_layer(RT, batch, 31)
    for b in range(batch.cfg.batch):
        check_query(batch, b, lp, gk, gv, gout, inp, attention=b in (0, 7))


def test_llama8b_long_context_sampled(RT):
    batch = W.draw_batch(W.get_config(4))
    lp, gk, gv, gout, inp = run_layer(RT, batch, 0)
    T = int(batch.n_fresh[0])
    rows = [0, 1, 4, 5, 9, 31, 32, 127, 128, 255, 256, 400, 499, 500, 501, 563, T - 2, T - 1]
    check_query(batch, 0, lp, gk, gv, gout, inp, rows=rows)


def test_llama8b_paged_serving_sampled(RT):
    batch = W.draw_batch(W.get_config(5))
    lp, gk, gv, gout, inp = run_layer(RT, batch, 0)
    for b in (0, 31, 63):
        check_query(batch, b, lp, gk, gv, gout, inp)
    for b in (1, 17, 40):
        check_query(batch, b, lp, gk, gv, gout, inp, attention=False)


def test_layers_from_host_pipeline_matches_per_layer_calls(RT):
    """The host-to-host pipelined helper gives the same bytes as per-layer device calls."""
    batch = W.draw_batch(W.get_config(2))
    dev = torch.device("cuda:0")
    L = 2
    lp = RT.LinkedPrefill.from_batch(batch, device=dev)
    pk, pv, qh, kh, vh = [], [], [], [], []
    for layer in range(L):
        a, b = W.pool_kv(batch, layer)
        q, k, v = W.fresh_qkv(batch, layer)
        pk.append(RT.bf16_from_bits(a, dev))
        pv.append(RT.bf16_from_bits(b, dev))
        qh.append(RT.bf16_from_bits(q).pin_memory())
        kh.append(RT.bf16_from_bits(k).pin_memory())
        vh.append(RT.bf16_from_bits(v).pin_memory())
    shape_q, shape_k = qh[0].shape, kh[0].shape
    dq = [torch.empty(shape_q, dtype=torch.bfloat16, device=dev) for _ in range(L)]
    dk = [torch.empty(shape_k, dtype=torch.bfloat16, device=dev) for _ in range(L)]
    dv = [torch.empty(shape_k, dtype=torch.bfloat16, device=dev) for _ in range(L)]
    caches = [lp.empty_cache() for _ in range(L)]
    dout = [torch.empty(shape_q, dtype=torch.bfloat16, device=dev) for _ in range(L)]
    hout = [torch.empty(shape_q, dtype=torch.bfloat16).pin_memory() for _ in range(L)]
    lp.linked_prefill_layers_from_host(pk, pv, qh, kh, vh, dq, dk, dv, [c[0] for c in caches],
                                       [c[1] for c in caches], dout, hout)
    for layer in range(L):
        ck, cv = lp.empty_cache()
        ref = torch.empty(shape_q, dtype=torch.bfloat16, device=dev)
        lp.linked_prefill(pk[layer], pv[layer], qh[layer].to(dev), kh[layer].to(dev), vh[layer].to(dev),
                          ck, cv, ref)
        torch.cuda.synchronize()
        assert torch.equal(hout[layer].view(torch.int16), ref.cpu().view(torch.int16))


@pytest.mark.parametrize("cfg_index", [2, 4])
def test_rope_fresh_within_one_ulp(RT, cfg_index):
    """Fresh q/k rotated at their global positions (positions up to 51.8k for workload 4)."""
    from paper_2502_16002_gb300 import kvlink as K
    batch = W.draw_batch(W.get_config(cfg_index))
    dev = torch.device("cuda:0")
    q, kn, _ = W.fresh_qkv(batch, 0)
    lp = RT.LinkedPrefill.from_batch(batch, device=dev)
    dq, dk = RT.bf16_from_bits(q, dev), RT.bf16_from_bits(kn, dev)
    lp.rope_fresh(dq, dk)
    torch.cuda.synchronize()
    pos = K.kvlink_plan_get_fresh_positions(lp.plan).astype(np.int64)
    theta = batch.cfg.theta
    for got, src in ((RT.bits_from_bf16(dq), q), (RT.bits_from_bf16(dk), kn)):
        want = O.f64_to_bf16_bits(O.rope_rotate(O.bf16_bits_to_f64(src), pos[:, None], theta))
        assert ulp_distance(got, want).max() <= 1


def test_ttft_comparison_harness_runs(RT):
    """The standard-vs-linked TTFT harness on a small case, with the caches in host memory."""
    from paper_2502_16002_gb300 import ttft
    dev = torch.device("cuda:0")
    layer = ttft.Layer(dev)
    t_std, t_lnk, n_ctx, T = ttft.measure(64, 3, 5, 16, True, dev, layer)
    assert n_ctx == 3 * 64 + 16 and T == 3 * 5 + 16
    assert t_std > 0 and t_lnk > 0
