"""Helpers shared by the GPU parity tests: run one layer through the C ABI, and check
one query's linked cache and attention rows against the fp64 oracle.

Tolerances: re-encoded keys within 1 bf16 ulp of the oracle's correctly rounded fp64
rotation; values, prefix and fresh rows bit-exact; attention output max |err| <= 1e-2
and mean |err| <= 1e-3 against the fp64 oracle.
"""
import numpy as np
import torch

import oracle as O
import workloads as W

MAX_ABS, MEAN_ABS = 1e-2, 1e-3
LAYOUTS = {"interleaved": 0, "links_at_end": 1}


def ulp_distance(a: np.ndarray, b: np.ndarray) -> np.ndarray:
    """Distance between bf16 bit patterns in representable steps (+0 and -0 equal)."""
    def ordinal(u):
        u = u.astype(np.int32)
        return np.where(u & 0x8000, -(u & 0x7FFF), u)
    return np.abs(ordinal(a) - ordinal(b))


def run_layer(RT, batch, layer, mode="fused", rows=None, layout=0, write_v=True):
    """Run one layer on the GPU.  Returns (lp, cache_k bits, cache_v bits, out float64, inputs).

    mode: "fused" = kvlink_linked_prefill (re-encode and attention kernels chained),
    "separate" = kvlink_reencode_concat then kvlink_suffix_attention,
    "onekernel" = kvlink_linked_prefill_fused (cache_v not written when write_v is False;
    its bits are then returned as None), "zero_copy" = kvlink_linked_prefill with cache_v
    NULL (zero-copy values: keys re-encoded, values read from the pool and v_new; cache_v
    bits returned as None)."""
    dev = torch.device("cuda:0")
    pk, pv = W.pool_kv(batch, layer)
    q, kn, vn = W.fresh_qkv(batch, layer)
    lp = RT.LinkedPrefill.from_batch(batch, device=dev, layout=layout)
    ck, cv = lp.empty_cache()
    ck.view(torch.int16).fill_(-1)   # NaN sentinel: every slot must be written
    cv.view(torch.int16).fill_(-1)
    out = torch.full(lp.fresh_shape(batch.cfg.h_q), float("nan"), dtype=torch.bfloat16, device=dev)
    t = {k: RT.bf16_from_bits(v, dev) for k, v in dict(pk=pk, pv=pv, q=q, kn=kn, vn=vn).items()}
    if mode == "zero_copy":
        write_v = False
    if mode == "fused":
        lp.linked_prefill(t["pk"], t["pv"], t["q"], t["kn"], t["vn"], ck, cv, out)
    elif mode == "zero_copy":
        lp.linked_prefill(t["pk"], t["pv"], t["q"], t["kn"], t["vn"], ck, None, out)
    elif mode == "onekernel":
        lp.linked_prefill_fused(t["pk"], t["pv"], t["q"], t["kn"], t["vn"], ck, cv if write_v else None, out)
    else:
        lp.reencode_concat(t["pk"], t["pv"], ck, cv)
        lp.suffix_attention(t["q"], t["kn"], t["vn"], ck, cv, out)
    torch.cuda.synchronize(dev)
    from paper_2502_16002_gb300 import kvlink as K
    assert K.kvlink_device_status() == 0
    return (lp, RT.bits_from_bf16(ck), RT.bits_from_bf16(cv) if write_v else None,
            out.float().cpu().numpy().astype(np.float64), (pk, pv, q, kn, vn))


def check_query(batch, b, lp, gk, gv, gout, inputs, rows=None, attention=True, layout=0):
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
    # cache row of every position: the position itself, or the oracle's links-at-end order
    row = c0 + (O.links_at_end_rows(cache.layout) if layout else np.arange(c1 - c0))
    k_gpu = gk[row]
    if gv is not None:
        assert np.array_equal(gv[row], cache.v_bits), "V concat not bit-exact"
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


# ----------------------------------------------------------------- edge cases

def custom_batch(index, *, h_q, h_kv, D, n_link, prefix, doc_lens_per_query, q_lens, theta=500000.0,
                 pool_block_size=0, seed=0):
    """A batch whose pool holds exactly the listed documents (plus one prefix entry)."""
    lens = [L for q in doc_lens_per_query for L in q]
    cfg = W.WorkloadConfig(index=index, name=f"edge{index}", batch=len(q_lens), layers=1, h_q=h_q,
                           h_kv=h_kv, head_dim=D, theta=theta, prefix_len=prefix, n_link=n_link,
                           docs_per_query=0, pool_docs=len(lens), pool_block_size=pool_block_size)
    # a pool needs one entry: with no documents and no prefix it holds one that no query uses
    pool_len = np.asarray(lens + ([prefix] if prefix else []) or [1], np.int32)
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
    # the standard full prefill that the TTFT comparison times: no documents, no prefix, the
    # whole context as one causal run of fresh rows
    "no_documents_causal_context": dict(h_q=32, h_kv=8, D=128, n_link=5, prefix=0,
                                        doc_lens_per_query=[[]], q_lens=[1523]),
    "prefix_only_no_documents": dict(h_q=32, h_kv=8, D=128, n_link=5, prefix=300,
                                     doc_lens_per_query=[[], [7]], q_lens=[200, 3]),
}


