"""Drives the oracle over one query and layer of a seeded workload draw.

TEST INFRASTRUCTURE ONLY (tests, smoke check, CPU-baseline timing).
"""
from __future__ import annotations

import numpy as np

from .kvlink_oracle import LinkedCache, linked_prefill_query, reencode_concat


def oracle_query_layer(batch, b: int, pool_k: np.ndarray, pool_v: np.ndarray,
                       q: np.ndarray, k_new: np.ndarray, v_new: np.ndarray,
                       with_attention: bool = True):
    """Linked cache and attention output of query b for one layer.

    batch is a workloads.Batch; pool_k/pool_v are that layer's pool tensors and
    q/k_new/v_new the layer's fresh rows of all queries (bf16 bits).
    Returns (LinkedCache, out float64 [T_b, H_q, D] or None).
    """
    cfg = batch.cfg
    nf = batch.n_fresh
    r0 = int(nf[:b].sum())
    r1 = r0 + int(nf[b])
    cache: LinkedCache = reencode_concat(
        pool_k, pool_v, batch.pool_start, batch.pool_len, int(batch.prefix_doc[b]),
        [int(d) for d in batch.docs_of(b)], cfg.n_link, k_new[r0:r1], v_new[r0:r1],
        int(batch.q_len[b]), cfg.theta, block_table=batch.pool_block_table,
        block_size=cfg.pool_block_size)
    out = linked_prefill_query(q[r0:r1], cache) if with_attention else None
    return cache, out
