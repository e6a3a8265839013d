"""Seeded draws for the linked-prefill workloads.

Every random number comes from numpy's PCG64 through a SeedSequence keyed by
(config index, stream, layer, seed), so any layer of any workload can be drawn
on its own and both sides of a parity test see identical inputs.

Values are N(0,1) float32 rounded to bf16 (round to nearest even) and are held
as uint16 bit patterns.  Cached document keys are drawn directly: a RoPE
rotation maps an isotropic Gaussian pair to an isotropic Gaussian pair, so an
N(0,1) draw has exactly the distribution of a key rotated at its local positions
0..len-1 (the storage form the pool holds), and this module never needs RoPE.
Fresh query/key rows are likewise taken as already rotated at their global
positions.
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import Optional

import numpy as np

from .configs import WorkloadConfig

# stream identifiers inside a SeedSequence
_S_STRUCT, _S_POOL_K, _S_POOL_V, _S_Q, _S_KNEW, _S_VNEW, _S_CACHE_BT, _S_POOL_BT = range(8)


def _rng(cfg_index: int, stream: int, layer: int = 0, seed: int = 0) -> np.random.Generator:
    return np.random.default_rng(np.random.SeedSequence([int(cfg_index), stream, int(layer), int(seed)]))


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """float32 -> bf16 bit patterns, round to nearest even (finite inputs)."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    bias = ((b >> 16) & np.uint32(1)) + np.uint32(0x7FFF)
    return ((b + bias) >> 16).astype(np.uint16)


def bf16_bits_to_f32(u: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(u, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def normal_bf16(rng: np.random.Generator, shape) -> np.ndarray:
    """N(0,1) draws rounded to bf16, as uint16 bit patterns."""
    return f32_to_bf16_bits(rng.standard_normal(size=shape, dtype=np.float32))


@dataclass
class Batch:
    """One batch of retrieval queries against a pool of cached documents.

    Pool entries 0..pool_docs-1 are documents; when the workload has a prefix,
    entry pool_docs is the shared cached system prompt.
    """
    cfg: WorkloadConfig
    seed: int
    pool_len: np.ndarray          # int32 [n_pool]
    pool_start: np.ndarray        # int64 [n_pool]: first row (contiguous) or first block-table slot (paged)
    pool_block_table: Optional[np.ndarray]  # int32 [sum blocks] (paged pool) or None
    pool_rows: int                # token rows of pool storage (paged: n_blocks * block_size)
    prefix_doc: np.ndarray        # int32 [B], -1 = no prefix
    n_docs: np.ndarray            # int32 [B]
    doc_ids: np.ndarray           # int32 [sum n_docs], per query in retrieval order
    q_len: np.ndarray             # int32 [B]

    @property
    def n_pool(self) -> int:
        return int(self.pool_len.shape[0])

    @property
    def n_fresh(self) -> np.ndarray:
        """Fresh rows per query: K link tokens after every document plus the question."""
        return (self.n_docs * self.cfg.n_link + self.q_len).astype(np.int32)

    def docs_of(self, b: int) -> np.ndarray:
        off = int(self.n_docs[:b].sum())
        return self.doc_ids[off: off + int(self.n_docs[b])]


def _zipf_without_replacement(rng: np.random.Generator, n_items: int, k: int, s: float) -> np.ndarray:
    """k distinct items; item r (rank r+1) has weight (r+1)^-s, renormalised after each draw."""
    w = np.arange(1, n_items + 1, dtype=np.float64) ** (-s)
    alive = np.ones(n_items, dtype=bool)
    out = []
    for _ in range(k):
        ww = np.where(alive, w, 0.0)
        cdf = np.cumsum(ww)
        u = rng.random() * cdf[-1]
        i = int(np.searchsorted(cdf, u, side="right"))
        i = min(i, n_items - 1)
        while not alive[i]:  # u landed exactly on a removed item's zero-width step
            i -= 1
        alive[i] = False
        out.append(i)
    return np.asarray(out, dtype=np.int32)


def draw_batch(cfg: WorkloadConfig, seed: int = 0) -> Batch:
    rng = _rng(cfg.index, _S_STRUCT, 0, seed)
    if cfg.doc_len_fixed:
        doc_len = np.full(cfg.pool_docs, cfg.doc_len_fixed, dtype=np.int32)
    else:
        lo, hi = cfg.doc_len_range
        doc_len = rng.integers(lo, hi + 1, size=cfg.pool_docs).astype(np.int32)
    pool_len = doc_len
    if cfg.prefix_len > 0:
        pool_len = np.concatenate([doc_len, np.asarray([cfg.prefix_len], np.int32)])
    n_pool = pool_len.shape[0]

    B = cfg.batch
    prefix_doc = np.full(B, cfg.pool_docs if cfg.prefix_len > 0 else -1, dtype=np.int32)
    n_docs = np.full(B, cfg.docs_per_query, dtype=np.int32)
    ids = []
    for b in range(B):
        if cfg.doc_select == "all":
            ids.append(np.arange(cfg.docs_per_query, dtype=np.int32))
        elif cfg.doc_select == "zipf":
            ids.append(_zipf_without_replacement(rng, cfg.pool_docs, cfg.docs_per_query, cfg.zipf_s))
        elif cfg.doc_select == "uniform":
            ids.append(rng.choice(cfg.pool_docs, size=cfg.docs_per_query, replace=False).astype(np.int32))
        else:
            raise ValueError(cfg.doc_select)
    doc_ids = np.concatenate(ids).astype(np.int32)
    if cfg.q_len_fixed:
        q_len = np.full(B, cfg.q_len_fixed, dtype=np.int32)
    else:
        lo, hi = cfg.q_len_range
        q_len = rng.integers(lo, hi + 1, size=B).astype(np.int32)

    if cfg.pool_block_size:
        bs = cfg.pool_block_size
        nblk = (pool_len.astype(np.int64) + bs - 1) // bs
        total = int(nblk.sum())
        perm = _rng(cfg.index, _S_POOL_BT, 0, seed).permutation(total).astype(np.int32)
        pool_start = np.concatenate([[0], np.cumsum(nblk)[:-1]]).astype(np.int64)
        block_table = perm
        pool_rows = total * bs
    else:
        pool_start = np.concatenate([[0], np.cumsum(pool_len.astype(np.int64))[:-1]]).astype(np.int64)
        block_table = None
        pool_rows = int(pool_len.astype(np.int64).sum())
    return Batch(cfg=cfg, seed=seed, pool_len=pool_len, pool_start=pool_start,
                 pool_block_table=block_table, pool_rows=pool_rows, prefix_doc=prefix_doc,
                 n_docs=n_docs, doc_ids=doc_ids, q_len=q_len)


def pool_kv(batch: Batch, layer: int):
    """Cached K (stored rotated at local positions) and V of one layer, bf16 bits.

    Contiguous pool: [pool_rows, H_kv, D].  Paged pool: [n_blocks, block, H_kv, D].
    """
    cfg = batch.cfg
    if cfg.pool_block_size:
        shape = (batch.pool_rows // cfg.pool_block_size, cfg.pool_block_size, cfg.h_kv, cfg.head_dim)
    else:
        shape = (batch.pool_rows, cfg.h_kv, cfg.head_dim)
    k = normal_bf16(_rng(cfg.index, _S_POOL_K, layer, batch.seed), shape)
    v = normal_bf16(_rng(cfg.index, _S_POOL_V, layer, batch.seed), shape)
    return k, v


def fresh_qkv(batch: Batch, layer: int):
    """Fresh link/question rows of one layer: q [T, H_q, D], k_new/v_new [T, H_kv, D].

    Rows of all queries are concatenated in query order; within a query they are in
    sequence order (links of document 1, ..., links of document N, question).
    """
    cfg = batch.cfg
    T = int(batch.n_fresh.sum())
    q = normal_bf16(_rng(cfg.index, _S_Q, layer, batch.seed), (T, cfg.h_q, cfg.head_dim))
    k = normal_bf16(_rng(cfg.index, _S_KNEW, layer, batch.seed), (T, cfg.h_kv, cfg.head_dim))
    v = normal_bf16(_rng(cfg.index, _S_VNEW, layer, batch.seed), (T, cfg.h_kv, cfg.head_dim))
    return q, k, v


def cache_block_tables(batch: Batch, blocks_per_query) -> np.ndarray:
    """Physical block ids of a paged linked cache: a seeded permutation of all blocks,
    handed out to the queries in order.  Returns int32 [sum blocks_per_query]."""
    total = int(np.sum(blocks_per_query))
    return _rng(batch.cfg.index, _S_CACHE_BT, 0, batch.seed).permutation(total).astype(np.int32)


def normal_bf16_torch(shape, seed: int, device):
    """N(0,1) bf16 tensor drawn on a device with torch's seeded generator.

    For timing runs whose inputs are too large to draw on the host quickly; the
    values differ from the numpy draws, the distribution does not.
    """
    import torch

    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return torch.randn(shape, generator=g, device=device, dtype=torch.float32).to(torch.bfloat16)
