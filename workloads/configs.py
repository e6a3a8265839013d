"""The five linked-prefill workloads, described by what they are.

Shapes follow the paper's backbones (Sec. 3.1, "Implementation"): Llama-3.2-1B
(32 query heads, 8 KV heads, head dim 64, 16 layers) and Llama-3.1-8B (32/8/128,
32 layers), and its efficiency setup of ten retrieved documents of a few hundred
tokens each (Sec. 3.3).  Link tokens per document follow KVLink5 (Sec. 2.3).
"""
from __future__ import annotations

from dataclasses import dataclass, field


@dataclass(frozen=True)
class WorkloadConfig:
    index: int                 # 1..5
    name: str
    batch: int                 # queries
    layers: int
    h_q: int
    h_kv: int
    head_dim: int
    theta: float               # RoPE base
    prefix_len: int            # cached system-prompt tokens at positions 0..P-1 (0 = none)
    n_link: int                # link tokens appended after every document
    docs_per_query: int
    # pool of precomputed document caches
    pool_docs: int
    doc_len_fixed: int = 0     # every pool document has this length, or 0 ...
    doc_len_range: tuple = (0, 0)  # ... lengths uniform in this inclusive range
    doc_select: str = "all"    # "all" (docs 0..N-1 in order), "zipf", "uniform"
    zipf_s: float = 1.1
    q_len_fixed: int = 0
    q_len_range: tuple = (0, 0)
    pool_block_size: int = 0   # 0 = contiguous pool, else paged with this many tokens per block
    cache_block_size: int = 0  # 0 = contiguous linked cache, else paged
    notes: str = field(default="", compare=False)

    @property
    def group(self) -> int:
        return self.h_q // self.h_kv


CONFIGS = {
    1: WorkloadConfig(
        index=1, name="tiny_2doc", batch=1, layers=1, h_q=4, h_kv=2, head_dim=64,
        theta=10000.0, prefix_len=0, n_link=2, docs_per_query=2, pool_docs=2,
        doc_len_fixed=64, doc_select="all", q_len_fixed=16,
        notes="single layer, two 64-token documents, 2 links each, 16 question tokens"),
    2: WorkloadConfig(
        index=2, name="llama1b_b1_10doc", batch=1, layers=16, h_q=32, h_kv=8, head_dim=64,
        theta=500000.0, prefix_len=16, n_link=5, docs_per_query=10, pool_docs=10,
        doc_len_range=(100, 300), doc_select="all", q_len_fixed=32,
        notes="Llama-3.2-1B shape, 10 documents of 100..300 tokens"),
    3: WorkloadConfig(
        index=3, name="llama8b_b8_zipf20of200", batch=8, layers=32, h_q=32, h_kv=8,
        head_dim=128, theta=500000.0, prefix_len=32, n_link=5, docs_per_query=20,
        pool_docs=200, doc_len_fixed=256, doc_select="zipf", zipf_s=1.1, q_len_fixed=64,
        notes="Llama-3.1-8B shape, batch 8, 20 of 200 pooled 256-token documents by Zipf(1.1), ~5.3k context"),
    4: WorkloadConfig(
        index=4, name="llama8b_b1_long100doc", batch=1, layers=32, h_q=32, h_kv=8,
        head_dim=128, theta=500000.0, prefix_len=0, n_link=5, docs_per_query=100,
        pool_docs=100, doc_len_fixed=512, doc_select="all", q_len_fixed=128,
        notes="Llama-3.1-8B shape, batch 1, 100 documents of 512 tokens, ~51.8k context"),
    5: WorkloadConfig(
        index=5, name="llama8b_b64_paged_serving", batch=64, layers=32, h_q=32, h_kv=8,
        head_dim=128, theta=500000.0, prefix_len=0, n_link=5, docs_per_query=10,
        pool_docs=1000, doc_len_range=(64, 512), doc_select="uniform",
        q_len_range=(16, 128), pool_block_size=16, cache_block_size=16,
        notes="Llama-3.1-8B shape, batch 64, 1000-document pool paged in 16-token blocks"),
}


def get_config(index: int) -> WorkloadConfig:
    return CONFIGS[int(index)]
