"""fp64 CPU oracle for the KVLink linked prefill.

TEST INFRASTRUCTURE ONLY: imported by the tests, by the smoke check in
__graft_entry__ and by bench.py's CPU-baseline leg, never by the product path.
"""
from .kvlink_oracle import *  # noqa: F401,F403
from .kvlink_oracle import (  # noqa: F401
    Layout, LinkedCache, bf16_bits_to_f64, f64_to_bf16_bits, rope_inv_freq, rope_rotate,
    linked_layout, training_mask, inference_mask, pool_doc_rows, reencode_concat,
    suffix_attention, linked_prefill_query, links_at_end_rows,
)
from .run import oracle_query_layer  # noqa: F401
