"""GPU parity of the one-kernel linked prefill (kvlink_linked_prefill_fused) and of the
links-at-end cache layout (Sec. 2.3, inference), through the C ABI.

The one-kernel path reads pool and fresh rows directly, rotates document keys on their
way to the tensor cores and writes the linked cache as a side output.  It is checked
against the fp64 oracle (same tolerances as the two-kernel path) and, bit for bit,
against the two-kernel path, which it must reproduce exactly: the same rotation code,
the same tiles and the same order of MMAs.  The links-at-end layout stores the same
positions in another row order; the attention masks by position, so its output must
equal the interleaved layout's up to the rounding of a different summation order.
"""
import numpy as np
import pytest

import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from _gpu_common import EDGE, LAYOUTS, check_query, custom_batch, run_layer  # noqa: E402


@pytest.fixture(scope="module")
def RT():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2502_16002_gb300 import runtime

    return runtime


def _same_bits(a, b):
    return np.array_equal(np.asarray(a).view(np.uint64) if a.dtype == np.float64 else a,
                          np.asarray(b).view(np.uint64) if b.dtype == np.float64 else b)


@pytest.mark.parametrize("layout", sorted(LAYOUTS))
def test_one_kernel_tiny_matches_oracle(RT, layout):
    batch = W.draw_batch(W.get_config(1))
    lp, gk, gv, gout, inp = run_layer(RT, batch, 0, "onekernel", layout=LAYOUTS[layout])
    check_query(batch, 0, lp, gk, gv, gout, inp, layout=LAYOUTS[layout])


@pytest.mark.parametrize("cfg_index,layer", [(2, 3), (3, 31), (5, 0)])
@pytest.mark.parametrize("layout", sorted(LAYOUTS))
def test_one_kernel_equals_two_kernel_path_bitwise(RT, cfg_index, layer, layout):
    batch = W.draw_batch(W.get_config(cfg_index))
    lo = LAYOUTS[layout]
    lp, gk, gv, gout, inp = run_layer(RT, batch, layer, "onekernel", layout=lo)
    _, rk, rv, rout, _ = run_layer(RT, batch, layer, "fused", layout=lo)
    assert np.array_equal(gk, rk) and np.array_equal(gv, rv), "linked cache differs from the two-kernel path"
    assert _same_bits(gout, rout), "output differs from the two-kernel path"
    if lo:
        # the same attention in the interleaved layout: the keys come in another order (the
        # cached rows, then the fresh rows), so the sums round differently, within the
        # attention tolerance of each other
        _, _, _, iout, _ = run_layer(RT, batch, layer, "fused", layout=0)
        d = np.abs(gout - iout)
        assert d.max() <= 1e-2 and d.mean() <= 1e-4, (d.max(), d.mean())
    for b in sorted({0, batch.cfg.batch - 1}):
        check_query(batch, b, lp, gk, gv, gout, inp, layout=lo)


@pytest.mark.parametrize("layout", sorted(LAYOUTS))
def test_split_ranges_merge_to_the_same_bits(RT, layout):
    """A plan whose KV ranges are cut between CTAs: the one-kernel path merges the partials in
    a separate merge kernel, the persistent suffix attention inside the kernel, with the same
    arithmetic, so the outputs must be the same bits."""
    name = "long_single_doc_split_kv"
    batch = custom_batch(50 + sorted(EDGE).index(name), **EDGE[name])
    lo = LAYOUTS[layout]
    lp, gk, gv, gout, inp = run_layer(RT, batch, 0, "onekernel", layout=lo)
    assert lp.info.n_attn_splits > 0
    _, rk, rv, rout, _ = run_layer(RT, batch, 0, "fused", layout=lo)
    assert np.array_equal(gk, rk) and np.array_equal(gv, rv)
    assert _same_bits(gout, rout), "in-kernel merge differs from the merge kernel"
    check_query(batch, 0, lp, gk, gv, gout, inp, layout=lo)


@pytest.mark.parametrize("name", sorted(EDGE))
@pytest.mark.parametrize("layout", sorted(LAYOUTS))
def test_one_kernel_edge_cases(RT, name, layout):
    batch = custom_batch(50 + sorted(EDGE).index(name), **EDGE[name])
    lp, gk, gv, gout, inp = run_layer(RT, batch, 0, "onekernel", layout=LAYOUTS[layout])
    for b in range(batch.cfg.batch):
        check_query(batch, b, lp, gk, gv, gout, inp, layout=LAYOUTS[layout])


@pytest.mark.parametrize("name", ["multi_query_ragged", "paged_pool_ragged", "no_link_tokens"])
def test_links_at_end_two_kernel_path(RT, name):
    """Re-encode into links-at-end rows, then the suffix attention over that cache (rows
    gathered in position order), and the CUDA-core cross-check over the same cache."""
    batch = custom_batch(50 + sorted(EDGE).index(name), **EDGE[name])
    lp, gk, gv, gout, inp = run_layer(RT, batch, 0, "separate", layout=1)
    for b in range(batch.cfg.batch):
        check_query(batch, b, lp, gk, gv, gout, inp, layout=1)
    dev = torch.device("cuda:0")
    q = RT.bf16_from_bits(inp[2], dev)
    ck, cv = RT.bf16_from_bits(gk, dev), RT.bf16_from_bits(gv, dev)
    out = torch.empty(lp.fresh_shape(batch.cfg.h_q), dtype=torch.bfloat16, device=dev)
    lp.suffix_attention_simt(q, None, None, ck, cv, out)
    torch.cuda.synchronize()
    assert np.abs(out.float().cpu().numpy() - gout).max() <= 1e-2


def test_zero_copy_values(RT):
    """cache_v NULL: values stay in the pool and k_new/v_new; output and keys unchanged."""
    batch = W.draw_batch(W.get_config(3))
    lp, gk, _, gout, inp = run_layer(RT, batch, 7, "onekernel", write_v=False)
    _, rk, _, rout, _ = run_layer(RT, batch, 7, "onekernel")
    assert np.array_equal(gk, rk) and _same_bits(gout, rout)
    check_query(batch, 2, lp, gk, None, gout, inp)
    # the sources say where every value row lives: gather them and compare with the oracle's cache
    from paper_2502_16002_gb300 import kvlink as K
    src = lp.sources()
    pv, vn = inp[1], inp[4]
    rows_v = np.where((src["kind"] == K.KVLINK_SRC_FRESH)[:, None, None], vn[np.minimum(src["row"], len(vn) - 1)],
                      pv.reshape(-1, *pv.shape[-2:])[src["row"]])
    _, _, rv, _, _ = run_layer(RT, batch, 7, "fused")
    assert np.array_equal(rows_v, rv[src["slot"]])


def test_one_kernel_long_context_sampled(RT):
    """100 documents x 512 tokens (51.8k context, split KV ranges and merges)."""
    batch = W.draw_batch(W.get_config(4))
    lp, gk, gv, gout, inp = run_layer(RT, batch, 0, "onekernel")
    T = int(batch.n_fresh[0])
    rows = [0, 1, 4, 5, 9, 31, 32, 127, 128, 255, 256, 400, 499, 500, 501, 563, T - 2, T - 1]
    check_query(batch, 0, lp, gk, gv, gout, inp, rows=rows)
