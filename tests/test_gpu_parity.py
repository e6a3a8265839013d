"""GPU parity of the linked prefill against the fp64 oracle, through the C ABI.

Tolerances: segment tables bit-exact (tests/test_abi_cpu.py); re-encoded keys
within 1 bf16 ulp of the oracle's correctly rounded fp64 rotation; values,
prefix and fresh rows bit-exact; attention output max |err| <= 1e-2 and mean
|err| <= 1e-3 against the fp64 oracle.
"""
import numpy as np
import pytest

import oracle as O
import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from _gpu_common import EDGE, check_query, custom_batch, run_layer, ulp_distance  # noqa: E402


@pytest.fixture(scope="module")
def RT():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2502_16002_gb300 import runtime

    return runtime


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


def test_rejected_calls_launch_nothing(RT):
    """A call that returns an error has launched nothing: the entry points that place the fresh
    rows (or re-encode the documents) before the attention check the attention's arguments
    first, so a misaligned q is rejected with the cache left as it was."""
    from paper_2502_16002_gb300 import kvlink as K
    batch = W.draw_batch(W.get_config(1))
    dev = torch.device("cuda:0")
    pk, pv = W.pool_kv(batch, 0)
    q, kn, vn = W.fresh_qkv(batch, 0)
    t = {k: RT.bf16_from_bits(v, dev) for k, v in dict(pk=pk, pv=pv, q=q, kn=kn, vn=vn).items()}
    lp = RT.LinkedPrefill.from_batch(batch, device=dev)
    ck, cv = lp.empty_cache()
    out = torch.zeros(lp.fresh_shape(batch.cfg.h_q), dtype=torch.bfloat16, device=dev)
    ws, wsb = lp.workspace.data_ptr(), lp.workspace.numel()
    bad_q = t["q"].data_ptr() + 2                 # not 16-byte aligned
    kn_p, vn_p, pk_p, pv_p = (t[k].data_ptr() for k in ("kn", "vn", "pk", "pv"))
    calls = {
        "kvlink_suffix_attention": lambda: K.kvlink_suffix_attention(
            lp.plan, bad_q, kn_p, vn_p, ck.data_ptr(), cv.data_ptr(), out.data_ptr(), ws, wsb, 0),
        "kvlink_suffix_attention_pool_values": lambda: K.kvlink_suffix_attention_pool_values(
            lp.plan, bad_q, kn_p, vn_p, pv_p, ck.data_ptr(), out.data_ptr(), ws, wsb, 0),
        "kvlink_linked_prefill": lambda: K.kvlink_linked_prefill(
            lp.plan, pk_p, pv_p, bad_q, kn_p, vn_p, ck.data_ptr(), cv.data_ptr(), out.data_ptr(), ws, wsb, 0),
    }
    for name, call in calls.items():
        ck.view(torch.int16).fill_(0x1234)
        cv.view(torch.int16).fill_(0x1234)
        torch.cuda.synchronize()
        with pytest.raises(K.KvlinkError) as e:
            call()
        assert e.value.code == K.KVLINK_EINVAL, name
        torch.cuda.synchronize()
        assert bool(torch.all(ck.view(torch.int16) == 0x1234)), name
        assert bool(torch.all(cv.view(torch.int16) == 0x1234)), name
    assert K.kvlink_device_status() == 0


# ----------------------------------------------------------------- full-size workloads, sampled

@pytest.mark.parametrize("layer", [0, 31])
def test_llama8b_batch8_zipf_sampled(RT, layer):
    batch = W.draw_batch(W.get_config(3))
    lp, gk, gv, gout, inp = run_layer(RT, batch, layer)
    for b in range(batch.cfg.batch):
        check_query(batch, b, lp, gk, gv, gout, inp, attention=b in (0, 7))


def test_llama8b_long_context_sampled(RT):
    batch = W.draw_batch(W.get_config(4))
    lp, gk, gv, gout, inp = run_layer(RT, batch, 0)
    T = int(batch.n_fresh[0])
    rows = ([0, 1, 4, 5, 9, 31, 32, 127, 128, 255, 256, 400, 499, 500, 501, 563] + list(range(540, 561)) +
            list(range(600, T)))
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


def test_ttft_arms_match_the_oracle(RT):
    """One layer of each TTFT arm, run once outside any graph: the standard arm's attention
    (a zero-document plan, the whole context as causal fresh rows) and the linked arm's
    linked cache and attention, each against the fp64 oracle on the tensors the arm gave the
    library (q, k, v after the projection and RoPE, the document pool).  The harness's
    weights give q, k and v unit variance, as in the workloads, so the attention bar is the
    same (an output of magnitude 4 or more would already carry a bf16 rounding error near
    the 1e-2 bar)."""
    from paper_2502_16002_gb300 import kvlink as K, ttft
    dev = torch.device("cuda:0")
    layer = ttft.Layer(dev)
    standard, linked, seen, n_ctx, T = ttft.layer_arms(100, 4, 5, 24, True, dev, layer)
    standard()
    linked()
    torch.cuda.synchronize(dev)
    assert K.kvlink_device_status() == 0
    bits = RT.bits_from_bf16
    s = seen["standard"]
    f64 = lambda t: O.bf16_bits_to_f64(bits(t))
    ref = O.suffix_attention(f64(s["q"]), f64(s["k"]), f64(s["v"]), np.arange(n_ctx))
    err = np.abs(s["out"].float().cpu().numpy() - ref)
    assert err.max() <= 1e-2 and err.mean() <= 1e-3, (err.max(), err.mean())
    ln = seen["linked"]
    cache = O.reencode_concat(bits(ln["pool_k"]), bits(ln["pool_v"]), np.arange(4) * 100, np.full(4, 100), -1,
                              [0, 1, 2, 3], 5, bits(ln["k"]), bits(ln["v"]), 24, ttft.THETA)
    gk, gv = bits(ln["cache_k"]), bits(ln["cache_v"])
    assert np.array_equal(gv, cache.v_bits)
    assert ulp_distance(gk, cache.k_bits).max() <= 1
    ref = O.suffix_attention(f64(ln["q"]), O.bf16_bits_to_f64(cache.k_bits), O.bf16_bits_to_f64(cache.v_bits),
                             cache.layout.fresh_pos)
    err = np.abs(ln["out"].float().cpu().numpy() - ref)
    assert err.max() <= 1e-2 and err.mean() <= 1e-3, (err.max(), err.mean())
