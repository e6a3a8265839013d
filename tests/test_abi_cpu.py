"""Host-side tests of the C ABI (no GPU): symbol exports, the segment table and
offsets against the oracle's layout (bit-exact), attention work coverage, and
argument validation."""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle as O
import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def K():
    from paper_2502_16002_gb300.build import build

    build()
    from paper_2502_16002_gb300 import kvlink

    return kvlink


def _declared_functions():
    src = open(os.path.join(ROOT, "include", "kvlink.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(kvlink_[a-z_0-9]+)\s*\(", src)))


def test_library_exports_every_declared_function(K):
    names = _declared_functions()
    assert len(names) >= 15
    lib = ctypes.CDLL(K._LIB_PATH)
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(K.DECLARED)


def test_debug_build_exports_the_same_functions(K):
    """libkvlink_debug.so (device-side index checks) is the same C ABI."""
    path = os.path.join(os.path.dirname(K._LIB_PATH), "libkvlink_debug.so")
    if not os.path.exists(path):
        pytest.skip("the debug library has not been built")
    lib = ctypes.CDLL(path)
    for n in _declared_functions():
        assert hasattr(lib, n), n


def _plan(K, batch, **over):
    cfg = batch.cfg
    kw = dict(n_link=cfg.n_link, h_q=cfg.h_q, h_kv=cfg.h_kv, head_dim=cfg.head_dim,
              pool_len=batch.pool_len, pool_start=batch.pool_start, pool_rows=batch.pool_rows,
              prefix_doc=batch.prefix_doc, n_docs=batch.n_docs, doc_ids=batch.doc_ids,
              q_len=batch.q_len, pool_block_size=cfg.pool_block_size,
              pool_block_table=batch.pool_block_table, num_sms=152)
    kw.update(over)
    return K.kvlink_plan_create(**kw)


def _oracle_layout(batch, b):
    cfg = batch.cfg
    P = int(batch.pool_len[batch.prefix_doc[b]]) if batch.prefix_doc[b] >= 0 else 0
    return O.linked_layout(P, [int(batch.pool_len[d]) for d in batch.docs_of(b)], cfg.n_link,
                           int(batch.q_len[b]))


@pytest.mark.parametrize("cfg_index", [1, 2, 3, 4, 5])
def test_segment_table_matches_oracle_layout(K, cfg_index):
    batch = W.draw_batch(W.get_config(cfg_index))
    plan = _plan(K, batch)
    seg = K.kvlink_plan_get_segments(plan)
    cu_ctx, cu_fresh = K.kvlink_plan_get_offsets(plan)
    fpos = K.kvlink_plan_get_fresh_positions(plan)
    ctx = fresh = 0
    for b in range(batch.cfg.batch):
        lay = _oracle_layout(batch, b)
        assert cu_ctx[b] == ctx and cu_fresh[b] == fresh
        # expected segments, in sequence order
        exp = []
        if lay.prefix_len:
            exp.append((K.KVLINK_SEG_PREFIX, int(batch.prefix_doc[b]), lay.prefix_len, 0))
        f = fresh
        for i, d in enumerate(batch.docs_of(b)):
            exp.append((K.KVLINK_SEG_DOC, int(d), int(lay.doc_len[i]), int(lay.doc_start[i])))
            if batch.cfg.n_link:
                exp.append((K.KVLINK_SEG_LINK, f, batch.cfg.n_link, int(lay.link_pos[i, 0])))
                f += batch.cfg.n_link
        exp.append((K.KVLINK_SEG_QUESTION, f, int(batch.q_len[b]), int(lay.question_pos[0])))
        mine = seg[seg["query"] == b]
        got = [(int(s["kind"]), int(s["src"]), int(s["len"]), int(s["pos"])) for s in mine]
        assert got == exp
        assert np.array_equal(mine["dst"], ctx + mine["pos"])
        T = len(lay.fresh_pos)
        assert np.array_equal(fpos[fresh: fresh + T], lay.fresh_pos)
        ctx += lay.total
        fresh += T
    assert cu_ctx[-1] == ctx and cu_fresh[-1] == fresh
    info = K.kvlink_plan_get_info(plan)
    assert info.ctx_rows == ctx and info.n_fresh == fresh
    docs = seg[seg["kind"] == K.KVLINK_SEG_DOC]
    assert np.array_equal(np.sort(docs["table"]), np.arange(len(docs)))
    assert info.attn_pairs == int(np.sum(fpos.astype(np.int64) + 1))


@pytest.mark.parametrize("cfg_index", [1, 2, 3, 4, 5])
@pytest.mark.parametrize("layout", [0, 1])
def test_sources_and_rows_match_oracle(K, cfg_index, layout):
    """Per-position sources: the cache row of every position (interleaved: the position;
    links at the end: the oracle's Sec. 2.3 order), and the pool or fresh row it is read
    from, checked by fetching row ids through the oracle's pool addressing."""
    batch = W.draw_batch(W.get_config(cfg_index))
    cfg = batch.cfg
    plan = _plan(K, batch, layout=layout)
    src = K.kvlink_plan_get_sources(plan)
    seg = K.kvlink_plan_get_segments(plan)
    cu_ctx, cu_fresh = K.kvlink_plan_get_offsets(plan)
    assert len(src) == cu_ctx[-1]
    bs = cfg.pool_block_size
    ids = np.arange(batch.pool_rows, dtype=np.int64)
    pool_ids = ids.reshape(-1, bs) if bs else ids
    for b in range(cfg.batch):
        lay = _oracle_layout(batch, b)
        rows = O.links_at_end_rows(lay) if layout else np.arange(lay.total)
        c0 = int(cu_ctx[b])
        mine = src[c0: c0 + lay.total]
        assert np.array_equal(mine["slot"], c0 + rows)
        fresh = (lay.kind == O.LINK) | (lay.kind == O.QUESTION)
        assert np.all(mine["kind"][fresh] == K.KVLINK_SRC_FRESH)
        assert np.array_equal(mine["row"][fresh], cu_fresh[b] + np.arange(int(fresh.sum())))
        assert np.all(mine["kind"][~fresh] == K.KVLINK_SRC_POOL)
        assert np.all(mine["table"][lay.kind != O.DOC] == -1)
        def entry_rows(e):
            return O.pool_doc_rows(pool_ids, int(e), batch.pool_start, batch.pool_len,
                                   batch.pool_block_table, bs)
        if lay.prefix_len:
            assert np.array_equal(mine["row"][: lay.prefix_len], entry_rows(batch.prefix_doc[b]))
        qseg = seg[(seg["query"] == b) & (seg["kind"] == K.KVLINK_SEG_DOC)]
        for i, d in enumerate(batch.docs_of(b)):
            s0, L = int(lay.doc_start[i]), int(lay.doc_len[i])
            assert np.array_equal(mine["row"][s0: s0 + L], entry_rows(d))
            assert np.all(mine["table"][s0: s0 + L] == qseg["table"][i])
        # every segment is one contiguous run of cache rows starting at its dst
        for sg in seg[seg["query"] == b]:
            p0, n = int(sg["pos"]), int(sg["len"])
            assert np.array_equal(rows[p0: p0 + n], int(sg["dst"]) - c0 + np.arange(n))


@pytest.mark.parametrize("cfg_index", [1, 2, 3, 4, 5])
@pytest.mark.parametrize("layout", [0, 1])
def test_value_groups_match_sources(K, cfg_index, layout):
    """The 8-row groups that the zero-copy value path (and the one-kernel path) copies as one
    tile each: an entry holds the first source row exactly when its 8 cache rows read 8
    consecutive rows of one tensor, flagged fresh for k_new / v_new rows; a group with a
    segment boundary inside, or a query's last partial group, is -1.  Checked against the
    per-position sources, which test_sources_and_rows_match_oracle ties to the oracle."""
    batch = W.draw_batch(W.get_config(cfg_index))
    plan = _plan(K, batch, layout=layout)
    src = K.kvlink_plan_get_sources(plan)
    cu_ctx, _ = K.kvlink_plan_get_offsets(plan)
    grp, cu = K.kvlink_plan_get_value_groups(plan)
    # sources in cache-row order (slot is the batch cache row of each position)
    kind = np.empty(len(src), np.int64)
    row = np.empty(len(src), np.int64)
    kind[src["slot"]] = src["kind"]
    row[src["slot"]] = src["row"]
    runs = 0
    for b in range(batch.cfg.batch):
        c0, C = int(cu_ctx[b]), int(cu_ctx[b + 1] - cu_ctx[b])
        n = (C + 7) // 8
        assert cu[b + 1] - cu[b] == n
        for m in range(n):
            e = int(grp[cu[b] + m])
            r = slice(c0 + 8 * m, c0 + 8 * m + 8)
            whole = 8 * m + 8 <= C
            run = whole and np.all(kind[r] == kind[r][0]) and np.array_equal(row[r], row[r][0] + np.arange(8))
            if run:
                flag = K.KVLINK_GROUP_FRESH if kind[r][0] == K.KVLINK_SRC_FRESH else 0
                assert e == (int(row[r][0]) | flag), (b, m)
                runs += 1
            else:
                assert e == -1, (b, m)
    assert cu[-1] == len(grp)
    assert runs > 0.5 * len(grp)       # documents of 64 to 512 rows: most groups are one tile


def _items(K, plan):
    """Attention items and merge groups, read back from the plan's device-buffer image."""
    import paper_2502_16002_gb300.kvlink as KK
    # items are not exported by the ABI; re-derive coverage from the public info instead
    return KK.kvlink_plan_get_info(plan)


@pytest.mark.parametrize("cfg_index", [1, 2, 3, 4, 5])
def test_attention_work_counts(K, cfg_index):
    batch = W.draw_batch(W.get_config(cfg_index))
    plan = _plan(K, batch)
    info = K.kvlink_plan_get_info(plan)
    cfg = batch.cfg
    tok_per_tile = 128 // cfg.group
    m_tiles = sum(-(-int(t) // tok_per_tile) for t in batch.n_fresh)
    assert info.n_attn_items >= m_tiles * cfg.h_kv
    assert info.workspace_bytes == info.n_attn_splits * 128 * (cfg.head_dim + 2) * 4


@pytest.mark.parametrize("num_sms", [152, 37])
@pytest.mark.parametrize("cfg_index,layout", [(1, 0), (2, 0), (2, 1), (3, 0), (3, 1), (4, 0), (5, 0)])
def test_attention_schedule_covers_every_key_tile_once(K, cfg_index, layout, num_sms):
    """Whatever schedule the plan picks (whole M-tiles, repaired, capped shares, gangs): per
    (query, KV head) the M-tiles partition the query's fresh tokens; per M-tile the pieces'
    key-tile entries partition [0, n) with n the tiles the M-tile's last row reaches
    (interleaved layout: ceil((position + 1) / 128)); every piece runs on exactly one CTA, and
    exactly the pieces of cut M-tiles write partials, to distinct slots."""
    batch = W.draw_batch(W.get_config(cfg_index))
    plan = _plan(K, batch, num_sms=num_sms, layout=layout)
    info = K.kvlink_plan_get_info(plan)
    items = K.kvlink_plan_get_attention_items(plan)
    assert len(items) == info.n_attn_items
    assert items["cta"].min() >= 0 and items["cta"].max() < info.n_attn_ctas
    assert np.all(np.diff(items["cta"]) >= 0)          # in run order, CTA by CTA
    cu_ctx, cu_fresh = K.kvlink_plan_get_offsets(plan)
    fresh_pos = K.kvlink_plan_get_fresh_positions(plan)
    mtiles = {}
    for it in items:
        key = (int(it["query"]), int(it["kv_head"]), int(it["tok0"]), int(it["tok1"]))
        mtiles.setdefault(key, []).append(it)
    slots = []
    per_group = {}
    for (b, g, t0, t1), pieces in mtiles.items():
        per_group.setdefault((b, g), []).append((t0, t1))
        ranges = sorted((int(p["entry0"]), int(p["entry1"])) for p in pieces)
        assert ranges[0][0] == 0 and all(r[0] < r[1] for r in ranges)
        assert all(ranges[i][1] == ranges[i + 1][0] for i in range(len(ranges) - 1))
        assert len({(int(p["a_tiles"]), int(p["b_tile0"])) for p in pieces}) == 1
        if layout == 0:
            last_pos = int(fresh_pos[int(cu_fresh[b]) + t1 - 1])
            assert ranges[-1][1] == -(-(last_pos + 1) // 128)
        if len(pieces) > 1:
            slots += [int(p["slot"]) for p in pieces]
        else:
            assert int(pieces[0]["slot"]) == -1
    assert len(slots) == len(set(slots)) == info.n_attn_splits
    assert min(slots, default=0) >= 0
    for b in range(batch.cfg.batch):
        T = int(cu_fresh[b + 1] - cu_fresh[b])
        for g in range(batch.cfg.h_kv):
            spans = sorted(per_group[(b, g)])
            assert spans[0][0] == 0 and spans[-1][1] == T
            assert all(spans[i][1] == spans[i + 1][0] for i in range(len(spans) - 1))


def test_invalid_arguments_are_rejected_before_launch(K):
    batch = W.draw_batch(W.get_config(1))
    with pytest.raises(K.KvlinkError) as e:
        _plan(K, batch, doc_ids=np.asarray([0, 5], np.int32))
    assert e.value.code == K.KVLINK_EBOUNDS
    with pytest.raises(K.KvlinkError) as e:
        _plan(K, batch, head_dim=96)
    assert e.value.code == K.KVLINK_EUNSUPPORTED
    with pytest.raises(K.KvlinkError) as e:
        _plan(K, batch, h_q=6)
    assert e.value.code == K.KVLINK_EUNSUPPORTED
    with pytest.raises(K.KvlinkError) as e:
        _plan(K, batch, pool_rows=100)            # docs need 128 rows
    assert e.value.code == K.KVLINK_EBOUNDS
    with pytest.raises(K.KvlinkError) as e:
        _plan(K, batch, prefix_doc=np.asarray([7], np.int32))
    assert e.value.code == K.KVLINK_EBOUNDS
    with pytest.raises(K.KvlinkError) as e:
        _plan(K, batch, q_len=np.asarray([0], np.int32), n_link=0)   # no fresh rows
    assert e.value.code == K.KVLINK_EINVAL
    with pytest.raises(K.KvlinkError) as e:
        _plan(K, batch, layout=2)
    assert e.value.code == K.KVLINK_EINVAL
    plan = _plan(K, batch)
    info = K.kvlink_plan_get_info(plan)
    with pytest.raises(K.KvlinkError) as e:       # too small: rejected before any CUDA call
        K.kvlink_plan_upload(plan, 1e4, 1 << 20, info.device_bytes - 1, 0)
    assert e.value.code == K.KVLINK_ECAPACITY
    with pytest.raises(K.KvlinkError) as e:       # not uploaded yet
        K.kvlink_reencode_concat(plan, 256, 256, 256, 256, 0)
    assert e.value.code == K.KVLINK_EINVAL
    with pytest.raises(K.KvlinkError) as e:       # not uploaded yet
        K.kvlink_linked_prefill_fused(plan, 256, 256, 256, 256, 256, None, None, 256, 256, 1 << 20, 0)
    assert e.value.code == K.KVLINK_EINVAL


def test_paged_pool_block_ids_are_validated(K):
    batch = W.draw_batch(W.get_config(5))
    bt = batch.pool_block_table.copy()
    bt[3] = batch.pool_rows // 16            # one past the last physical block
    with pytest.raises(K.KvlinkError) as e:
        _plan(K, batch, pool_block_table=bt)
    assert e.value.code == K.KVLINK_EBOUNDS


def test_plan_is_deterministic(K):
    batch = W.draw_batch(W.get_config(3))
    a = K.kvlink_plan_get_segments(_plan(K, batch))
    b = K.kvlink_plan_get_segments(_plan(K, batch))
    assert a.tobytes() == b.tobytes()


def test_attention_exp2_polynomial_accuracy():
    """The FMA-pipe 2^x used for part of the softmax: evaluate the kernel's own constants,
    clamp and range reduction in float32 and check them against 2^x in float64, including
    inputs far below the clamp (masked scores are -inf)."""
    src = open(os.path.join(ROOT, "paper_2502_16002_gb300", "csrc", "kvlink_attention_common.cuh")).read()
    c = {k: np.float32(v) for k, v in re.findall(r"\b(kC[0-3]) = ([0-9.]+)f", src)}
    assert set(c) == {"kC0", "kC1", "kC2", "kC3"}
    floor = np.float32(re.search(r"kExpFloor = (-?[0-9.]+)f", src).group(1))
    x = np.concatenate([np.linspace(-140, 8, 3_000_001), np.arange(-140, 9) + 0.5,
                        [-1e30, -np.inf]]).astype(np.float32)
    xc = np.maximum(x, floor)
    rnd = np.float32(12582912.0)
    t = (xc + rnd).astype(np.float32)
    n = (t - rnd).astype(np.float32)
    f = (xc - n).astype(np.float32)
    assert np.all(np.abs(f) <= 0.5)
    p = ((c["kC3"] * f + c["kC2"]) * f + c["kC1"]) * f + c["kC0"]
    bits = p.astype(np.float32).view(np.int32) + (t.view(np.uint32) << np.uint32(23)).view(np.int32)
    got = bits.view(np.float32).astype(np.float64)
    assert np.all(np.isfinite(got)) and np.all(got >= 0)
    normal = x >= floor + 1          # results in the normal float range
    want = np.exp2(x[normal].astype(np.float64))
    assert np.max(np.abs(got[normal] / want - 1)) < 1e-4
    assert np.all(got[~normal] < 2.0 ** -124)   # at or near the clamp: negligible, never negative


def _plan_kwargs(batch, **over):
    cfg = batch.cfg
    kw = dict(n_link=cfg.n_link, h_q=cfg.h_q, h_kv=cfg.h_kv, head_dim=cfg.head_dim,
              pool_len=batch.pool_len, pool_start=batch.pool_start, pool_rows=batch.pool_rows,
              prefix_doc=batch.prefix_doc, n_docs=batch.n_docs, doc_ids=batch.doc_ids,
              q_len=batch.q_len, pool_block_size=cfg.pool_block_size,
              pool_block_table=batch.pool_block_table, num_sms=152)
    kw.update(over)
    return kw


def _tables(K, plan):
    info = K.kvlink_plan_get_info(plan)
    fields = {f: getattr(info, f) for f, _ in type(info)._fields_}
    return (fields, K.kvlink_plan_get_segments(plan).tobytes(), [a.tobytes() for a in K.kvlink_plan_get_offsets(plan)],
            K.kvlink_plan_get_fresh_positions(plan).tobytes(), K.kvlink_plan_get_sources(plan).tobytes())


def test_rebuilt_plan_equals_a_created_one(K):
    """kvlink_plan_rebuild reuses a plan's storage for another batch (other shapes, a paged
    pool, the other layout) and must give exactly the tables kvlink_plan_create gives."""
    plan = _plan(K, W.draw_batch(W.get_config(3)))
    for cfg_index, layout in ((2, 0), (5, 0), (3, 1), (1, 0), (3, 0)):
        batch = W.draw_batch(W.get_config(cfg_index))
        K.kvlink_plan_rebuild(plan, **_plan_kwargs(batch, layout=layout))
        assert _tables(K, plan) == _tables(K, _plan(K, batch, layout=layout)), (cfg_index, layout)


def test_failed_rebuild_leaves_no_batch(K):
    batch = W.draw_batch(W.get_config(1))
    plan = _plan(K, batch)
    bad = np.array(batch.doc_ids, copy=True)
    bad[0] = len(batch.pool_len) + 5                  # a document id outside the pool
    with pytest.raises(K.KvlinkError):
        K.kvlink_plan_rebuild(plan, **_plan_kwargs(batch, doc_ids=bad))
    with pytest.raises(K.KvlinkError) as e:           # nothing to upload
        K.kvlink_plan_upload(plan, 1e4, 1 << 20, 1 << 20, 0)
    assert e.value.code == K.KVLINK_EINVAL
    K.kvlink_plan_rebuild(plan, **_plan_kwargs(batch))  # usable again
    assert _tables(K, plan) == _tables(K, _plan(K, batch))


def test_null_tables_in_the_description_are_rejected(K):
    """A NULL host table in kvlink_batch_desc_t (or a NULL description / output) is EINVAL."""
    import ctypes as C
    batch = W.draw_batch(W.get_config(1))
    d, keep = K._batch_desc(batch.cfg.n_link, batch.cfg.h_q, batch.cfg.h_kv, batch.cfg.head_dim, batch.pool_len,
                            batch.pool_start, batch.pool_rows, batch.prefix_doc, batch.n_docs, batch.doc_ids,
                            batch.q_len, 0, None, 152, 0)
    h = C.c_void_p()
    assert K.lib.kvlink_plan_create(C.byref(d), C.byref(h)) == 0
    K.lib.kvlink_plan_destroy(h)
    for field in ("pool_len", "pool_start", "prefix_doc", "n_docs", "q_len", "doc_ids"):
        saved = getattr(d, field)
        setattr(d, field, None)
        h = C.c_void_p()
        assert K.lib.kvlink_plan_create(C.byref(d), C.byref(h)) == K.KVLINK_EINVAL, field
        assert not h.value
        setattr(d, field, saved)
    assert K.lib.kvlink_plan_create(None, C.byref(h)) == K.KVLINK_EINVAL
    assert K.lib.kvlink_plan_create(C.byref(d), None) == K.KVLINK_EINVAL
    assert K.lib.kvlink_plan_rebuild(None, C.byref(d)) == K.KVLINK_EINVAL
