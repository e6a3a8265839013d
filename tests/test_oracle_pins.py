"""Pins of the fp64 oracle against what the paper and the mathematics fix.

Each test checks the oracle against something other than itself: a worked
example from the paper (Fig. 2), closed forms, invariants, a textbook
formulation written differently (complex rotation), a library routine (torch's
float32->bf16 rounding), or brute force in plain Python loops on tiny inputs.
"""
import cmath
import math
import os

import numpy as np
import pytest

import oracle as O
import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ---------------------------------------------------------------- bf16 rounding

def _f64_from_bits(b):
    return O.bf16_bits_to_f64(np.asarray([b], dtype=np.uint16))[0]


def test_bf16_roundtrip_all_patterns():
    u = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    x = O.bf16_bits_to_f64(u)
    ok = ~np.isnan(x)
    assert np.array_equal(O.f64_to_bf16_bits(x[ok]), u[ok])


def test_bf16_rounding_matches_torch_on_float32_values():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(7)
    bits = rng.integers(0, 2**32, size=200000, dtype=np.uint64).astype(np.uint32)
    # force many exact ties (low half == 0x8000) and near ties
    bits[:20000] = (bits[:20000] & np.uint32(0xFFFF0000)) | np.uint32(0x8000)
    bits[20000:30000] = (bits[20000:30000] & np.uint32(0xFFFF0000)) | np.uint32(0x7FFF)
    f = bits.view(np.float32)
    f = f[np.isfinite(f)]
    ours = O.f64_to_bf16_bits(f.astype(np.float64))
    ref = torch.from_numpy(f.copy()).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(ours, ref)


def test_bf16_rounding_is_single_rounding_from_double():
    # 1 + 2^-8 + 2^-30 is just above the halfway point between 1 and 1+2^-7:
    # direct rounding gives 1+2^-7; rounding through float32 first would tie to 1.
    x = 1.0 + 2.0**-8 + 2.0**-30
    assert O.f64_to_bf16_bits(np.asarray([x]))[0] == 0x3F81
    assert O.f64_to_bf16_bits(np.asarray([1.0 + 2.0**-8]))[0] == 0x3F80  # exact tie -> even


def test_bf16_rounding_subnormals_overflow_signs():
    r = lambda v: int(O.f64_to_bf16_bits(np.asarray([v]))[0])
    assert r(2.0**-133) == 0x0001
    assert r(2.0**-134) == 0x0000            # tie between 0 and 2^-133 -> even (0)
    assert r(3 * 2.0**-134) == 0x0002        # tie between 1 and 2 quanta -> even (2)
    assert r(2.0**128) == 0x7F80             # overflow -> +inf
    assert r(-(2.0**128)) == 0xFF80
    assert r(_f64_from_bits(0x7F7F)) == 0x7F7F
    assert r(-0.0) == 0x8000
    assert r(-1.5) == 0xBFC0


# ---------------------------------------------------------------- RoPE

def _rope_complex(x, pos, theta):
    """Textbook form: pair (x_j, x_{j+D/2}) as z_j, rotated by exp(i * pos * w_j)."""
    D = len(x)
    h = D // 2
    out = [0.0] * D
    for j in range(h):
        w = math.exp(-(2.0 * j / D) * math.log(theta))
        z = complex(x[j], x[j + h]) * cmath.exp(1j * pos * w)
        out[j], out[j + h] = z.real, z.imag
    return np.asarray(out)


@pytest.mark.parametrize("D,theta", [(8, 10000.0), (64, 10000.0), (128, 500000.0)])
def test_rope_matches_complex_rotation(D, theta):
    rng = np.random.default_rng(D)
    for pos in [0, 1, 7, 513, 51827]:
        x = rng.standard_normal(D)
        np.testing.assert_allclose(O.rope_rotate(x, pos, theta), _rope_complex(x, pos, theta),
                                   rtol=0, atol=1e-9)


def test_rope_inv_freq_endpoints():
    f = O.rope_inv_freq(500000.0, 128)
    assert f[0] == 1.0
    assert abs(f[-1] - 500000.0 ** (-126 / 128)) < 1e-18
    assert np.all(np.diff(f) < 0)


@pytest.mark.parametrize("D,theta", [(64, 10000.0), (128, 500000.0)])
def test_rope_composition_identity(D, theta):
    """R_delta R_p x == R_{p+delta} x (Sec. 2.2: positions are fixed after caching)."""
    rng = np.random.default_rng(1)
    x = rng.standard_normal((200, D))
    p = rng.integers(0, 60000, size=200)
    d = rng.integers(0, 60000, size=200)
    a = O.rope_rotate(O.rope_rotate(x, p, theta), d, theta)
    b = O.rope_rotate(x, p + d, theta)
    assert np.max(np.abs(a - b)) < 1e-9


def test_rope_zero_is_identity_and_preserves_pair_norms():
    rng = np.random.default_rng(2)
    x = rng.standard_normal((50, 128))
    assert np.array_equal(O.rope_rotate(x, 0, 500000.0), x)
    y = O.rope_rotate(x, 12345, 500000.0)
    n0 = x[:, :64] ** 2 + x[:, 64:] ** 2
    n1 = y[:, :64] ** 2 + y[:, 64:] ** 2
    np.testing.assert_allclose(n0, n1, rtol=1e-12)


def test_rope_scores_depend_on_relative_position_only():
    rng = np.random.default_rng(3)
    q, k = rng.standard_normal(64), rng.standard_normal(64)
    s1 = O.rope_rotate(q, 900, 1e4) @ O.rope_rotate(k, 400, 1e4)
    s2 = O.rope_rotate(q, 3500, 1e4) @ O.rope_rotate(k, 3000, 1e4)
    assert abs(s1 - s2) < 1e-10


# ---------------------------------------------------------------- layout and masks

def _golden_mask():
    rows = []
    with open(os.path.join(GOLDEN, "figure2_mask.txt")) as fh:
        for line in fh:
            if line.strip() and not line.startswith("#"):
                rows.append([int(t) for t in line.split()])
    return np.asarray(rows, dtype=bool)


def test_figure2_layout_and_training_mask():
    lay = O.linked_layout(0, [2, 2, 1], 1, 1)
    assert lay.total == 9
    assert list(lay.link_pos[:, 0] + 1) == [3, 6, 8]      # 1-based tokens 3, 6, 8
    assert list(lay.question_pos + 1) == [9]
    assert np.array_equal(O.training_mask(lay), _golden_mask())


def test_figure2_inference_map_equals_training_map():
    lay = O.linked_layout(0, [2, 2, 1], 1, 1)
    fp = lay.fresh_pos
    assert np.array_equal(O.inference_mask(fp, 9), _golden_mask()[fp])


def test_figure2_links_appended_at_end():
    """Sec. 2.3 (inference): the caches of the documents (tokens 1, 2, 4, 5, 7) are loaded
    and concatenated, and the new link tokens 3, 6 and 8 are appended at the end of the
    reordered sequence; the question token 9 follows them."""
    lay = O.linked_layout(0, [2, 2, 1], 1, 1)
    rows = O.links_at_end_rows(lay)
    held = np.empty(9, np.int64)
    held[rows] = np.arange(9)
    assert list(held + 1) == [1, 2, 4, 5, 7, 3, 6, 8, 9]


@pytest.mark.parametrize("seed", range(6))
def test_links_at_end_rows_invariants(seed):
    rng = np.random.default_rng(300 + seed)
    P = int(rng.integers(0, 5))
    lens = rng.integers(1, 9, size=int(rng.integers(1, 6))).tolist()
    K, Q = int(rng.choice([0, 1, 3])), int(rng.integers(1, 5))
    lay = O.linked_layout(P, lens, K, Q)
    rows = O.links_at_end_rows(lay)
    assert sorted(rows.tolist()) == list(range(lay.total))          # a permutation
    n_cached = P + sum(lens)
    cached = (lay.kind == O.PREFIX) | (lay.kind == O.DOC)
    assert np.array_equal(np.sort(rows[cached]), np.arange(n_cached))  # caches first
    assert np.all(np.diff(rows[cached]) > 0) and np.all(np.diff(rows[lay.fresh_pos]) > 0)
    assert np.array_equal(rows[lay.fresh_pos], np.arange(n_cached, lay.total))


@pytest.mark.parametrize("seed", range(4))
def test_links_at_end_cache_gives_the_interleaved_attention(seed):
    """The same keys and values stored links-at-end and masked by position give the output
    of the interleaved cache (itself pinned to the brute-force training map); masking by row
    index instead of position would not."""
    rng = np.random.default_rng(400 + seed)
    lens = rng.integers(2, 7, size=3).tolist()
    lay = O.linked_layout(int(rng.integers(0, 3)), lens, 2, 3)
    C, Hq, Hkv, D = lay.total, 4, 2, 8
    q = rng.standard_normal((C, Hq, D))
    k = rng.standard_normal((C, Hkv, D))
    v = rng.standard_normal((C, Hkv, D))
    fp = lay.fresh_pos
    want = O.suffix_attention(q[fp], k, v, fp)
    rows = O.links_at_end_rows(lay)
    k_phys, v_phys = np.empty_like(k), np.empty_like(v)
    k_phys[rows], v_phys[rows] = k, v
    key_pos = np.empty(C, np.int64)
    key_pos[rows] = np.arange(C)
    got = O.suffix_attention(q[fp], k_phys, v_phys, fp, key_pos=key_pos)
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-12)
    wrong = O.suffix_attention(q[fp], k_phys, v_phys, fp)
    assert not np.allclose(wrong, want)


def test_second_token_of_second_document_position():
    # Sec. 2.2: with no link tokens, the second token of Doc_b sits at |Doc_a| + 2 (1-based)
    for la in [1, 5, 37]:
        lay = O.linked_layout(0, [la, 9], 0, 1)
        assert lay.doc_start[1] + 1 + 1 == la + 2


@pytest.mark.parametrize("seed", range(6))
def test_inference_mask_equals_training_mask_rows(seed):
    """Sec. 2.3 / Fig. 2: the inference map of the fresh rows equals the training map."""
    rng = np.random.default_rng(seed)
    P = int(rng.integers(0, 5))
    lens = rng.integers(1, 6, size=int(rng.integers(1, 5))).tolist()
    K = int(rng.choice([0, 1, 2, 5]))
    Q = int(rng.integers(1, 4))
    lay = O.linked_layout(P, lens, K, Q)
    fp = lay.fresh_pos
    assert len(fp) == len(lens) * K + Q
    assert np.array_equal(O.inference_mask(fp, lay.total), O.training_mask(lay)[fp])


def test_workload_context_lengths():
    expect = {1: (148, 20), 3: (5316, 164), 4: (51828, 628)}
    for i, (C, T) in expect.items():
        b = W.draw_batch(W.get_config(i))
        cfg = b.cfg
        for q in range(cfg.batch):
            P = int(b.pool_len[b.prefix_doc[q]]) if b.prefix_doc[q] >= 0 else 0
            lay = O.linked_layout(P, [int(b.pool_len[d]) for d in b.docs_of(q)], cfg.n_link,
                                  int(b.q_len[q]))
            assert (lay.total, len(lay.fresh_pos)) == (C, T)


# ---------------------------------------------------------------- attention

def _bruteforce_full_attention(qs, ks, vs, allowed, Hq, Hkv):
    """Every row of a full sequence, plain loops: softmax over the allowed keys."""
    C = len(qs)
    D = len(qs[0][0])
    G = Hq // Hkv
    out = [[None] * Hq for _ in range(C)]
    for r in range(C):
        for h in range(Hq):
            g = h // G
            sc = []
            for j in range(C):
                if allowed[r][j]:
                    sc.append((j, sum(qs[r][h][d] * ks[j][g][d] for d in range(D)) / math.sqrt(D)))
            mx = max(s for _, s in sc)
            w = [(j, math.exp(s - mx)) for j, s in sc]
            z = sum(e for _, e in w)
            out[r][h] = [sum(e * vs[j][g][d] for j, e in w) / z for d in range(D)]
    return np.asarray(out)


@pytest.mark.parametrize("seed", range(4))
def test_suffix_attention_matches_bruteforce_training_map(seed):
    """Fresh rows of the oracle's suffix attention == rows of full-sequence attention under
    the dense training-time KVLink map (Sec. 2.3), computed by brute force."""
    rng = np.random.default_rng(100 + seed)
    P = int(rng.integers(0, 3))
    lens = rng.integers(1, 5, size=3).tolist()
    K = int(rng.choice([0, 1, 2]))
    Q = int(rng.integers(1, 3))
    Hq, Hkv, D = 4, 2, 8
    lay = O.linked_layout(P, lens, K, Q)
    C = lay.total
    q = rng.standard_normal((C, Hq, D))
    k = rng.standard_normal((C, Hkv, D))
    v = rng.standard_normal((C, Hkv, D))
    full = _bruteforce_full_attention(q.tolist(), k.tolist(), v.tolist(),
                                      O.training_mask(lay).tolist(), Hq, Hkv)
    fp = lay.fresh_pos
    ours = O.suffix_attention(q[fp], k, v, fp)
    np.testing.assert_allclose(ours, full[fp], rtol=0, atol=1e-12)


def test_single_visible_key_returns_its_value():
    rng = np.random.default_rng(5)
    k = rng.standard_normal((6, 2, 8))
    v = rng.standard_normal((6, 2, 8))
    q = rng.standard_normal((1, 4, 8)) * 50
    out = O.suffix_attention(q, k, v, np.asarray([0]))
    for h in range(4):
        np.testing.assert_allclose(out[0, h], v[0, h // 2], rtol=0, atol=1e-15)


def test_zero_keys_average_exactly_the_visible_values():
    rng = np.random.default_rng(6)
    C = 11
    k = np.zeros((C, 1, 8))
    v = rng.standard_normal((C, 1, 8))
    pos = np.asarray([0, 3, 10])
    out = O.suffix_attention(rng.standard_normal((3, 1, 8)), k, v, pos)
    for r, p in enumerate(pos):
        np.testing.assert_allclose(out[r, 0], v[: p + 1, 0].mean(axis=0), rtol=0, atol=1e-14)


def test_score_scale_is_inverse_sqrt_head_dim():
    D = 16
    q = np.zeros((1, 1, D)); q[0, 0, 0] = 3.0
    k = np.zeros((2, 1, D)); k[0, 0, 0] = 2.0
    v = np.zeros((2, 1, D)); v[0, 0, 1] = 1.0; v[1, 0, 2] = 1.0
    out = O.suffix_attention(q, k, v, np.asarray([1]))
    w0 = 1.0 / (1.0 + math.exp(-6.0 / math.sqrt(D)))
    np.testing.assert_allclose(out[0, 0, 1:3], [w0, 1 - w0], rtol=0, atol=1e-15)


# ---------------------------------------------------------------- re-encode + concat

def _tiny_pool(rng, lens, H, D):
    starts = np.concatenate([[0], np.cumsum(lens)[:-1]]).astype(np.int64)
    n = int(np.sum(lens))
    pk = W.f32_to_bf16_bits(rng.standard_normal((n, H, D)).astype(np.float32))
    pv = W.f32_to_bf16_bits(rng.standard_normal((n, H, D)).astype(np.float32))
    return pk, pv, starts, np.asarray(lens, dtype=np.int32)


def test_reencode_keys_equal_rotation_at_global_position():
    """A key stored rotated at local position t (y = R_t x), re-encoded by delta = s_i,
    equals R_{s_i + t} x: the paper's storage form rotated at the global position."""
    rng = np.random.default_rng(8)
    H, D, theta = 2, 64, 10000.0
    lens = [5, 7, 3, 4]                 # entry 3 is the prefix
    pk, pv, st, ln = _tiny_pool(rng, lens, H, D)
    docs, K, Q = [2, 0, 1], 2, 3
    T = len(docs) * K + Q
    kn = W.f32_to_bf16_bits(rng.standard_normal((T, H, D)).astype(np.float32))
    vn = W.f32_to_bf16_bits(rng.standard_normal((T, H, D)).astype(np.float32))
    c = O.reencode_concat(pk, pv, st, ln, 3, docs, K, kn, vn, Q, theta)
    lay = c.layout
    assert lay.total == 4 + 3 + 5 + 7 + len(docs) * K + Q
    for i, d in enumerate(docs):
        y = O.bf16_bits_to_f64(pk[st[d]: st[d] + ln[d]])            # stored: R_t x
        t = np.arange(ln[d])[:, None].repeat(H, 1)
        x = O.rope_rotate(y, -t, theta)                              # un-rotated W_k x
        g = lay.doc_start[i] + t
        want = O.rope_rotate(x, g, theta)
        s = lay.doc_start[i]
        assert np.max(np.abs(c.k_exact[s: s + ln[d]] - want)) < 1e-9
        assert np.array_equal(c.v_bits[s: s + ln[d]], pv[st[d]: st[d] + ln[d]])
    # prefix copied bit-exactly (delta 0), fresh rows at their positions
    assert np.array_equal(c.k_bits[:4], pk[st[3]: st[3] + 4])
    assert np.array_equal(c.k_bits[lay.fresh_pos], kn)
    assert np.array_equal(c.v_bits[lay.fresh_pos], vn)


def test_one_document_no_links_is_standard_causal_attention():
    """One document, no link tokens and no other documents: the linked prefill of the
    question equals standard causal attention over [prefix, doc, question] with every
    key rotated directly at its global position (Sec. 2.2-2.3)."""
    rng = np.random.default_rng(9)
    H, Hq, D, theta = 2, 4, 16, 10000.0
    P, L, Q = 3, 6, 4
    raw_prefix = rng.standard_normal((P, H, D))
    raw_doc = rng.standard_normal((L, H, D))
    # pool stores keys rotated at local positions; keep exact doubles by rounding the raw
    # draws so that the stored bf16 values are the rotated keys' nearest bf16
    stored_doc = O.f64_to_bf16_bits(O.rope_rotate(raw_doc, np.arange(L)[:, None], theta))
    stored_pre = O.f64_to_bf16_bits(O.rope_rotate(raw_prefix, np.arange(P)[:, None], theta))
    pk = np.concatenate([stored_doc, stored_pre])
    pv = W.f32_to_bf16_bits(rng.standard_normal((L + P, H, D)).astype(np.float32))
    st = np.asarray([0, L], np.int64)
    ln = np.asarray([L, P], np.int32)
    kn = W.f32_to_bf16_bits(rng.standard_normal((Q, H, D)).astype(np.float32))
    vn = W.f32_to_bf16_bits(rng.standard_normal((Q, H, D)).astype(np.float32))
    qn = rng.standard_normal((Q, Hq, D))
    c = O.reencode_concat(pk, pv, st, ln, 1, [0], 0, kn, vn, Q, theta)
    ours = O.suffix_attention(qn, c.k_exact, O.bf16_bits_to_f64(c.v_bits), c.layout.fresh_pos)

    # standard causal attention over the full sequence, keys rotated at global positions
    seq_k = np.concatenate([
        O.rope_rotate(O.rope_rotate(O.bf16_bits_to_f64(stored_pre), -np.arange(P)[:, None], theta),
                      np.arange(P)[:, None], theta),
        O.rope_rotate(O.rope_rotate(O.bf16_bits_to_f64(stored_doc), -np.arange(L)[:, None], theta),
                      P + np.arange(L)[:, None], theta),
        O.bf16_bits_to_f64(kn)])
    seq_v = np.concatenate([O.bf16_bits_to_f64(pv[L:]), O.bf16_bits_to_f64(pv[:L]),
                            O.bf16_bits_to_f64(vn)])
    C = P + L + Q
    causal = [[j <= r for j in range(C)] for r in range(C)]
    seq_q = np.zeros((C, Hq, D)); seq_q[P + L:] = qn
    full = _bruteforce_full_attention(seq_q.tolist(), seq_k.tolist(), seq_v.tolist(), causal, Hq, H)
    np.testing.assert_allclose(ours, full[P + L:], rtol=0, atol=1e-9)


def _page_out(contig, starts, lens, bs, rng):
    """Store a contiguous pool as pages, the way a paged cache manager would: each
    document's rows are padded to whole blocks (the padding filled with values that occur
    nowhere in the documents), cut into [blocks, bs] with a reshape, and the blocks are
    written to physical pages drawn as a random permutation.  Returns (pages, block table,
    first logical block of each document)."""
    H, D = contig.shape[1:]
    nblk = [(int(L) + bs - 1) // bs for L in lens]
    first = np.concatenate([[0], np.cumsum(nblk)[:-1]]).astype(np.int64)
    n_pages = int(sum(nblk)) + 3                   # spare pages nothing maps to
    table = rng.permutation(n_pages)[: int(sum(nblk))].astype(np.int32)
    pages = np.full((n_pages, bs, H, D), 0xFFFF, dtype=np.uint16)     # NaN patterns
    for d, L in enumerate(lens):
        padded = np.full((nblk[d] * bs, H, D), 0xFFFE, dtype=np.uint16)
        padded[:L] = contig[starts[d]: starts[d] + L]
        for i, blk in enumerate(padded.reshape(nblk[d], bs, H, D)):
            pages[table[first[d] + i]] = blk
    return pages, table, first


@pytest.mark.parametrize("bs", [16, 8])
def test_paged_pool_reads_the_same_documents(bs):
    """The paged read of every document equals its contiguous slice, for lengths around
    the block size (1, bs-1, bs, bs+1) and a long one, through a block table drawn
    independently of the reader: the pages are written by a reshape of each padded
    document, not by the row arithmetic the oracle reads them with."""
    rng = np.random.default_rng(10 + bs)
    H, D = 2, 8
    lens = np.asarray([1, bs - 1, bs, bs + 1, 100, 37], np.int32)
    starts = np.concatenate([[0], np.cumsum(lens)[:-1]]).astype(np.int64)
    contig = rng.integers(0, 2**15, size=(int(lens.sum()), H, D)).astype(np.uint16)
    pages, table, first = _page_out(contig, starts, lens, bs, rng)
    for d in range(len(lens)):
        want = O.pool_doc_rows(contig, d, starts, lens)
        assert np.array_equal(want, contig[starts[d]: starts[d] + lens[d]])
        got = O.pool_doc_rows(pages, d, first, lens, table, bs)
        assert got.shape == want.shape
        assert np.array_equal(got, want), f"document {d} (length {lens[d]})"


def test_paged_pool_gives_the_contiguous_linked_cache():
    """The whole re-encode + concat from a paged pool equals the one from the same
    documents stored contiguously, bit for bit (keys and values)."""
    rng = np.random.default_rng(12)
    H, D, bs, K, theta = 2, 16, 16, 2, 10000.0
    lens = np.asarray([17, 1, 16, 40, 15], np.int32)
    starts = np.concatenate([[0], np.cumsum(lens)[:-1]]).astype(np.int64)
    ck = rng.integers(0, 2**15, size=(int(lens.sum()), H, D)).astype(np.uint16) & 0xBFFF   # finite
    cv = rng.integers(0, 2**15, size=(int(lens.sum()), H, D)).astype(np.uint16) & 0xBFFF
    pk, table, first = _page_out(ck, starts, lens, bs, np.random.default_rng(1))
    pv, table_v, _ = _page_out(cv, starts, lens, bs, np.random.default_rng(1))
    assert np.array_equal(table, table_v)
    docs, prefix, Q = [3, 0, 1], 4, 3
    T = len(docs) * K + Q
    kn = rng.integers(0, 2**15, size=(T, H, D)).astype(np.uint16) & 0xBFFF
    vn = rng.integers(0, 2**15, size=(T, H, D)).astype(np.uint16) & 0xBFFF
    a = O.reencode_concat(ck, cv, starts, lens, prefix, docs, K, kn, vn, Q, theta)
    b = O.reencode_concat(pk, pv, first, lens, prefix, docs, K, kn, vn, Q, theta, block_table=table, block_size=bs)
    assert np.array_equal(a.k_bits, b.k_bits) and np.array_equal(a.v_bits, b.v_bits)


def test_no_link_tokens_is_block_reuse_with_causal_question():
    """K = 0 link tokens (the PromptCache / block-attention style reuse the paper compares
    with): the question attends causally over [prefix, documents in retrieval order,
    question], every cached key rotated straight to its global position."""
    rng = np.random.default_rng(11)
    H, Hq, D, theta = 2, 4, 16, 10000.0
    P, lens, Q = 3, [5, 2, 4], 3                      # pool entries 0..2: documents, 3: prefix
    raw = [rng.standard_normal((n, H, D)) for n in lens + [P]]
    stored = [O.f64_to_bf16_bits(O.rope_rotate(x, np.arange(len(x))[:, None], theta)) for x in raw]
    pk = np.concatenate(stored)
    pv = W.f32_to_bf16_bits(rng.standard_normal((sum(lens) + P, H, D)).astype(np.float32))
    st = np.cumsum([0] + lens)[:4].astype(np.int64)
    ln = np.asarray(lens + [P], np.int32)
    order = [2, 0, 1]                                  # retrieval order
    kn = W.f32_to_bf16_bits(rng.standard_normal((Q, H, D)).astype(np.float32))
    vn = W.f32_to_bf16_bits(rng.standard_normal((Q, H, D)).astype(np.float32))
    qn = rng.standard_normal((Q, Hq, D))
    c = O.reencode_concat(pk, pv, st, ln, 3, order, 0, kn, vn, Q, theta)
    ours = O.suffix_attention(qn, c.k_exact, O.bf16_bits_to_f64(c.v_bits), c.layout.fresh_pos)

    # the full sequence written out by hand: each entry un-rotated from its local positions
    # and rotated at its global ones
    ks, vs, pos = [], [], 0
    for e in [3] + order:
        n = int(ln[e])
        local = np.arange(n)[:, None]
        raw_k = O.rope_rotate(O.bf16_bits_to_f64(stored[e]), -local, theta)
        ks.append(O.rope_rotate(raw_k, pos + local, theta))
        vs.append(O.bf16_bits_to_f64(pv[st[e]:st[e] + n]))
        pos += n
    assert pos == P + sum(lens)
    seq_k = np.concatenate(ks + [O.bf16_bits_to_f64(kn)])
    seq_v = np.concatenate(vs + [O.bf16_bits_to_f64(vn)])
    C = pos + Q
    causal = [[j <= r for j in range(C)] for r in range(C)]
    seq_q = np.zeros((C, Hq, D)); seq_q[pos:] = qn
    full = _bruteforce_full_attention(seq_q.tolist(), seq_k.tolist(), seq_v.tolist(), causal, Hq, H)
    np.testing.assert_allclose(ours, full[pos:], rtol=0, atol=1e-9)


def test_byte_model_of_the_8b_shape():
    """The paper's cache size for Llama-3-8B, about 131 MB per 1000 tokens, is K and V x 32
    layers x 8 KV heads x 128 dims x 2 bytes = 131072 B per token.  The 8B-shaped workloads
    and the bench's algorithmic byte count (cache bytes written per cached token and layer)
    must follow the same formula."""
    import bench
    for idx in (3, 4, 5):
        cfg = W.get_config(idx)
        assert 2 * cfg.layers * cfg.h_kv * cfg.head_dim * 2 == 131072, idx
    assert abs(131072 * 1000 / 1e6 - 131) < 0.1

    class Info:                                        # the plan fields the count reads
        cached_tokens, n_fresh, ctx_rows, attn_pairs = 1000, 0, 1000, 0

    batch = W.draw_batch(W.get_config(3))
    cnt = bench.algorithmic_counts(batch, Info())
    written_per_layer = cnt["reencode_bytes"] - 2 * batch.cfg.h_kv * batch.cfg.head_dim * 2 * cnt["unique_pool_tokens"]
    assert written_per_layer * batch.cfg.layers == 131072 * 1000
