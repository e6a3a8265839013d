"""fp64 CPU oracle for KVLink's linked prefill (arXiv 2502.16002).

TEST INFRASTRUCTURE ONLY.  Only the tests, the smoke check in __graft_entry__
and bench.py's CPU-baseline leg may import this module.  The product path (the
CUDA library and its Python binding) never calls it, and it shares no code with
that path: it has its own position bookkeeping, RoPE, bf16 rounding, masks and
attention, each written as the plain definition from the paper in float64.

What it computes, per layer and per query (Sec. 2.1-2.3):
  * the interleaved global layout [prefix, doc_1, links_1, ..., doc_N, links_N,
    question], with K link tokens after every document (Sec. 2.3);
  * positional re-encoding of cached keys (Sec. 2.2): a key stored rotated at
    its local position t is rotated once more by the document's global start
    s_i, which by composition of RoPE rotations equals the rotation at the
    global position s_i + t (the paper's own storage form, un-rotated keys
    rotated at the global position, is the same map and is checked by the pins);
  * concatenation of the re-encoded caches and the fresh link/question rows into
    the query's linked cache (Sec. 2.1, Sec. 2.3 "Inference");
  * the KVLink attention mask, built two independent ways: by global position
    for the fresh rows, and as the dense training-time map (Sec. 2.3, Fig. 2,
    whose caption states the two maps are identical);
  * softmax attention of the fresh link and question rows over the linked cache.

Readings where the paper is silent (each also listed in the design notes):
  * RoPE pairs dimension j with j + D/2 ("rotate-half"), inverse frequencies
    theta^(-2j/D) in float64, no frequency scaling;
  * a query head h reads KV head floor(h / G), G = H_q / H_kv;
  * scores are scaled by 1/sqrt(D), nothing else (no soft-cap, no bias);
  * link tokens see every earlier global position, including the prefix;
  * the cached prefix (system prompt) sits at positions 0..P-1 and is causal
    within itself; document tokens see only earlier tokens of their own document.

Parity pins for every function are in tests/test_oracle_pins.py.
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import List, Optional, Sequence

import numpy as np

# ---------------------------------------------------------------------------
# bf16 <-> float64
# ---------------------------------------------------------------------------


def bf16_bits_to_f64(u: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float64."""
    u32 = np.asarray(u, dtype=np.uint16).astype(np.uint32) << 16
    with np.errstate(invalid="ignore"):  # signalling-NaN patterns widen to quiet NaN
        return u32.view(np.float32).astype(np.float64)


_BF16_MANT = 8          # significant bits of bf16 (7 stored + hidden bit)
_BF16_EMIN = -126       # smallest normal exponent
_BF16_QUANT_MIN = _BF16_EMIN - (_BF16_MANT - 1)  # spacing of subnormals: 2^-133


def f64_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float64 directly to bf16 (round to nearest, ties to even).

    Rounds once, from the exact double, at the bf16 quantum of the value's
    binade (never via float32, which would round twice).  Overflow gives inf,
    NaN stays NaN.
    """
    x = np.asarray(x, dtype=np.float64)
    out = np.empty(x.shape, dtype=np.float64)
    finite = np.isfinite(x)
    xf = np.where(finite, x, 0.0)
    ax = np.abs(xf)
    # exponent e with 2^e <= |x| < 2^(e+1)
    _, e = np.frexp(ax)
    e = e.astype(np.int64) - 1
    e = np.maximum(e, _BF16_EMIN)                     # subnormals share the min-normal quantum
    q_exp = e - (_BF16_MANT - 1)                      # quantum 2^(e-7)
    q_exp = np.maximum(q_exp, _BF16_QUANT_MIN)
    r = np.ldexp(np.rint(np.ldexp(xf, -q_exp)), q_exp)  # rint = round half to even
    out[...] = r
    out[~finite] = x[~finite]
    # overflow: anything that rounded beyond the largest finite bf16 becomes inf
    bf16_max = np.ldexp(255.0, 127 - 7)               # (2 - 2^-7) * 2^127
    big = np.isfinite(out) & (np.abs(out) > bf16_max)
    out[big] = np.sign(out[big]) * np.inf
    f32 = out.astype(np.float32)                      # exact: out is representable in bf16
    return (f32.view(np.uint32) >> 16).astype(np.uint16)


# ---------------------------------------------------------------------------
# RoPE (Sec. 2.2: k_i = R_i W_k x_i)
# ---------------------------------------------------------------------------


def rope_inv_freq(theta: float, head_dim: int) -> np.ndarray:
    """theta^(-2j/D) for j = 0..D/2-1, in float64."""
    j = np.arange(head_dim // 2, dtype=np.float64)
    return np.power(np.float64(theta), -2.0 * j / np.float64(head_dim))


def rope_rotate(x: np.ndarray, pos, theta: float) -> np.ndarray:
    """Apply R_pos to vectors x[..., D] (float64); pos broadcasts against x[..., 0].

    Pair (j, j + D/2) is rotated by the angle pos * theta^(-2j/D):
        y_j       = x_j cos a - x_{j+D/2} sin a
        y_{j+D/2} = x_{j+D/2} cos a + x_j sin a
    """
    x = np.asarray(x, dtype=np.float64)
    D = x.shape[-1]
    h = D // 2
    a = np.asarray(pos, dtype=np.float64)[..., None] * rope_inv_freq(theta, D)
    c, s = np.cos(a), np.sin(a)
    x1, x2 = x[..., :h], x[..., h:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


# ---------------------------------------------------------------------------
# Layout of one query's linked sequence (Sec. 2.1, Sec. 2.3)
# ---------------------------------------------------------------------------

PREFIX, DOC, LINK, QUESTION = 0, 1, 2, 3


@dataclass
class Layout:
    prefix_len: int
    doc_start: np.ndarray      # int64 [N]: global position of each document's first token
    doc_len: np.ndarray        # int64 [N]
    link_pos: np.ndarray       # int64 [N, K]: global positions of the link tokens
    question_pos: np.ndarray   # int64 [Q]
    kind: np.ndarray           # int8 [C]: PREFIX/DOC/LINK/QUESTION of each position
    owner: np.ndarray          # int64 [C]: document index for DOC/LINK positions, -1 otherwise

    @property
    def total(self) -> int:
        return int(self.kind.shape[0])

    @property
    def fresh_pos(self) -> np.ndarray:
        """Positions of the fresh rows (links and question) in sequence order."""
        return np.flatnonzero((self.kind == LINK) | (self.kind == QUESTION)).astype(np.int64)


def linked_layout(prefix_len: int, doc_lens: Sequence[int], n_link: int, q_len: int) -> Layout:
    """Global positions of [prefix, doc_1, links_1, ..., doc_N, links_N, question].

    Each document c of length L is followed by its K link tokens
    (c_1..c_L, c_link1..c_linkK), Sec. 2.3; documents follow one another in
    retrieval order and the question comes last.  Built token by token.
    """
    kind: List[int] = []
    owner: List[int] = []
    kind += [PREFIX] * prefix_len
    owner += [-1] * prefix_len
    doc_start, link_pos = [], []
    for i, L in enumerate(doc_lens):
        doc_start.append(len(kind))
        kind += [DOC] * int(L)
        owner += [i] * int(L)
        link_pos.append(list(range(len(kind), len(kind) + n_link)))
        kind += [LINK] * n_link
        owner += [i] * n_link
    q0 = len(kind)
    kind += [QUESTION] * q_len
    owner += [-1] * q_len
    return Layout(prefix_len=prefix_len,
                  doc_start=np.asarray(doc_start, dtype=np.int64),
                  doc_len=np.asarray(list(doc_lens), dtype=np.int64),
                  link_pos=np.asarray(link_pos, dtype=np.int64).reshape(len(doc_lens), n_link),
                  question_pos=np.arange(q0, q0 + q_len, dtype=np.int64),
                  kind=np.asarray(kind, dtype=np.int8),
                  owner=np.asarray(owner, dtype=np.int64))


def links_at_end_rows(layout: Layout) -> np.ndarray:
    """Cache row of every position in the physical order of Sec. 2.3 ("Inference"): the
    precomputed caches are loaded and concatenated, and the new link tokens are appended
    at the end of the reordered sequence (for Fig. 2: tokens 1, 2, 4, 5, 7, then links 3,
    6, 8); the question, also run in the forward pass, follows the links.  Positions, and
    so RoPE and the mask, are unchanged; only the row that holds a position moves.
    Returns rows[pos] (int64 [C]).  Built by listing the positions in physical order.
    """
    order = [p for p in range(layout.total) if layout.kind[p] in (PREFIX, DOC)]
    order += [p for p in range(layout.total) if layout.kind[p] == LINK]
    order += [p for p in range(layout.total) if layout.kind[p] == QUESTION]
    rows = np.empty(layout.total, dtype=np.int64)
    for r, p in enumerate(order):
        rows[p] = r
    return rows


# ---------------------------------------------------------------------------
# Masks (Sec. 2.3, Fig. 2)
# ---------------------------------------------------------------------------


def training_mask(layout: Layout) -> np.ndarray:
    """Dense training-time attention map, allowed[r, j], built from the rules in Sec. 2.3:
      * document tokens: local causal, only earlier tokens of the same document;
      * the cached prefix: causal within the prefix;
      * link tokens: every preceding token (earlier documents, earlier links,
        their own document, earlier links of their own group) and themselves;
      * question tokens: standard causal over everything before them.
    """
    C = layout.total
    m = np.zeros((C, C), dtype=bool)
    for r in range(C):
        k = layout.kind[r]
        for j in range(r + 1):
            if k == DOC:
                m[r, j] = layout.kind[j] == DOC and layout.owner[j] == layout.owner[r]
            elif k == PREFIX:
                m[r, j] = layout.kind[j] == PREFIX
            else:  # LINK, QUESTION
                m[r, j] = True
    return m


def inference_mask(fresh_pos: np.ndarray, total: int) -> np.ndarray:
    """Inference-time map for the fresh rows: key position j visible iff j <= pos(r)."""
    fresh_pos = np.asarray(fresh_pos, dtype=np.int64)
    return np.arange(total, dtype=np.int64)[None, :] <= fresh_pos[:, None]


# ---------------------------------------------------------------------------
# Pool access (storage addressing of the cached documents)
# ---------------------------------------------------------------------------


def pool_doc_rows(pool: np.ndarray, doc: int, pool_start, pool_len,
                  block_table: Optional[np.ndarray] = None, block_size: int = 0) -> np.ndarray:
    """Rows [len, H_kv, D] of one cached document from a contiguous or paged pool."""
    L = int(pool_len[doc])
    s = int(pool_start[doc])
    if block_table is None or block_size == 0:
        return pool[s: s + L]
    rows = [pool[int(block_table[s + t // block_size]), t % block_size] for t in range(L)]
    return np.stack(rows) if rows else pool[:0, 0]


# ---------------------------------------------------------------------------
# Re-encode + concat (Sec. 2.2, Sec. 2.1)
# ---------------------------------------------------------------------------


@dataclass
class LinkedCache:
    layout: Layout
    k_bits: np.ndarray     # uint16 [C, H_kv, D]: bf16 keys of the linked cache
    v_bits: np.ndarray     # uint16 [C, H_kv, D]
    k_exact: np.ndarray    # float64 [C, H_kv, D]: re-encoded keys before rounding


def reencode_concat(pool_k: np.ndarray, pool_v: np.ndarray, pool_start, pool_len,
                    prefix_doc: int, doc_ids: Sequence[int], n_link: int,
                    k_new: np.ndarray, v_new: np.ndarray, q_len: int, theta: float,
                    block_table: Optional[np.ndarray] = None, block_size: int = 0) -> LinkedCache:
    """Linked cache of one query.

    pool_k/pool_v: bf16 bits, keys stored rotated at local positions 0..len-1.
    k_new/v_new: bf16 bits [T, H_kv, D] of the query's fresh rows in sequence
    order (links of doc 1, ..., links of doc N, question).
    Document i's keys are rotated by delta_i = its global start position and
    rounded once to bf16; values, the prefix (delta 0) and fresh rows are copied.
    """
    P = int(pool_len[prefix_doc]) if prefix_doc >= 0 else 0
    lens = [int(pool_len[d]) for d in doc_ids]
    lay = linked_layout(P, lens, n_link, q_len)
    C = lay.total
    H, D = pool_k.shape[-2], pool_k.shape[-1]
    kb = np.zeros((C, H, D), dtype=np.uint16)
    vb = np.zeros((C, H, D), dtype=np.uint16)
    kx = np.zeros((C, H, D), dtype=np.float64)

    if P:
        pk = pool_doc_rows(pool_k, prefix_doc, pool_start, pool_len, block_table, block_size)
        pv = pool_doc_rows(pool_v, prefix_doc, pool_start, pool_len, block_table, block_size)
        kb[0:P], vb[0:P] = pk, pv
        kx[0:P] = bf16_bits_to_f64(pk)
    for i, d in enumerate(doc_ids):
        s, L = int(lay.doc_start[i]), lens[i]
        pk = pool_doc_rows(pool_k, d, pool_start, pool_len, block_table, block_size)
        pv = pool_doc_rows(pool_v, d, pool_start, pool_len, block_table, block_size)
        rot = rope_rotate(bf16_bits_to_f64(pk), np.full((L, H), s, dtype=np.int64), theta)
        kx[s: s + L] = rot
        kb[s: s + L] = f64_to_bf16_bits(rot)
        vb[s: s + L] = pv
    fp = lay.fresh_pos
    assert k_new.shape[0] == fp.shape[0], "fresh rows must be N*K + Q"
    kb[fp], vb[fp] = k_new, v_new
    kx[fp] = bf16_bits_to_f64(k_new)
    return LinkedCache(layout=lay, k_bits=kb, v_bits=vb, k_exact=kx)


# ---------------------------------------------------------------------------
# Suffix attention (Sec. 2.3 "Inference"): fresh rows over the linked cache
# ---------------------------------------------------------------------------


def suffix_attention(q: np.ndarray, cache_k: np.ndarray, cache_v: np.ndarray,
                     fresh_pos: np.ndarray, key_pos: Optional[np.ndarray] = None) -> np.ndarray:
    """out[r, h] = softmax_j( q[r,h] . K[j,g] / sqrt(D), pos(j) <= pos(r) ) . V[:, g], g = h // G.

    All arguments float64: q [T, H_q, D], cache_k/cache_v [C, H_kv, D].  key_pos[j] is
    the position held by cache row j (default: row j holds position j, the interleaved
    layout); the mask compares positions, so any physical order of the rows gives the
    same result.
    """
    T, Hq, D = q.shape
    C, Hkv, _ = cache_k.shape
    G = Hq // Hkv
    if key_pos is None:
        allowed = inference_mask(fresh_pos, C)
    else:
        allowed = np.asarray(key_pos, dtype=np.int64)[None, :] <= np.asarray(fresh_pos, dtype=np.int64)[:, None]
    out = np.zeros((T, Hq, D), dtype=np.float64)
    for h in range(Hq):
        g = h // G
        s = (q[:, h, :] @ cache_k[:, g, :].T) / np.sqrt(np.float64(D))
        s = np.where(allowed, s, -np.inf)
        m = s.max(axis=1, keepdims=True)
        p = np.exp(s - m)
        p = p / p.sum(axis=1, keepdims=True)
        out[:, h, :] = p @ cache_v[:, g, :]
    return out


def linked_prefill_query(q_bits: np.ndarray, cache: LinkedCache) -> np.ndarray:
    """Attention output (float64) of one query's fresh rows over its bf16 linked cache."""
    return suffix_attention(bf16_bits_to_f64(q_bits), bf16_bits_to_f64(cache.k_bits),
                            bf16_bits_to_f64(cache.v_bits), cache.layout.fresh_pos)
