// Host plan builder: the segment table of a batch (layout of Sec. 2.3), the
// re-encode work units and the attention work items.  Integer bookkeeping only.
#include <algorithm>
#include <climits>
#include <cstdint>
#include <cstring>
#include <numeric>
#include <queue>
#include <string>

#include "kvlink_internal.h"

namespace kvlink {
namespace {

bool is_pow2(int64_t x) { return x > 0 && (x & (x - 1)) == 0; }

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

int fail(std::string* why, int code, const std::string& msg) {
    if (why) *why = msg;
    return code;
}

}  // namespace

int build_plan(const kvlink_batch_desc_t* d, int32_t num_sms, kvlink_plan* p, std::string* why) {
    if (!d || !p) return fail(why, KVLINK_EINVAL, "null argument");
    if (d->batch <= 0 || d->n_link < 0 || d->pool_docs <= 0 || d->pool_rows <= 0)
        return fail(why, KVLINK_EINVAL, "batch, pool_docs and pool_rows must be > 0, n_link >= 0");
    if (!d->pool_len || !d->pool_start || !d->prefix_doc || !d->n_docs || !d->q_len)
        return fail(why, KVLINK_EINVAL, "null table in the batch description");
    if (d->head_dim != 64 && d->head_dim != 128)
        return fail(why, KVLINK_EUNSUPPORTED, "head_dim must be 64 or 128");
    if (!is_pow2(d->h_kv) || d->h_kv > 16)
        return fail(why, KVLINK_EUNSUPPORTED, "h_kv must be a power of two <= 16");
    if (d->h_q <= 0 || d->h_q % d->h_kv != 0 || !is_pow2(d->h_q / d->h_kv) || d->h_q / d->h_kv > 16)
        return fail(why, KVLINK_EUNSUPPORTED, "h_q / h_kv must be a power of two <= 16");
    const int bs = d->pool_block_size;
    if (bs < 0 || (bs > 0 && bs % 8 != 0))
        return fail(why, KVLINK_EUNSUPPORTED, "pool_block_size must be 0 or a multiple of 8");
    if (bs > 0 && (!d->pool_block_table || d->pool_block_table_len <= 0))
        return fail(why, KVLINK_EINVAL, "paged pool needs its block table");
    if (bs > 0 && d->pool_rows % bs != 0)
        return fail(why, KVLINK_EINVAL, "paged pool_rows must be a multiple of pool_block_size");
    if (num_sms <= 0) return fail(why, KVLINK_EINVAL, "num_sms must be resolved");
    if (d->layout != KVLINK_LAYOUT_INTERLEAVED && d->layout != KVLINK_LAYOUT_LINKS_AT_END)
        return fail(why, KVLINK_EINVAL, "unknown layout");
    if (d->pool_rows > kGrpRowMask) return fail(why, KVLINK_EUNSUPPORTED, "pool_rows above 2^30 - 1");

    p->batch = d->batch;
    p->n_link = d->n_link;
    p->h_q = d->h_q;
    p->h_kv = d->h_kv;
    p->head_dim = d->head_dim;
    p->pool_docs = d->pool_docs;
    p->pool_block_size = bs;
    p->pool_rows = d->pool_rows;
    p->num_sms = num_sms;
    p->layout = d->layout;
    p->pool_len.assign(d->pool_len, d->pool_len + d->pool_docs);
    p->pool_start.assign(d->pool_start, d->pool_start + d->pool_docs);

    // ---- validate the pool: every entry's rows (or blocks) lie inside the pool tensor
    const int64_t n_phys_blocks = bs > 0 ? d->pool_rows / bs : 0;
    if (bs > 0) {
        p->pool_block_table.assign(d->pool_block_table, d->pool_block_table + d->pool_block_table_len);
        for (int64_t i = 0; i < d->pool_block_table_len; ++i)
            if (p->pool_block_table[i] < 0 || p->pool_block_table[i] >= n_phys_blocks)
                return fail(why, KVLINK_EBOUNDS, "pool block id out of range");
    } else {
        p->pool_block_table.clear();
    }
    for (int e = 0; e < d->pool_docs; ++e) {
        const int64_t L = p->pool_len[e], s = p->pool_start[e];
        if (L < 0 || s < 0) return fail(why, KVLINK_EINVAL, "negative pool length or start");
        if (bs > 0) {
            const int64_t nb = (L + bs - 1) / bs;
            if (s + nb > d->pool_block_table_len)
                return fail(why, KVLINK_EBOUNDS, "pool entry runs past the block table");
        } else if (s + L > d->pool_rows) {
            return fail(why, KVLINK_EBOUNDS, "pool entry runs past pool_rows");
        }
    }

    // ---- layout of every query.  Positions: [prefix, doc_1, link_1, ..., doc_N, link_N,
    // question].  Cache rows: the same (interleaved), or the cached entries first and the
    // fresh rows after them in fresh order (links at the end).
    const int B = d->batch, K = d->n_link;
    const bool at_end = d->layout == KVLINK_LAYOUT_LINKS_AT_END;
    int64_t total_docs = 0;
    for (int b = 0; b < B; ++b) {
        if (d->n_docs[b] < 0 || d->q_len[b] < 0) return fail(why, KVLINK_EINVAL, "negative count");
        total_docs += d->n_docs[b];
    }
    if (total_docs > 0 && !d->doc_ids) return fail(why, KVLINK_EINVAL, "doc_ids is null");
    for (int64_t i = 0; i < total_docs; ++i)
        if (d->doc_ids[i] < 0 || d->doc_ids[i] >= d->pool_docs) return fail(why, KVLINK_EBOUNDS, "doc id out of range");

    p->seg.clear();
    p->cu_ctx.assign(B + 1, 0);
    p->cu_fresh.assign(B + 1, 0);
    p->fresh_pos.clear();
    p->fresh_query.clear();
    p->n_rope_rows = 0;
    p->cached_tokens = 0;
    int64_t doc_off = 0, ctx = 0;
    int64_t fresh = 0;
    for (int b = 0; b < B; ++b) {
        p->cu_ctx[b] = ctx;
        p->cu_fresh[b] = (int32_t)fresh;
        int64_t pos = 0;
        const int pre = d->prefix_doc[b];
        if (pre >= d->pool_docs || pre < -1) return fail(why, KVLINK_EBOUNDS, "prefix_doc out of range");
        // cache rows: cached entries from row 0, fresh rows from n_cached (links at the end)
        int64_t n_cached = pre >= 0 ? p->pool_len[pre] : 0;
        for (int i = 0; i < d->n_docs[b]; ++i) n_cached += p->pool_len[d->doc_ids[doc_off + i]];
        int64_t cached_row = 0, fresh_row = n_cached;
        auto row_of = [&](bool cached, int32_t len) -> int64_t {
            if (!at_end) return ctx + pos;
            int64_t& r = cached ? cached_row : fresh_row;
            const int64_t out = ctx + r;
            r += len;
            return out;
        };
        if (pre >= 0 && p->pool_len[pre] > 0) {
            const int32_t P = p->pool_len[pre];
            p->seg.push_back({b, KVLINK_SEG_PREFIX, pre, P, row_of(true, P), (int32_t)pos, -1});
            pos += P;
            p->cached_tokens += P;
        }
        for (int i = 0; i < d->n_docs[b]; ++i) {
            const int doc = d->doc_ids[doc_off + i];
            const int32_t L = p->pool_len[doc];
            if (L > 0) {
                p->seg.push_back({b, KVLINK_SEG_DOC, doc, L, row_of(true, L), (int32_t)pos, p->n_rope_rows++});
                pos += L;
                p->cached_tokens += L;
            }
            if (K > 0) {
                p->seg.push_back({b, KVLINK_SEG_LINK, (int32_t)fresh, K, row_of(false, K), (int32_t)pos, -1});
                for (int k = 0; k < K; ++k) {
                    p->fresh_pos.push_back((int32_t)(pos + k));
                    p->fresh_query.push_back(b);
                }
                fresh += K;
                pos += K;
            }
        }
        doc_off += d->n_docs[b];
        const int Q = d->q_len[b];
        if (Q > 0) {
            p->seg.push_back({b, KVLINK_SEG_QUESTION, (int32_t)fresh, Q, row_of(false, Q), (int32_t)pos, -1});
            for (int k = 0; k < Q; ++k) {
                p->fresh_pos.push_back((int32_t)(pos + k));
                p->fresh_query.push_back(b);
            }
            fresh += Q;
            pos += Q;
        }
        if (p->cu_fresh[b] == fresh) return fail(why, KVLINK_EINVAL, "a query has no fresh rows");
        if (pos > INT32_MAX / 2) return fail(why, KVLINK_EUNSUPPORTED, "context too long");
        ctx += pos;
    }
    p->cu_ctx[B] = ctx;
    p->cu_fresh[B] = (int32_t)fresh;
    if (fresh > INT32_MAX / 64) return fail(why, KVLINK_EUNSUPPORTED, "too many fresh rows");
    if (ctx > kGrpRowMask) return fail(why, KVLINK_EUNSUPPORTED, "linked cache above 2^30 - 1 rows");

    // ---- per-position sources: where each position's K/V row is read from, and its cache row
    p->src.assign((size_t)ctx, kvlink_source_t{0, 0, 0, -1});
    for (const kvlink_segment_t& sg : p->seg) {
        const bool cached = sg.kind == KVLINK_SEG_PREFIX || sg.kind == KVLINK_SEG_DOC;
        for (int t = 0; t < sg.len; ++t) {
            kvlink_source_t& e = p->src[(size_t)(p->cu_ctx[sg.query] + sg.pos + t)];
            if (!cached) {
                e.kind = KVLINK_SRC_FRESH;
                e.row = sg.src + t;
            } else {
                e.kind = KVLINK_SRC_POOL;
                e.row = (int32_t)(bs == 0 ? p->pool_start[sg.src] + t
                                          : (int64_t)p->pool_block_table[p->pool_start[sg.src] + t / bs] * bs + t % bs);
            }
            e.slot = (int32_t)(sg.dst + t);
            e.table = sg.table;
        }
    }

    // ---- the same records in cache-row order, and the visibility of every fresh row
    p->src_row.assign((size_t)ctx, kvlink_source_t{0, 0, 0, -1});
    for (const kvlink_source_t& e : p->src) p->src_row[(size_t)e.slot] = e;
    p->fresh_vis.assign(p->fresh_pos.size(), 0);
    p->fresh_row0.assign(B, kNoFreshRegion);
    for (int b = 0; b < B; ++b) {
        const int32_t f0 = p->cu_fresh[b], T = p->cu_fresh[b + 1] - f0;
        const int64_t C = p->cu_ctx[b + 1] - p->cu_ctx[b];
        if (at_end) p->fresh_row0[b] = (int32_t)(C - T);
        for (int32_t f = 0; f < T; ++f) {
            const int32_t pos = p->fresh_pos[f0 + f];
            // links at the end: the cached rows before the position (f of the pos earlier
            // positions are fresh); interleaved: every row up to the position
            p->fresh_vis[f0 + f] = at_end ? pos - f : pos + 1;
        }
    }

    // ---- the cache row of every fresh row (the fresh-row placement)
    p->fresh_dst.assign(p->fresh_pos.size(), 0);
    for (const kvlink_segment_t& sg : p->seg)
        if (sg.kind == KVLINK_SEG_LINK || sg.kind == KVLINK_SEG_QUESTION)
            for (int t = 0; t < sg.len; ++t) p->fresh_dst[(size_t)sg.src + t] = (int32_t)(sg.dst + t);

    // ---- groups of 8 cache rows whose sources are consecutive in one tensor: each is one
    // 8-row TMA copy in the one-kernel path
    p->cu_grp.assign(B + 1, 0);
    p->grp_src.clear();
    for (int b = 0; b < B; ++b) {
        const int64_t c0 = p->cu_ctx[b], C = p->cu_ctx[b + 1] - c0;
        p->cu_grp[b] = (int32_t)p->grp_src.size();
        for (int64_t m = 0; m * 8 < C; ++m) {
            int32_t gs = -1;
            if (m * 8 + 8 <= C) {
                const kvlink_source_t* e = &p->src_row[(size_t)(c0 + m * 8)];
                bool run = true;
                for (int i = 1; i < 8; ++i) run = run && e[i].kind == e[0].kind && e[i].row == e[0].row + i;
                if (run) gs = e[0].row | (e[0].kind == KVLINK_SRC_FRESH ? kGrpFresh : 0);
            }
            p->grp_src.push_back(gs);
        }
    }
    p->cu_grp[B] = (int32_t)p->grp_src.size();

    // ---- re-encode work units: cached segments first, then fresh segments.  A unit never
    // crosses a pool block, so its source rows, like its cache rows, are contiguous.
    p->chunks.clear();
    const int ct = copy_chunk_tokens(d->h_kv * d->head_dim * 2);
    for (int pass = 0; pass < 2; ++pass) {
        for (size_t s = 0; s < p->seg.size(); ++s) {
            const kvlink_segment_t& sg = p->seg[s];
            const bool cached = sg.kind == KVLINK_SEG_PREFIX || sg.kind == KVLINK_SEG_DOC;
            if (cached != (pass == 0)) continue;
            for (int t = 0; t < sg.len;) {
                int n = std::min(ct, sg.len - t);
                int64_t src;
                if (!cached) {
                    src = (int64_t)sg.src + t;
                } else if (bs == 0) {
                    src = p->pool_start[sg.src] + t;
                } else {
                    n = std::min(n, bs - t % bs);
                    src = (int64_t)p->pool_block_table[p->pool_start[sg.src] + t / bs] * bs + t % bs;
                }
                p->chunks.push_back({src, sg.dst + t, n, sg.kind, sg.table, (int32_t)s});
                t += n;
            }
        }
        if (pass == 0) p->n_chunks_cached = (int32_t)p->chunks.size();
    }
    // the cached chunks ordered by source row, for the all-layer re-encode: the chunks of a
    // document that several queries retrieved become adjacent, and the kernel loads their
    // rows once for all destinations
    p->chunks_sorted.assign(p->chunks.begin(), p->chunks.begin() + p->n_chunks_cached);
    std::stable_sort(p->chunks_sorted.begin(), p->chunks_sorted.end(), [](const CopyChunk& a, const CopyChunk& b) {
        return a.src_row != b.src_row ? a.src_row < b.src_row : a.n < b.n;
    });
    // ---- attention work items
    // M-tiles of one (query, KV head) cut the query's fresh tokens into runs of kAttnBM / G
    // tokens counted back from the last one, the remainder going to the first run: a tile's
    // key range ends at its last token, so the padding rows of a partial tile cost least in
    // the tile with the shortest range (the earliest link tokens).
    const int G = d->h_q / d->h_kv;
    const int tok_per_tile = kAttnBM / G;
    struct Tile { int32_t b, g, t0, t1, n_tiles, min_vis, owner, a_tiles, b_tile0; };
    std::vector<Tile> tiles;
    int64_t work = 0;
    p->attn_pairs = 0;
    for (int b = 0; b < B; ++b) {
        const int32_t f0 = p->cu_fresh[b], T = p->cu_fresh[b + 1] - f0;
        for (int r = 0; r < T; ++r) p->attn_pairs += (int64_t)p->fresh_pos[f0 + r] + 1;
        const int n_mt = (T + tok_per_tile - 1) / tok_per_tile;
        for (int g = 0; g < d->h_kv; ++g) {
            for (int mt = 0; mt < n_mt; ++mt) {
                const int t0 = mt == 0 ? 0 : T - (n_mt - mt) * tok_per_tile;
                const int t1 = T - (n_mt - 1 - mt) * tok_per_tile;
                // visibility grows with position, so the tile's last row sees the most
                int32_t a_tiles = (p->fresh_vis[f0 + t1 - 1] + kAttnBN - 1) / kAttnBN;
                int32_t b_tile0 = 0, b_tiles = 0;
                if (p->fresh_row0[b] != kNoFreshRegion) {
                    const int32_t F = p->fresh_row0[b];
                    b_tile0 = F / kAttnBN;
                    const int32_t b_end = (F + t1 + kAttnBN - 1) / kAttnBN;
                    if (b_tile0 <= a_tiles) {  // the runs touch: one run from row 0
                        a_tiles = std::max(a_tiles, b_end);
                    } else {
                        b_tiles = b_end - b_tile0;
                    }
                }
                const int32_t nt = a_tiles + b_tiles;
                tiles.push_back({b, g, t0, t1, nt, p->fresh_vis[f0 + t0], mt == n_mt - 1 ? 1 : 0, a_tiles, b_tile0});
                work += nt;
            }
        }
    }
    // Split KV ranges into pieces of at most max_tiles key tiles (partials merged afterwards).
    auto make_items = [&](int32_t max_tiles, std::vector<AttnItem>& items, std::vector<MergeGroup>& merges,
                          int32_t& n_slots) {
        items.clear();
        merges.clear();
        n_slots = 0;
        for (const Tile& t : tiles) {
            const int32_t n_split = (t.n_tiles + max_tiles - 1) / max_tiles;
            if (n_split <= 1) {
                items.push_back({t.b, t.g, t.t0, t.t1, 0, t.n_tiles, -1, t.min_vis, t.owner, t.a_tiles, t.b_tile0});
                continue;
            }
            merges.push_back({t.b, t.g, t.t0, t.t1, n_slots, n_split, 0, 0});
            for (int s = 0; s < n_split; ++s) {
                const int32_t a = (int32_t)((int64_t)t.n_tiles * s / n_split);
                const int32_t e = (int32_t)((int64_t)t.n_tiles * (s + 1) / n_split);
                items.push_back({t.b, t.g, t.t0, t.t1, a, e, n_slots + s, t.min_vis, t.owner, t.a_tiles, t.b_tile0});
            }
            n_slots += n_split;
        }
        // Launch order.  The items of one (query, KV head) stay adjacent, so that CTAs running
        // at the same time read the same K/V tiles (served from L2 after the first); groups go
        // longest first, and so do the items inside a group.  Items of at most 55% of the
        // longest item's key tiles are held back to the end, longest first: run inside their
        // groups they leave the long items of the last groups to start late and run alone at
        // the end of the grid, while at the end they fill the gaps of the last wave (their K/V
        // tiles, a prefix of their group's, are read once more).
        std::vector<int64_t> group_cost((size_t)B * d->h_kv, 0);
        int64_t longest = 0;
        for (const AttnItem& it : items) {
            const int64_t c = it.kv_tile1 - it.kv_tile0;
            int64_t& g = group_cost[(size_t)it.query * d->h_kv + it.kv_head];
            g = std::max(g, c);
            longest = std::max(longest, c);
        }
        std::stable_sort(items.begin(), items.end(), [&](const AttnItem& x, const AttnItem& y) {
            const int64_t cx = x.kv_tile1 - x.kv_tile0, cy = y.kv_tile1 - y.kv_tile0;
            const bool late_x = cx * 100 <= longest * 55, late_y = cy * 100 <= longest * 55;
            if (late_x != late_y) return late_y;
            if (!late_x) {
                const int64_t gx = group_cost[(size_t)x.query * d->h_kv + x.kv_head];
                const int64_t gy = group_cost[(size_t)y.query * d->h_kv + y.kv_head];
                if (gx != gy) return gx > gy;
            } else if (cx != cy) {
                return cx > cy;
            }
            if (x.query != y.query) return x.query < y.query;
            if (x.kv_head != y.kv_head) return x.kv_head < y.kv_head;
            return cx > cy;
        });
    };

    // The persistent attention's schedule: one CTA per SM (fewer with fewer items), each item
    // handed to the CTA that would be free first (list scheduling on the estimated cost in
    // half tiles: two per key tile, one for the item's own start and finish, two more for a
    // piece of a split range, whose partial is stored and merged).  Two hand-out orders are
    // estimated: the launch order (the items of one (query, KV head) run together and share
    // their K/V tiles in L2) and longest first over all items; the launch order is kept
    // unless longest first finishes more than 3% earlier (a few long groups filling the
    // grid: one long query's last KV head would otherwise start only after a first item
    // elsewhere).
    using Slot = std::pair<int64_t, int32_t>;
    auto cost = [](const AttnItem& it) { return 2 * (int64_t)(it.kv_tile1 - it.kv_tile0) + 1 + (it.slot >= 0 ? 2 : 0); };
    auto schedule = [&](const std::vector<AttnItem>& items, const std::vector<int32_t>& order, int32_t n_ctas,
                        std::vector<std::vector<int32_t>>* lists) {
        std::priority_queue<Slot, std::vector<Slot>, std::greater<Slot>> free_at;
        for (int32_t c = 0; c < n_ctas; ++c) free_at.push({0, c});
        if (lists) lists->assign((size_t)n_ctas, {});
        int64_t makespan = 0;
        for (int32_t i : order) {
            const Slot sl = free_at.top();
            free_at.pop();
            if (lists) (*lists)[(size_t)sl.second].push_back(i);
            makespan = std::max(makespan, sl.first + cost(items[(size_t)i]));
            free_at.push({sl.first + cost(items[(size_t)i]), sl.second});
        }
        return makespan;
    };
    // returns the estimated makespan and the better order
    auto best_order = [&](const std::vector<AttnItem>& items, int32_t n_ctas, std::vector<int32_t>& order) {
        std::vector<int32_t> launch(items.size()), longest_first;
        std::iota(launch.begin(), launch.end(), 0);
        longest_first = launch;
        std::stable_sort(longest_first.begin(), longest_first.end(),
                         [&](int32_t a, int32_t b) { return cost(items[(size_t)a]) > cost(items[(size_t)b]); });
        const int64_t m_launch = schedule(items, launch, n_ctas, nullptr);
        const int64_t m_longest = schedule(items, longest_first, n_ctas, nullptr);
        const bool use_longest = m_longest * 103 < m_launch * 100;
        order = use_longest ? longest_first : launch;
        return use_longest ? m_longest : m_launch;
    };

    // Split granularity: pieces of at most W / (k * SMs) key tiles (W the batch's key tiles),
    // for the k in 1..4 whose estimated time is shortest (a larger k only when it is more
    // than 2% shorter): with many short items nothing is split; one long query, or a batch
    // whose longest items would hold the grid up, is split just enough to balance.  The
    // estimate adds the merge pass, which runs after the attention and reads every partial
    // (O, m, l: about 130 KB for head_dim 128, written once and read once): at HBM speed
    // one half tile of attention time moves about 19 partials, plus about 5 half tiles for
    // the launch.
    int64_t best_span = INT64_MAX;
    std::vector<int32_t> best_ord;
    for (int k = 1; k <= 4; ++k) {
        const int32_t max_tiles = (int32_t)std::max<int64_t>(8, (work + (int64_t)num_sms * k - 1) / ((int64_t)num_sms * k));
        std::vector<AttnItem> items;
        std::vector<MergeGroup> merges;
        int32_t n_slots = 0;
        make_items(max_tiles, items, merges, n_slots);
        const int32_t n_ctas = std::min<int32_t>(num_sms, (int32_t)items.size());
        std::vector<int32_t> order;
        const int64_t span = best_order(items, n_ctas, order) + (n_slots > 0 ? 5 + n_slots / 19 : 0);
        if (k == 1 || span * 100 < best_span * 98) {
            best_span = span;
            p->items.swap(items);
            p->merges.swap(merges);
            p->n_slots = n_slots;
            best_ord.swap(order);
        }
        if (max_tiles == 8) break;   // finer pieces are not made
    }
    p->workspace_bytes = (size_t)p->n_slots * (size_t)kAttnBM * ((size_t)d->head_dim + 2) * sizeof(float);
    {
        const int32_t n_ctas = std::min<int32_t>(num_sms, (int32_t)p->items.size());
        std::vector<std::vector<int32_t>> lists;
        schedule(p->items, best_ord, n_ctas, &lists);
        p->sched.clear();
        p->cu_sched.assign((size_t)n_ctas + 1, 0);
        for (int32_t c = 0; c < n_ctas; ++c) {
            p->cu_sched[(size_t)c] = (int32_t)p->sched.size();
            p->sched.insert(p->sched.end(), lists[(size_t)c].begin(), lists[(size_t)c].end());
        }
        p->cu_sched[(size_t)n_ctas] = (int32_t)p->sched.size();
    }

    // ---- device buffer layout (256-byte aligned tables)
    size_t off = 0;
    auto take = [&](size_t bytes) { size_t o = off; off = align_up(off + bytes, 256); return o; };
    p->off_seg = take(p->seg.size() * sizeof(kvlink_segment_t));
    p->off_chunks = take(p->chunks.size() * sizeof(CopyChunk));
    p->off_chunks_sorted = take(p->chunks_sorted.size() * sizeof(CopyChunk));
    p->off_rope = take((size_t)p->n_rope_rows * (d->head_dim / 2) * sizeof(float4));
    p->off_pool_start = take(p->pool_start.size() * sizeof(int64_t));
    p->off_pool_bt = take(p->pool_block_table.size() * sizeof(int32_t));
    p->off_cu_ctx = take(p->cu_ctx.size() * sizeof(int64_t));
    p->off_cu_fresh = take(p->cu_fresh.size() * sizeof(int32_t));
    p->off_fresh_pos = take(p->fresh_pos.size() * sizeof(int32_t));
    p->off_fresh_query = take(p->fresh_query.size() * sizeof(int32_t));
    p->off_items = take(p->items.size() * sizeof(AttnItem));
    p->off_merges = take(p->merges.size() * sizeof(MergeGroup));
    p->off_src = take(p->src.size() * sizeof(kvlink_source_t));
    p->off_cu_grp = take(p->cu_grp.size() * sizeof(int32_t));
    p->off_grp_src = take(p->grp_src.size() * sizeof(int32_t));
    p->off_src_row = take(p->src_row.size() * sizeof(kvlink_source_t));
    p->off_fresh_vis = take(p->fresh_vis.size() * sizeof(int32_t));
    p->off_fresh_row0 = take(p->fresh_row0.size() * sizeof(int32_t));
    p->off_fresh_dst = take(p->fresh_dst.size() * sizeof(int32_t));
    p->off_sched = take(p->sched.size() * sizeof(int32_t));
    p->off_cu_sched = take(p->cu_sched.size() * sizeof(int32_t));
    p->device_bytes = off;
    p->uploaded = false;
    return KVLINK_OK;
}

}  // namespace kvlink
