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
    // ---- work items and the persistent attention's schedule.
    // Costs are in half tiles: two per key tile, one for an item's own start and finish.  The
    // schedules below are built and the one with the shorter estimated time is kept:
    //  A  whole M-tiles in launch order, each to the CTA with the least work so far (list
    //     scheduling; also tried longest first over all M-tiles).  The launch order keeps the
    //     M-tiles of one (query, KV head) together, groups with the longest M-tile first, so
    //     that CTAs working at the same time share their K/V tiles in L2; M-tiles of at most
    //     55% of the longest are held back to the end, longest first, where they fill the
    //     gaps of the last wave (when the longest M-tile is more than a quarter of a CTA's
    //     share; otherwise the groups simply go by their key tiles).  Balance is limited by the
    //     M-tile size: a CTA holding two long M-tiles ends late.
    //  B  the same list scheduling (M-tiles of a group together, groups with the most key
    //     tiles first) with every CTA capped at an equal share of the whole: an M-tile that
    //     would carry a CTA past its share is cut, the CTA keeps the key tiles that fit and the
    //     rest goes on to the next CTA with the least work.  The pieces of a cut M-tile write
    //     partial results (O, m, l), merged inside the persistent kernel by the piece that
    //     completes the group (or by attn_merge_kernel after the one-item-per-CTA kernels).
    //     The estimate charges every CTA holding a piece kMergeCost for the partial store and
    //     the merge (epilogue work that also takes issue slots from the softmax), so B is also
    //     tried with shares 5% and 10% above the mean, where fewer M-tiles are cut.  One long
    //     query (M-tiles of a few hundred key tiles) needs B.
    //  G  gangs (below): every group whole on one gang of CTAs, for many short M-tiles.
    // Small batches use fewer CTAs (at least kMinShare half tiles each) and never cut a piece
    // under kMinPiece key tiles.
    struct Sched {
        std::vector<AttnItem> items;
        std::vector<MergeGroup> merges;
        std::vector<std::vector<int32_t>> lists;
        int32_t n_slots = 0;
        int64_t span = 0;
    };
    constexpr int64_t kItemCost = 1;   // half tiles for an item's start and finish (4, 8, 14: no change)
    constexpr int64_t kMinShare = 2 * 8 + kItemCost;
    constexpr int32_t kMinPiece = 4;
    constexpr int64_t kMergeCost = 14;
    int64_t total = 0;
    for (const Tile& t : tiles) total += 2 * (int64_t)t.n_tiles + kItemCost;
    const int32_t n_ctas = (int32_t)std::max<int64_t>(1, std::min<int64_t>(num_sms, total / kMinShare));
    using Slot = std::pair<int64_t, int32_t>;      // (work so far, CTA)
    auto item_of = [](const Tile& t, int32_t a, int32_t e) {
        return AttnItem{t.b, t.g, t.t0, t.t1, a, e, -1, t.min_vis, t.owner, t.a_tiles, t.b_tile0};
    };
    auto group_key = [&](const std::vector<int64_t>& gc, const Tile& t) { return gc[(size_t)t.b * d->h_kv + t.g]; };

    // A: whole M-tiles, list scheduled in the given order
    auto schedule_whole = [&](const std::vector<Tile>& order) {
        Sched s;
        s.lists.assign((size_t)n_ctas, {});
        std::priority_queue<Slot, std::vector<Slot>, std::greater<Slot>> least;
        for (int32_t c = 0; c < n_ctas; ++c) least.push({0, c});
        for (const Tile& t : order) {
            const Slot sl = least.top();
            least.pop();
            s.lists[(size_t)sl.second].push_back((int32_t)s.items.size());
            s.items.push_back(item_of(t, 0, t.n_tiles));
            const int64_t load = sl.first + 2 * (int64_t)t.n_tiles + kItemCost;
            s.span = std::max(s.span, load);
            least.push({load, sl.second});
        }
        return s;
    };
    // B: capped shares, M-tiles cut at the cap
    auto schedule_capped = [&](const std::vector<Tile>& order, int slack_pct) {
        Sched s;
        s.lists.assign((size_t)n_ctas, {});
        std::vector<int32_t> pieces_on((size_t)n_ctas, 0);
        // the equal share, plus room for the starts of two more pieces and slack_pct percent:
        // with slack, an M-tile is cut only where a CTA would otherwise end well past the mean
        int64_t share = (total + n_ctas - 1) / n_ctas * (100 + slack_pct) / 100 + 2 * kItemCost;
        std::priority_queue<Slot, std::vector<Slot>, std::greater<Slot>> least;
        for (int32_t c = 0; c < n_ctas; ++c) least.push({0, c});
        for (const Tile& t : order) {
            const size_t first_piece = s.items.size();
            std::vector<int32_t> ctas;
            int32_t done = 0;
            while (done < t.n_tiles) {
                // every CTA full (a cut adds a start the shares did not count): all shares grow
                while (least.top().first + kItemCost + 2 > share) share += 2;
                const Slot sl = least.top();
                least.pop();
                const int32_t rest = t.n_tiles - done;
                int32_t m = (int32_t)std::min<int64_t>(rest, (share - sl.first - kItemCost) / 2);
                // no piece under kMinPiece key tiles: the CTA rather runs a little past its share
                if (m < rest) {
                    if (m < kMinPiece) m = std::min(rest, kMinPiece);
                    else if (rest - m < kMinPiece) m = rest;
                }
                s.lists[(size_t)sl.second].push_back((int32_t)s.items.size());
                s.items.push_back(item_of(t, done, done + m));
                ctas.push_back(sl.second);
                least.push({sl.first + 2 * (int64_t)m + kItemCost, sl.second});
                done += m;
            }
            const int32_t n_split = (int32_t)(s.items.size() - first_piece);
            if (n_split > 1) {
                s.merges.push_back({t.b, t.g, t.t0, t.t1, s.n_slots, n_split, 0, 0});
                for (int32_t i = 0; i < n_split; ++i) s.items[first_piece + (size_t)i].slot = s.n_slots + i;
                s.n_slots += n_split;
                for (int32_t c : ctas) ++pieces_on[(size_t)c];
            }
        }
        while (!least.empty()) {
            const Slot sl = least.top();
            least.pop();
            s.span = std::max(s.span, sl.first + kMergeCost * pieces_on[(size_t)sl.second]);
        }
        return s;
    };

    // G: gangs of S CTAs.  Every (query, KV head) group goes whole to one gang (the gang with
    // the least work, groups by decreasing work), its M-tiles to the gang's CTAs with the least
    // work, so the CTAs of a gang run the same group's M-tiles at about the same time and read
    // its K/V tiles once from DRAM between them (the others hit L2).
    auto schedule_gang = [&](const std::vector<Tile>& order, int32_t S) {
        Sched s;
        s.lists.assign((size_t)n_ctas, {});
        const int32_t n_gangs = n_ctas / S;
        std::vector<int64_t> load((size_t)n_ctas, 0);
        std::priority_queue<Slot, std::vector<Slot>, std::greater<Slot>> gangs;   // (work, gang)
        for (int32_t q = 0; q < n_gangs; ++q) gangs.push({0, q});
        for (size_t i = 0; i < order.size();) {
            size_t j = i;
            while (j < order.size() && order[j].b == order[i].b && order[j].g == order[i].g) ++j;
            const Slot gs = gangs.top();
            gangs.pop();
            const int32_t c0 = gs.second * S;
            for (size_t k = i; k < j; ++k) {
                int32_t c = c0;
                for (int32_t x = c0 + 1; x < c0 + S; ++x)
                    if (load[(size_t)x] < load[(size_t)c]) c = x;
                s.lists[(size_t)c].push_back((int32_t)s.items.size());
                s.items.push_back(item_of(order[k], 0, order[k].n_tiles));
                load[(size_t)c] += 2 * (int64_t)order[k].n_tiles + kItemCost;
            }
            int64_t gl = 0;
            for (int32_t x = c0; x < c0 + S; ++x) gl = std::max(gl, load[(size_t)x]);
            gangs.push({gl, gs.second});
            i = j;
        }
        s.span = *std::max_element(load.begin(), load.end());
        return s;
    };

    std::vector<int64_t> longest_in_group((size_t)B * d->h_kv, 0), tiles_in_group((size_t)B * d->h_kv, 0);
    int64_t longest = 0;
    for (const Tile& t : tiles) {
        int64_t& lg = longest_in_group[(size_t)t.b * d->h_kv + t.g];
        lg = std::max<int64_t>(lg, t.n_tiles);
        tiles_in_group[(size_t)t.b * d->h_kv + t.g] += t.n_tiles;
        longest = std::max<int64_t>(longest, t.n_tiles);
    }
    auto by_group = [&](const std::vector<int64_t>& gc, bool defer_short) {
        std::vector<Tile> v = tiles;
        std::stable_sort(v.begin(), v.end(), [&](const Tile& x, const Tile& y) {
            const int64_t cx = x.n_tiles, cy = y.n_tiles;
            const bool late_x = defer_short && cx * 100 <= longest * 55, late_y = defer_short && cy * 100 <= longest * 55;
            if (late_x != late_y) return late_y;
            if (!late_x) {
                const int64_t gx = group_key(gc, x), gy = group_key(gc, y);
                if (gx != gy) return gx > gy;
            } else if (cx != cy) {
                return cx > cy;
            }
            if (x.b != y.b) return x.b < y.b;
            if (x.g != y.g) return x.g < y.g;
            return cx > cy;
        });
        return v;
    };
    std::vector<Tile> longest_first = tiles;
    std::stable_sort(longest_first.begin(), longest_first.end(),
                     [](const Tile& x, const Tile& y) { return x.n_tiles > y.n_tiles; });
    // holding short M-tiles back pays when the longest M-tile is a large part of a CTA's share
    // (its tail decides when the grid ends); otherwise the plain group order keeps the
    // groups' K/V tiles together longer
    const bool defer_short = 2 * longest * 4 > (total + n_ctas - 1) / n_ctas;
    Sched a_launch = schedule_whole(defer_short ? by_group(longest_in_group, true) : by_group(tiles_in_group, false));
    Sched a_longest = schedule_whole(longest_first);
    Sched best = std::move(a_longest.span * 103 < a_launch.span * 100 ? a_longest : a_launch);
    // A repaired: while the most loaded CTA ends more than two piece costs after the least
    // loaded one, its last whole M-tile is cut in two and the second piece moves to the end of
    // the least loaded CTA (a two-piece merge); only the CTAs that hold the grid up are cut.
    {
        Sched r = best;
        std::vector<int64_t> load((size_t)n_ctas, 0);
        for (int32_t c = 0; c < n_ctas; ++c)
            for (int32_t i : r.lists[(size_t)c])
                load[(size_t)c] += 2 * (int64_t)(r.items[(size_t)i].kv_tile1 - r.items[(size_t)i].kv_tile0) + kItemCost;
        for (int32_t step = 0; step < n_ctas; ++step) {
            const int32_t hi = (int32_t)(std::max_element(load.begin(), load.end()) - load.begin());
            const int32_t lo = (int32_t)(std::min_element(load.begin(), load.end()) - load.begin());
            const int64_t gap = load[(size_t)hi] - load[(size_t)lo];
            if (gap <= 4 * kMergeCost || r.lists[(size_t)hi].empty()) break;
            const int32_t idx = r.lists[(size_t)hi].back();
            AttnItem& it = r.items[(size_t)idx];
            if (it.slot >= 0) break;
            const int32_t n = it.kv_tile1 - it.kv_tile0;
            // move x tiles so that both ends meet: 2x = (gap - 1) / 2 (each side pays kMergeCost)
            int32_t x = (int32_t)std::min<int64_t>(n - kMinPiece, (gap - 1) / 4);
            if (x < kMinPiece) break;
            AttnItem moved = it;
            moved.kv_tile0 = it.kv_tile1 - x;
            it.kv_tile1 = moved.kv_tile0;
            it.slot = r.n_slots;
            moved.slot = r.n_slots + 1;
            r.merges.push_back({it.query, it.kv_head, it.tok0, it.tok1, r.n_slots, 2, 0, 0});
            r.n_slots += 2;
            r.lists[(size_t)lo].push_back((int32_t)r.items.size());
            r.items.push_back(moved);
            load[(size_t)hi] += -2 * (int64_t)x + kMergeCost;
            load[(size_t)lo] += 2 * (int64_t)x + kItemCost + kMergeCost;
        }
        r.span = *std::max_element(load.begin(), load.end());
        if (r.span * 100 < best.span * 97) best = std::move(r);
    }
    for (int slack : {0, 5, 10}) {
        Sched capped = schedule_capped(by_group(tiles_in_group, false), slack);
        if (capped.span * 100 < best.span * 97) best = std::move(capped);
    }
    // Many short M-tiles per CTA: the list schedules scatter a group's M-tiles over time and the
    // attention turns DRAM-bound on re-read K/V tiles; gangs of as many CTAs as a group has
    // M-tiles (at most 8) keep them together.  Taken when the CTAs run at least four M-tiles each
    // and the gangs' estimated time is within 10 % of the best, which the shared K/V tiles more
    // than repay: workload 5 (64 queries, 2096 M-tiles of about 23 key tiles, estimate 596
    // against 562) measured 258.9 against 291.1 us per layer with gangs of 6 (gangs of 2: 298.2,
    // 4: 259.1, 8: 253.9 with a slower step); forced on workloads 3 and 4 (384 and 160 M-tiles,
    // estimates 21 % and 121 % above the best) gangs measured 93.8 against 81.9 and 454 against
    // 226 us.
    {
        constexpr int64_t kGangMinItemsPerCta = 4;
        constexpr int64_t kGangSlackPct = 10;
        int32_t mt_max = 0;
        std::vector<int32_t> mt_in_group((size_t)B * d->h_kv, 0);
        for (const Tile& t : tiles) mt_max = std::max(mt_max, ++mt_in_group[(size_t)t.b * d->h_kv + t.g]);
        const int32_t S = std::min<int32_t>(mt_max, 8);
        if (S >= 2 && n_ctas >= 4 * S && (int64_t)tiles.size() >= kGangMinItemsPerCta * (int64_t)n_ctas) {
            Sched gang = schedule_gang(by_group(tiles_in_group, false), S);
            if (gang.span * 100 <= best.span * (100 + kGangSlackPct)) best = std::move(gang);
        }
    }

    p->items.swap(best.items);
    p->merges.swap(best.merges);
    p->n_slots = best.n_slots;
    p->sched.clear();
    p->cu_sched.assign((size_t)n_ctas + 1, 0);
    for (int32_t c = 0; c < n_ctas; ++c) {
        p->cu_sched[(size_t)c] = (int32_t)p->sched.size();
        p->sched.insert(p->sched.end(), best.lists[(size_t)c].begin(), best.lists[(size_t)c].end());
    }
    p->cu_sched[(size_t)n_ctas] = (int32_t)p->sched.size();
    (void)work;
    p->workspace_bytes = (size_t)p->n_slots * (size_t)kAttnBM * ((size_t)d->head_dim + 2) * sizeof(float);
    p->slot_group.assign((size_t)p->n_slots, -1);
    for (size_t g = 0; g < p->merges.size(); ++g)
        for (int32_t s = 0; s < p->merges[g].n_split; ++s) p->slot_group[(size_t)(p->merges[g].slot0 + s)] = (int32_t)g;

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
    p->off_slot_group = take(p->slot_group.size() * sizeof(int32_t));
    p->off_merge_count = take(p->merges.size() * sizeof(unsigned long long));
    p->device_bytes = off;
    p->uploaded = false;
    return KVLINK_OK;
}

}  // namespace kvlink
