/*
 * kvlink.h - C ABI of the GB300 (sm_103a) KVLink linked-prefill library.
 *
 * KVLink (arXiv 2502.16002) precomputes every document's KV cache on its own
 * (Sec. 2.1).  At inference the retrieved documents' caches are re-encoded to
 * their global positions (Sec. 2.2), concatenated with K link tokens after every
 * document (Sec. 2.3), and only the fresh link and question tokens are run,
 * attending over the linked cache under KVLink's mask (Sec. 2.3, Fig. 2).  This
 * library is the per-layer attention-side work of that step:
 *
 *   kvlink_plan_create / _rebuild / _upload     segment table and RoPE delta table
 *   kvlink_reencode_concat                      re-encode + gather/concat cached K/V
 *   kvlink_suffix_attention                     fresh rows attend over the linked cache
 *   kvlink_linked_prefill                       both, chained, for one layer
 *   kvlink_linked_prefill_layers[_overlapped]   every layer in one call (the re-encode of
 *                                               all layers on a second stream)
 *   kvlink_linked_prefill_layers_host           the same from and to host memory
 *   kvlink_reencode_concat_host_pool,           the document cache pool in host memory
 *   kvlink_linked_prefill_layers_host_pool      (Sec. 3.3), read over the host link
 *   kvlink_linked_prefill_fused                 one kernel per layer (keys rotated on load)
 *   kvlink_reencode_concat_layers, kvlink_rope_fresh, kvlink_suffix_attention_simt,
 *   kvlink_suffix_attention_noalloc, kvlink_device_status, kvlink_selftest_wait_timeout
 *
 * libkvlink_debug.so is the same ABI built with device-side checks of every index table
 * entry the kernels use (KVLINK_STATUS_BAD_INDEX_*).
 *
 * Conventions shared by every call
 *   - Tensors are bf16, "NHD" per layer: [rows][heads][head_dim], rows contiguous.
 *   - Pointers named d_* or documented as "device" are device memory; "host"
 *     pointers are read during the call only.  The caller owns every buffer; the
 *     library allocates no device memory.  A plan owns host memory only: its tables
 *     (kvlink_plan_create), a pinned staging buffer (kvlink_plan_upload) and the CUDA
 *     events of the all-layers calls, all freed by kvlink_plan_destroy.  Calls that use
 *     one plan must not run concurrently from several host threads.
 *   - Device work is enqueued on `stream` (a cudaStream_t; NULL = legacy default)
 *     and is asynchronous.  Arguments are validated on the host before anything is
 *     launched; a call that returns an error has launched nothing.
 *   - Return value: KVLINK_OK (0) or a negative KVLINK_E* code.  No C++ exception
 *     crosses the ABI.  kvlink_strerror() names a code.
 *   - Kernels never trap.  A wait inside a kernel that exceeds its bounded spin
 *     count records a code in a device status word (kvlink_device_status) and the
 *     kernel returns early; its outputs are then undefined.
 *
 * Sequence layout of one query b (Sec. 2.3: link tokens follow every document):
 *   [prefix (P tokens), doc_1 (l_1), link_1 (K), doc_2, link_2, ..., doc_N, link_N,
 *    question (Q_b)]
 *   In the default (interleaved) layout a position's row in the query's linked
 *   cache equals its global position; the links-at-end layout (KVLINK_LAYOUT_*)
 *   stores the same positions in another order.
 *   The prefix is an optional cached pool entry (e.g. a system prompt) at
 *   positions 0..P-1.  Cached document i starts at s_i and its keys, stored rotated
 *   at local positions 0..l_i-1, are rotated by delta_i = s_i (Sec. 2.2).
 *   Fresh rows of query b (link tokens then question tokens, in sequence order)
 *   are rows cu_fresh[b] .. cu_fresh[b+1]-1 of q/k_new/v_new/out.
 */
#ifndef KVLINK_H
#define KVLINK_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* kvlink_stream_t; /* same type as cudaStream_t */

enum {
    KVLINK_OK = 0,
    KVLINK_EINVAL = -1,       /* null pointer, negative count, inconsistent description */
    KVLINK_EBOUNDS = -2,      /* document id, pool row or block id out of range        */
    KVLINK_ECAPACITY = -3,    /* a caller buffer is smaller than required                */
    KVLINK_EUNSUPPORTED = -4, /* shape outside what the kernels implement (see below)  */
    KVLINK_ECUDA = -5,        /* a CUDA runtime call or launch failed                     */
    KVLINK_EDEVICE = -6       /* a kernel recorded an error in the device status word    */
};

/* Supported shapes: head_dim 64 or 128; h_kv a power of two <= 16; h_q a multiple of
 * h_kv with G = h_q / h_kv a power of two <= 16; n_link >= 0; every query has at least
 * one fresh row; pool and cache block sizes 0 (contiguous) or a multiple of 8. */

/* Description of one batch of queries (all pointers host, read during the call). */
typedef struct {
    int32_t batch;             /* B queries                                               */
    int32_t n_link;            /* K link tokens appended after every document (Sec. 2.3)  */
    int32_t h_q, h_kv, head_dim;

    /* document cache pool (Sec. 2.1: caches precomputed per document) */
    int32_t pool_docs;         /* entries in the pool (documents and cached prefixes)     */
    const int32_t* pool_len;   /* [pool_docs] tokens per entry                            */
    const int64_t* pool_start; /* [pool_docs] contiguous: first row of the entry;
                                  paged: first slot of the entry in pool_block_table      */
    int64_t pool_rows;         /* contiguous: rows of the pool tensor;
                                  paged: physical blocks * pool_block_size                */
    int32_t pool_block_size;   /* 0 = contiguous pool [pool_rows][h_kv][D];
                                  else paged pool [blocks][pool_block_size][h_kv][D]      */
    const int32_t* pool_block_table; /* paged: physical block of each logical block      */
    int64_t pool_block_table_len;

    /* queries */
    const int32_t* prefix_doc; /* [B] pool entry placed at positions 0..P-1, or -1        */
    const int32_t* n_docs;     /* [B] retrieved documents per query                       */
    const int32_t* doc_ids;    /* [sum n_docs] pool entries, per query in sequence order  */
    const int32_t* q_len;      /* [B] question tokens per query                           */

    int32_t num_sms;           /* SMs the attention work is balanced over (0 = query the
                                  current device; 152 if none is visible)                 */
    int32_t layout;            /* physical order of the linked cache, KVLINK_LAYOUT_*     */
} kvlink_batch_desc_t;

/* Physical order of a query's rows in the linked cache.  Positions (and so RoPE and
 * the mask) are the same in both; only the cache row of a position differs.
 *   INTERLEAVED   row = global position: [prefix, doc_1, link_1, ..., doc_N, link_N,
 *                 question]
 *   LINKS_AT_END  the cached entries concatenated first, then the fresh rows in fresh
 *                 order: [prefix, doc_1, ..., doc_N, link_1, ..., link_N, question]
 *                 (Sec. 2.3, inference: the caches are loaded and concatenated and the
 *                 link tokens are appended at the end of the reordered sequence).  */
enum { KVLINK_LAYOUT_INTERLEAVED = 0, KVLINK_LAYOUT_LINKS_AT_END = 1 };

/* One contiguous run of the linked sequence (Sec. 2.3 layout). */
typedef struct {
    int32_t query;   /* b                                                            */
    int32_t kind;    /* KVLINK_SEG_*                                                 */
    int32_t src;     /* cached: pool entry id; fresh: first fresh row (global index) */
    int32_t len;     /* tokens                                                       */
    int64_t dst;     /* first row in the batch's contiguous linked cache
                        (= cu_ctx[b] + pos in the interleaved layout)                */
    int32_t pos;     /* global position of the first token within query b; for a
                        cached document this is also its RoPE delta (Sec. 2.2)       */
    int32_t table;   /* row of the RoPE delta table (cached documents), else -1      */
} kvlink_segment_t;

enum {
    KVLINK_SEG_PREFIX = 0,   /* cached, delta 0: copied                      */
    KVLINK_SEG_DOC = 1,      /* cached, rotated by delta = pos (Sec. 2.2)    */
    KVLINK_SEG_LINK = 2,     /* fresh link-token rows (Sec. 2.3)             */
    KVLINK_SEG_QUESTION = 3  /* fresh question rows                          */
};

/* Where the key and value of one position of the linked sequence come from, and the
 * linked-cache row they occupy.  The plan holds one per position, indexed by
 * cu_ctx[b] + position. */
typedef struct {
    int32_t kind;    /* KVLINK_SRC_POOL or KVLINK_SRC_FRESH                              */
    int32_t row;     /* POOL: row of the pool tensor (paged pool: physical block *
                        pool_block_size + offset); FRESH: row of k_new / v_new            */
    int32_t slot;    /* row of the batch's linked cache that holds this position         */
    int32_t table;   /* RoPE delta table row when the key is re-encoded (documents), else -1 */
} kvlink_source_t;

enum { KVLINK_SRC_POOL = 0, KVLINK_SRC_FRESH = 1 };

typedef struct kvlink_plan kvlink_plan_t; /* opaque */

typedef struct {
    int32_t batch, h_q, h_kv, head_dim, n_link;
    int32_t n_segments;       /* all segments, cached and fresh                       */
    int32_t n_rope_rows;      /* rows of the RoPE delta table (= cached documents)    */
    int32_t n_fresh;          /* fresh rows of the whole batch                        */
    int64_t ctx_rows;         /* rows of the contiguous linked cache (sum C_b)        */
    int64_t cached_tokens;    /* pool tokens gathered per layer (prefix + documents)  */
    int32_t n_copy_chunks;    /* re-encode work units                                 */
    int32_t n_attn_items;     /* attention work items (M-tile x KV range)             */
    int32_t n_attn_splits;    /* items that write a partial result                    */
    int32_t num_sms;
    size_t device_bytes;      /* size of the device buffer kvlink_plan_upload needs   */
    size_t workspace_bytes;   /* scratch of kvlink_suffix_attention / linked_prefill  */
    int64_t attn_pairs;       /* unmasked (fresh row, key) pairs, per KV head group   */
    int32_t n_attn_ctas;      /* CTAs of the persistent suffix attention (one per SM at
                                 most), each running its own list of work items       */
} kvlink_plan_info_t;

/* Build the host tables of a batch: the layout of every query (Sec. 2.3), the
 * segment table, the per-position sources, the re-encode work units and the attention
 * work items.  Validates every id and length against the pool.  Integer only; the
 * result is deterministic.  On success *out owns host memory until
 * kvlink_plan_destroy.  Errors: EINVAL, EBOUNDS, EUNSUPPORTED. */
int kvlink_plan_create(const kvlink_batch_desc_t* desc, kvlink_plan_t** out);
/* Rebuild an existing plan for another batch, as kvlink_plan_create would, reusing the
 * plan's host storage: a serving loop that keeps one plan per stream avoids allocating
 * (and first touching) its per-position tables for every batch.  The plan must be
 * uploaded again before use; device work already enqueued with the old tables is not
 * affected (kvlink_plan_upload orders its copy after it on the upload's stream).  On error
 * the plan holds no batch: rebuild it or destroy it.  Errors: as kvlink_plan_create. */
int kvlink_plan_rebuild(kvlink_plan_t* plan, const kvlink_batch_desc_t* desc);
/* Waits for the plan's last upload copy, then frees its host memory. */
void kvlink_plan_destroy(kvlink_plan_t* plan);
int kvlink_plan_get_info(const kvlink_plan_t* plan, kvlink_plan_info_t* info);

/* Host copies of the plan's tables.  seg: [cap] segments; cu_ctx: [B+1] first cache
 * row of every query (cu_ctx[B] = ctx_rows); cu_fresh: [B+1] first fresh row;
 * fresh_pos: [n_fresh] global position of every fresh row within its query.
 * Errors: EINVAL, ECAPACITY (cap smaller than the table). */
int kvlink_plan_get_segments(const kvlink_plan_t* plan, kvlink_segment_t* seg, int32_t cap);
int kvlink_plan_get_offsets(const kvlink_plan_t* plan, int64_t* cu_ctx, int32_t* cu_fresh);
int kvlink_plan_get_fresh_positions(const kvlink_plan_t* plan, int32_t* fresh_pos, int32_t cap);
/* src: [cap] sources, one per position of every query (ctx_rows of them), at
 * cu_ctx[b] + position.  With zero-copy values (d_cache_v NULL in the linked-prefill calls,
 * kvlink_suffix_attention_pool_values) this is where each position's value row lives.
 * Errors: EINVAL, ECAPACITY. */
int kvlink_plan_get_sources(const kvlink_plan_t* plan, kvlink_source_t* src, int64_t cap);

/* Bit set in a value-group entry whose rows are fresh rows (k_new / v_new), not pool rows. */
#define KVLINK_GROUP_FRESH (1 << 30)
/* The plan's groups of 8 cache rows, as the zero-copy value path and the one-kernel path
 * read them.  Query b owns entries cu_grp[b] .. cu_grp[b+1]), one per 8 cache rows
 * (ceil(rows of b / 8)); entry m covers its cache rows 8m .. 8m+7 and holds the first
 * source row when those 8 rows come from 8 consecutive rows of one tensor (a pool row, or
 * KVLINK_GROUP_FRESH | a fresh row): the kernels copy such a group as one tile.  Else -1
 * (a segment boundary inside, or the query's last, partial group): its rows are copied one
 * by one.  grp: [cap] host int32, cu_grp: [B+1] host int32, both owned by the caller.
 * Errors: EINVAL, ECAPACITY (cap below cu_grp[B]). */
int kvlink_plan_get_value_groups(const kvlink_plan_t* plan, int32_t* grp, int32_t* cu_grp, int64_t cap);

/* One work item of the persistent suffix attention: the fresh tokens [tok0, tok1) of query
 * `query` (query-relative) with the query heads of KV head `kv_head` (an M-tile), over the
 * entries [entry0, entry1) of the M-tile's key-tile list (entry e < a_tiles is key tile e of
 * the query's linked cache; entry a_tiles + i is key tile b_tile0 + i, the fresh rows at the
 * end of the links-at-end layout), run by CTA `cta`.  slot >= 0: the item is one piece of a
 * cut key range and writes a partial result to that workspace slot. */
typedef struct {
    int32_t query, kv_head, tok0, tok1;
    int32_t entry0, entry1, a_tiles, b_tile0;
    int32_t slot, cta;
} kvlink_attn_item_t;

/* items: [cap] work items in the order the CTAs run them (CTA 0's list first); one per
 * scheduled item (n_attn_items of them).  Plan introspection: the schedule is the plan's
 * business, this exposes it for checks and tuning.  Errors: EINVAL, ECAPACITY. */
int kvlink_plan_get_attention_items(const kvlink_plan_t* plan, kvlink_attn_item_t* items, int32_t cap);

/* Copy the plan's tables to the caller's device buffer d_buf (>= device_bytes,
 * 256-byte aligned) and build the RoPE delta table there: cos and sin of
 * delta_i * theta^(-2j/D) for every cached document i and j < D/2, with the angle
 * formed and reduced in float64 and stored as float32 (Sec. 2.2; done once per
 * batch, shared by all layers).  The plan records d_buf; later calls read it.
 * The buffer also holds the arrival counters of the attention's in-kernel merges, which the
 * upload zeroes and the attention kernels update (the buffer is not read-only on the device).
 * Asynchronous: the tables go through a pinned staging buffer owned by the plan, and the
 * call returns once the copy is enqueued (a later upload of the same plan first waits for
 * it).  d_buf must stay valid, and the plan alive, until the last call using them has
 * completed on the device.  Errors: EINVAL (not built), ECAPACITY, ECUDA. */
int kvlink_plan_upload(kvlink_plan_t* plan, double theta, void* d_buf, size_t bytes,
                       kvlink_stream_t stream);

/* Re-encode and concatenate one layer's cached K/V (Sec. 2.2, Sec. 2.1):
 *   for every cached segment (prefix, documents) and token t < len:
 *     cache_k[dst + t] = R_delta(pool_k[entry][t])   (bf16, round to nearest even)
 *     cache_v[dst + t] = pool_v[entry][t]            (bit copy)
 *   with delta = pos (0 for the prefix: bit copy).  R_delta pairs dimension j with
 *   j + D/2 (rotate-half) at angle delta * theta^(-2j/D).
 * The pool entries, their global offsets (pos) and theta come from the plan.
 * d_pool_k/d_pool_v: one layer of the pool (contiguous or paged as described);
 * d_cache_k/d_cache_v: one layer of the linked cache, [ctx_rows][h_kv][D].
 * d_cache_v may be NULL (zero-copy values): only the keys are re-encoded and written, and
 * d_pool_v is not read (may be NULL); the attention then reads the values where they are
 * (kvlink_suffix_attention_pool_values).
 * Fresh (link/question) slots are left untouched.  Errors: EINVAL, ECUDA. */
int kvlink_reencode_concat(const kvlink_plan_t* plan, const void* d_pool_k, const void* d_pool_v,
                           void* d_cache_k, void* d_cache_v, kvlink_stream_t stream);

/* Suffix attention of one layer (Sec. 2.3, "inference"):
 *   if d_k_new/d_v_new are non-NULL, fresh rows are first written to their slots:
 *     cache_k[slot(r)] = k_new[r] (same for v), slot(r) = cu_ctx[b] + fresh_pos[r] in
 *     the interleaved layout, the query's fresh region in the links-at-end layout;
 *   then for every fresh row r of query b (global position p_r), query head h,
 *   KV head g = h / G:
 *     out[r][h] = sum_j softmax_j(q[r][h] . cache_k[j][g] / sqrt(D)) cache_v[j][g]
 *   over the slots j <= p_r of query b: a link token sees every earlier position
 *   (all earlier documents and links, its own document, earlier links of its group),
 *   a question token is causal over everything before it (Sec. 2.3, Fig. 2).
 * d_q: [n_fresh][h_q][D]; d_k_new/d_v_new: [n_fresh][h_kv][D]; d_out: [n_fresh][h_q][D];
 * all bf16.  Scores and softmax in fp32, products of bf16 on the tensor cores.
 * d_workspace: >= workspace_bytes of scratch (may be NULL when that is 0).
 * The attention runs as one persistent kernel, one CTA per SM over its share of the work;
 * a KV range cut between CTAs is merged inside the kernel through arrival counters kept in
 * the plan's device buffer (zeroed by kvlink_plan_upload), so attention calls with one plan
 * must not overlap on the device, and after a wait that ran out (kvlink_device_status) the
 * plan must be uploaded again before its next use.
 * Errors: EINVAL, ECAPACITY, EUNSUPPORTED, ECUDA. */
int kvlink_suffix_attention(const kvlink_plan_t* plan, const void* d_q, const void* d_k_new,
                            const void* d_v_new, void* d_cache_k, void* d_cache_v, void* d_out,
                            void* d_workspace, size_t workspace_bytes, kvlink_stream_t stream);

/* kvlink_suffix_attention with zero-copy values (Sec. 2.3, "inference": the cached values
 * are concatenated unchanged, so they need not be copied): the same keys, mask and output,
 * with every value row read where it already is instead of from a linked cache:
 *   value of cache row j = pool_v[src(j)] for a prefix or document position,
 *                          v_new[src(j)]  for a fresh (link or question) row,
 * src the plan's source table (kvlink_plan_get_sources: kind KVLINK_SRC_POOL or
 * KVLINK_SRC_FRESH, row).  Runs of 8 cache rows whose sources are 8 consecutive rows of one
 * tensor are read as 8-row TMA boxes, the other rows one by one.
 * d_q, d_k_new, d_out: as for kvlink_suffix_attention; d_k_new may be NULL when the fresh keys
 * are already in d_cache_k (only keys are placed; d_cache_k holds keys only).
 * d_v_new: [n_fresh][h_kv][D], required.  d_pool_v: one layer of the pool's values (the
 * tensor kvlink_reencode_concat reads, contiguous or paged), required.
 * The output equals kvlink_suffix_attention's bit for bit on the same keys and values (same
 * tiles, same order of operations).  Errors: EINVAL, ECAPACITY, EUNSUPPORTED, ECUDA. */
int kvlink_suffix_attention_pool_values(const kvlink_plan_t* plan, const void* d_q, const void* d_k_new,
                                        const void* d_v_new, const void* d_pool_v, void* d_cache_k,
                                        void* d_out, void* d_workspace, size_t workspace_bytes,
                                        kvlink_stream_t stream);

/* The same computation as kvlink_suffix_attention on the CUDA cores: one CTA per
 * (fresh row, KV head) streams the row's visible keys with an online softmax in
 * fp32; no tensor cores, no workspace.  A second, independent GPU implementation
 * for cross-checking and for debugging.  Errors: EINVAL, ECUDA. */
int kvlink_suffix_attention_simt(const kvlink_plan_t* plan, const void* d_q, const void* d_k_new,
                                 const void* d_v_new, void* d_cache_k, void* d_cache_v, void* d_out,
                                 kvlink_stream_t stream);

/* RoPE of the fresh rows at their global positions, in place (Sec. 2.2: the token at
 * position i carries R_i; Sec. 2.3: link and question tokens are encoded at their
 * positions in the linked sequence):
 *   q[r][h]     = R_{p_r}(q[r][h])      for every query head h,
 *   k_new[r][g] = R_{p_r}(k_new[r][g])  for every KV head g,
 * p_r the global position of fresh row r, theta the plan's (kvlink_plan_upload), pairs
 * (j, j + D/2).  For producers that project fresh rows without RoPE:
 * kvlink_suffix_attention and kvlink_linked_prefill take q and k_new already rotated.
 * d_q: [n_fresh][h_q][D], d_k_new: [n_fresh][h_kv][D], bf16; each result within one bf16
 * ulp of the fp64 rotation.  Errors: EINVAL, ECUDA. */
int kvlink_rope_fresh(const kvlink_plan_t* plan, void* d_q, void* d_k_new, kvlink_stream_t stream);

/* One layer of the linked prefill: kvlink_reencode_concat with the fresh-row
 * placement fused into the same launch, then the suffix attention.  Same arguments
 * and errors as the two calls it chains.  d_cache_v NULL selects zero-copy values: the
 * re-encode writes keys only and the attention is kvlink_suffix_attention_pool_values
 * (same output bits). */
int kvlink_linked_prefill(const kvlink_plan_t* plan, const void* d_pool_k, const void* d_pool_v,
                          const void* d_q, const void* d_k_new, const void* d_v_new,
                          void* d_cache_k, void* d_cache_v, void* d_out,
                          void* d_workspace, size_t workspace_bytes, kvlink_stream_t stream);

/* One layer of the linked prefill in a single attention kernel (Sec. 2.2 + Sec. 2.3):
 * the same result as kvlink_linked_prefill, but the attention reads every key and
 * value where it already is (pool rows for the prefix and documents, k_new / v_new
 * for the fresh rows), rotates document keys by their delta in shared memory on the
 * way to the tensor cores, and writes the linked cache as a side output, so the cache
 * is written once and never read back.
 *   - d_cache_k / d_cache_v receive the linked cache exactly as kvlink_linked_prefill
 *     writes it (same bits), in the plan's layout.  Either may be NULL: that half is
 *     then not written.  With d_cache_v NULL the values stay in the pool and in v_new
 *     (zero-copy values: kvlink_plan_get_sources says where each position's value row
 *     is), halving the cache bytes written.
 *   - d_q, d_k_new, d_v_new: as for kvlink_suffix_attention (q and k_new rotated at
 *     their positions).  d_workspace: >= workspace_bytes.
 * The output equals kvlink_linked_prefill's bit for bit (same tiles, same order of
 * operations).  Errors: EINVAL, ECAPACITY, EUNSUPPORTED, ECUDA. */
int kvlink_linked_prefill_fused(const kvlink_plan_t* plan, const void* d_pool_k, const void* d_pool_v,
                                const void* d_q, const void* d_k_new, const void* d_v_new,
                                void* d_cache_k, void* d_cache_v, void* d_out,
                                void* d_workspace, size_t workspace_bytes, kvlink_stream_t stream);

/* Re-encode + concat (Sec. 2.2, Sec. 2.1) of the document caches of n_layers layers in
 * one launch: the same result as kvlink_reencode_concat(plan, pool_k[l], pool_v[l],
 * cache_k[l], cache_v[l]) for every layer l, bit for bit (d_cache_v itself NULL: keys only
 * in every layer, d_pool_v not read).  The precomputed document
 * caches do not depend on the forward pass of the fresh rows, so a prefill can rotate
 * every layer's caches before its first layer runs, in one launch instead of one per
 * layer (the fresh rows are then placed per layer by kvlink_suffix_attention with
 * k_new / v_new).  Each argument is a HOST array
 * of n_layers device pointers (each 16-byte aligned; per layer, the shapes of
 * kvlink_reencode_concat).  Errors: EINVAL (a NULL or misaligned pointer, n_layers <= 0),
 * the plan errors of kvlink_reencode_concat, ECUDA. */
int kvlink_reencode_concat_layers(const kvlink_plan_t* plan, int32_t n_layers, const void* const* d_pool_k,
                                  const void* const* d_pool_v, void* const* d_cache_k, void* const* d_cache_v,
                                  kvlink_stream_t stream);

/* The linked prefill of n_layers layers (the attention side of one whole prefill) in
 * one call, with the same results, bit for bit, as kvlink_linked_prefill(plan,
 * pool_k[l], pool_v[l], q[l], k_new[l], v_new[l], cache_k[l], cache_v[l], out[l], ...)
 * for every layer l in order, which is what it enqueues.  Each argument is a HOST array
 * of n_layers device pointers; d_cache_v itself may be NULL (zero-copy values in every layer).  One workspace serves all layers (they run in stream
 * order).  Every pointer is checked before the first launch.  Errors: as
 * kvlink_linked_prefill. */
int kvlink_linked_prefill_layers(const kvlink_plan_t* plan, int32_t n_layers, const void* const* d_pool_k,
                                 const void* const* d_pool_v, const void* const* d_q,
                                 const void* const* d_k_new, const void* const* d_v_new, void* const* d_cache_k,
                                 void* const* d_cache_v, void* const* d_out, void* d_workspace,
                                 size_t workspace_bytes, kvlink_stream_t stream);

/* The same results as kvlink_linked_prefill_layers, bit for bit, with the re-encode on a
 * second stream.  reencode_stream first waits for the work already enqueued on `stream`,
 * then re-encodes every layer's document caches (kvlink_reencode_concat) back to back;
 * layer l's fresh-row placement and suffix attention run on `stream` once layer l's
 * caches are in place.  The document caches do not depend on the forward pass, so the
 * re-encode of later layers fills the SMs that the attention of earlier layers leaves
 * idle (the ends of its grid, the gaps between launches).  When the call returns,
 * `stream` is ordered after all of its work.  The plan keeps the events it uses: calls
 * with one plan must not run concurrently.  d_cache_v NULL: zero-copy values in every layer,
 * as for kvlink_linked_prefill_layers.  The call may be captured in a CUDA graph on `stream`
 * (the second stream joins the capture through the plan's events) and the graph replayed with
 * the same results.  Errors: as kvlink_linked_prefill_layers;
 * EINVAL also when the two streams are the same. */
int kvlink_linked_prefill_layers_overlapped(kvlink_plan_t* plan, int32_t n_layers, const void* const* d_pool_k,
                                            const void* const* d_pool_v, const void* const* d_q,
                                            const void* const* d_k_new, const void* const* d_v_new,
                                            void* const* d_cache_k, void* const* d_cache_v, void* const* d_out,
                                            void* d_workspace, size_t workspace_bytes, kvlink_stream_t stream,
                                            kvlink_stream_t reencode_stream);

/* The linked prefill of n_layers layers end to end from host memory, as a serving step
 * runs it: the same results as kvlink_linked_prefill_layers_overlapped, bit for bit, with
 * every layer's fresh rows brought in from, and its output taken back to, host memory.
 *   h_q[l], h_k_new[l], h_v_new[l]: host rows of layer l, [n_fresh][h_q or h_kv][D] bf16,
 *     copied to d_q[l], d_k_new[l], d_v_new[l] on copy_in_stream (pinned memory makes the
 *     copies asynchronous);
 *   the document caches of every layer are re-encoded on reencode_stream, which first
 *     waits for the work already on `stream` (the plan upload);
 *   layer l's fresh-row placement and suffix attention run on `stream` once its inputs
 *     and caches are in place;
 *   d_out[l] is copied to h_out[l] ([n_fresh][h_q][D]) on copy_out_stream.
 * Returns once everything is enqueued: the outputs are on the host when copy_out_stream
 * has completed the call's work.  Successive calls with one plan (also across
 * kvlink_plan_rebuild) chain through events the plan keeps for this function alone: a
 * layer's device inputs and caches are rewritten only after the previous call's kernels of
 * that layer have read them, and its device output only after the previous call's copy of
 * it to the host, so a caller may prepare and enqueue the next batch while one runs.  A
 * call with another layer count than the previous one is ordered after the whole previous
 * call instead (its copies in and its re-encode start after the previous call's last
 * output copy).  The chain links calls
 * of this function only: other work that touches the same buffers in between (another
 * entry point, the caller's kernels) must be ordered by the caller, e.g. by making
 * copy_in_stream wait for it.  The four streams must be distinct.  d_cache_v NULL: zero-copy
 * values in every layer, as for kvlink_linked_prefill_layers.  Errors: as
 * kvlink_linked_prefill_layers; EINVAL also for a NULL host pointer or repeated
 * streams. */
int kvlink_linked_prefill_layers_host(kvlink_plan_t* plan, int32_t n_layers, const void* const* d_pool_k,
                                      const void* const* d_pool_v, const void* const* h_q,
                                      const void* const* h_k_new, const void* const* h_v_new, void* const* d_q,
                                      void* const* d_k_new, void* const* d_v_new, void* const* d_cache_k,
                                      void* const* d_cache_v, void* const* d_out, void* const* h_out,
                                      void* d_workspace, size_t workspace_bytes, kvlink_stream_t stream,
                                      kvlink_stream_t reencode_stream, kvlink_stream_t copy_in_stream,
                                      kvlink_stream_t copy_out_stream);

/* Re-encode + concat of one layer (as kvlink_reencode_concat, the same bits) with that
 * layer's document cache pool in host memory (Sec. 3.3: the precomputed caches are kept in
 * CPU memory and loaded for every request).  h_pool_k / h_pool_v: page-locked host memory
 * (cudaHostAlloc, or cudaHostRegister'ed) holding the pool in the plan's layout; the kernel
 * reads the rows it needs through the device's mapping of that memory (NVLink-C2C on a
 * Grace system), rotates the document keys and writes the linked cache in device memory, so
 * the rows cross the host link once and are never staged.  The host memory must stay valid
 * and unchanged until the work has completed on the device.  Errors: EINVAL (also for
 * pageable or device memory), ECUDA. */
int kvlink_reencode_concat_host_pool(const kvlink_plan_t* plan, const void* h_pool_k, const void* h_pool_v,
                                     void* d_cache_k, void* d_cache_v, kvlink_stream_t stream);

/* The linked prefill of n_layers layers with every layer's document cache pool in host
 * memory: the same results as kvlink_linked_prefill_layers_overlapped, bit for bit, with
 * kvlink_reencode_concat_host_pool in place of the device-pool re-encode.  load_stream
 * first waits for the work already on `stream`, then loads and re-encodes every layer's
 * document caches from host memory back to back; layer l's fresh-row placement and suffix
 * attention run on `stream` once layer l's caches are in place, so the loading of later
 * layers overlaps the attention of earlier ones.  h_pool_k / h_pool_v: HOST arrays of
 * n_layers page-locked host pointers; the other arrays as for
 * kvlink_linked_prefill_layers_overlapped.  When the call returns, `stream` is ordered after
 * all of its work.  The plan keeps the events it uses: calls with one plan must not run
 * concurrently.  The values are loaded into d_cache_v (required here: a host pool's values
 * are not read by the attention in place).  Errors: as
 * kvlink_linked_prefill_layers_overlapped; EINVAL also for a pool pointer that is not
 * page-locked host memory, or when the two streams are the same. */
int kvlink_linked_prefill_layers_host_pool(kvlink_plan_t* plan, int32_t n_layers, const void* const* h_pool_k,
                                           const void* const* h_pool_v, const void* const* d_q,
                                           const void* const* d_k_new, const void* const* d_v_new,
                                           void* const* d_cache_k, void* const* d_cache_v, void* const* d_out,
                                           void* d_workspace, size_t workspace_bytes, kvlink_stream_t stream,
                                           kvlink_stream_t load_stream);

/* Allocation-free variant of kvlink_suffix_attention.  The paper has no counterpart:
 * this entry point serves callers that may not allocate device memory at all, such as
 * a serving loop whose memory budget is fixed at start-up (cudaMalloc can synchronise
 * the device and fragments a pre-carved pool) or code that enqueues work where
 * allocation is not permitted.  Same arguments and result as kvlink_suffix_attention,
 * minus the workspace: the split-KV scratch is a static device array of
 * KVLINK_NOALLOC_MAX_WORKSPACE_BYTES inside this library, which every GPU that loads
 * the library holds until the process exits.  The call allocates nothing.
 *   - Plans whose workspace_bytes exceed KVLINK_NOALLOC_MAX_WORKSPACE_BYTES are
 *     rejected with KVLINK_ECAPACITY before anything is launched.
 *   - The first call on a device looks up the array's device address (once per
 *     device, with that device current); make that first call before any stream
 *     capture.  The address is kept for the life of the process: resetting the device
 *     (cudaDeviceReset) after that first call is not supported.
 *   - CUDA failures are recorded for kvlink_last_cuda_error() like those of every
 *     other entry point.
 *   - All calls share the array and it keeps the last call's contents; nothing in it
 *     needs to start at zero.  Calls whose work overlaps on the GPU race on it.
 * Errors: EINVAL, ECAPACITY, EUNSUPPORTED, ECUDA. */
#define KVLINK_NOALLOC_MAX_WORKSPACE_BYTES (8u << 20)
int kvlink_suffix_attention_noalloc(const kvlink_plan_t* plan, const void* d_q, const void* d_k_new,
                                    const void* d_v_new, void* d_cache_k, void* d_cache_v, void* d_out,
                                    kvlink_stream_t stream);

/* Device status word: 0 when no kernel reported an error since the last clear, else the
 * first code recorded: KVLINK_STATUS_WAIT_TIMEOUT (an attention pipeline wait ran out)
 * or KVLINK_STATUS_COPY_TIMEOUT (a re-encode pipeline wait ran out).  While it is set,
 * later launches skip their work (outputs undefined) instead of waiting out their
 * bounds; kvlink_clear_device_status() re-arms them.  Reading synchronises with the
 * current device.  Errors: ECUDA. */
#define KVLINK_STATUS_WAIT_TIMEOUT 0x41
#define KVLINK_STATUS_COPY_TIMEOUT 0x21
/* Only in the build with KVLINK_DEBUG_CHECKS (libkvlink_debug.so): a work item or merge
 * group of the suffix attention (0x42), or a re-encode unit or fresh-row destination (0x22),
 * lies outside the plan's tables; the CTA that found it did nothing else. */
#define KVLINK_STATUS_BAD_INDEX_ATTN 0x42
#define KVLINK_STATUS_BAD_INDEX_COPY 0x22
int kvlink_device_status(int32_t* status);
int kvlink_clear_device_status(void);

/* Failure-path self-test: one GPU thread waits, through the same bounded mbarrier wait
 * the attention kernels use, on a barrier that nothing arrives at, with a limit of
 * limit_ms (1..2000).  The wait runs out and records KVLINK_STATUS_WAIT_TIMEOUT in the
 * status word, as a stalled pipeline would; nothing traps and the context stays usable.
 * Errors: EINVAL (limit out of range), ECUDA. */
int kvlink_selftest_wait_timeout(uint32_t limit_ms, kvlink_stream_t stream);

const char* kvlink_strerror(int code);
/* Text of the last CUDA error seen by this thread (empty if none). */
const char* kvlink_last_cuda_error(void);
int kvlink_version(void); /* major*10000 + minor*100 + patch */

#ifdef __cplusplus
}
#endif
#endif /* KVLINK_H */
