// Internal types shared by the host plan builder and the CUDA kernels.
#pragma once

#include <stdint.h>
#include <vector_types.h>

#include <string>
#include <vector>

#include "kvlink.h"

namespace kvlink {

constexpr int kAttnBM = 128;     // (fresh token, query head) rows per attention tile
constexpr int kAttnBN = 128;     // keys per KV tile
constexpr int kCopyStageBytes = 32768;   // K (or V) bytes of one re-encode work unit
constexpr int kCopyMaxTokens = 128;

// Tokens per re-encode work unit for a given K row size (H_kv * D * 2 bytes).
inline int copy_chunk_tokens(int row_bytes) {
    int t = kCopyStageBytes / row_bytes;
    return t < 8 ? 8 : (t > kCopyMaxTokens ? kCopyMaxTokens : t);
}

// One re-encode work unit: n consecutive tokens whose K/V rows are contiguous both in
// the source (pool or fresh rows) and in the linked cache.  Resolved on the host.
struct CopyChunk {
    int64_t src_row;   // first source row (pool row, or fresh row for LINK/QUESTION)
    int64_t dst_row;   // first linked-cache row
    int32_t n;         // tokens
    int32_t kind;      // KVLINK_SEG_*
    int32_t table;     // RoPE delta table row (documents), else -1
    int32_t seg;       // segment index
};
static_assert(sizeof(CopyChunk) == 32, "CopyChunk layout");

// One attention work item: an M-tile of (token, head) rows of one query and KV head,
// over KV tiles [kv_tile0, kv_tile1).
struct AttnItem {
    int32_t query;
    int32_t kv_head;
    int32_t tok0, tok1;          // fresh tokens [tok0, tok1) of the query (query-relative)
    int32_t kv_tile0, kv_tile1;  // key tiles of kAttnBN keys
    int32_t slot;                // partial-result slot, or -1: write the output directly
    int32_t min_pos;             // smallest position of the tile's rows: keys <= min_pos
                                 // are visible to every row of the tile
    int32_t owner;               // 1: the item's key range is written to the linked cache
                                 // by the fused kernel (the last M-tile of each (query,
                                 // KV head) covers every position exactly once)
};
static_assert(sizeof(AttnItem) == 36, "AttnItem layout");

// Rows of one (query, KV head, M-tile) whose KV range was split over several items.
struct MergeGroup {
    int32_t query;
    int32_t kv_head;
    int32_t tok0, tok1;
    int32_t slot0;               // first partial slot; the group's slots are consecutive
    int32_t n_split;
    int32_t pad0, pad1;
};
static_assert(sizeof(MergeGroup) == 32, "MergeGroup layout");

// Device view of an uploaded plan (pointers into the caller's device buffer).
struct DevicePlan {
    const kvlink_segment_t* seg;
    const CopyChunk* chunks;     // cached-segment chunks first, then fresh-segment chunks
    const float4* rope;          // [n_rope_rows][D/2] (cos hi, cos lo, sin hi, sin lo)
    const int64_t* pool_start;   // [pool_docs]
    const int32_t* pool_block_table;
    const int64_t* cu_ctx;       // [B+1]
    const int32_t* cu_fresh;     // [B+1]
    const int32_t* fresh_pos;    // [n_fresh]
    const int32_t* fresh_query;  // [n_fresh]
    const AttnItem* items;       // [n_items]
    const MergeGroup* merges;    // [n_merges]
    const kvlink_source_t* src;  // [ctx_rows] by cu_ctx[b] + position
    // Groups of 8 positions (8m .. 8m+7 of a query), at cu_grp[b] + m: the first row of
    // the group when its 8 rows are consecutive in one tensor (one 8-row TMA copy), else
    // -1 (rows copied one by one; also the query's last, partial group).
    const int32_t* cu_grp;       // [B+1]
    const int32_t* grp_src;      // pool row, or kGrpFresh | fresh row
    const int32_t* grp_slot;     // linked-cache row
};
constexpr int32_t kGrpFresh = 1 << 30;
constexpr int32_t kGrpRowMask = kGrpFresh - 1;

}  // namespace kvlink

struct kvlink_plan {
    // scalars of the description
    int32_t batch = 0, n_link = 0, h_q = 0, h_kv = 0, head_dim = 0;
    int32_t pool_docs = 0, pool_block_size = 0;
    int64_t pool_rows = 0;
    int32_t num_sms = 0;
    int32_t layout = KVLINK_LAYOUT_INTERLEAVED;

    // host tables
    std::vector<int64_t> pool_start;
    std::vector<int32_t> pool_len;
    std::vector<int32_t> pool_block_table;
    std::vector<kvlink_segment_t> seg;
    std::vector<kvlink::CopyChunk> chunks;
    int32_t n_chunks_cached = 0;
    int32_t n_rope_rows = 0;
    std::vector<int64_t> cu_ctx;
    std::vector<int32_t> cu_fresh;
    std::vector<int32_t> fresh_pos;
    std::vector<int32_t> fresh_query;
    std::vector<kvlink_source_t> src;
    std::vector<int32_t> cu_grp, grp_src, grp_slot;
    std::vector<kvlink::AttnItem> items;
    std::vector<kvlink::MergeGroup> merges;
    int32_t n_slots = 0;
    int64_t cached_tokens = 0;
    int64_t attn_pairs = 0;

    // layout of the device buffer (byte offsets) and its total size
    size_t off_seg = 0, off_chunks = 0, off_rope = 0, off_pool_start = 0, off_pool_bt = 0,
           off_cu_ctx = 0, off_cu_fresh = 0, off_fresh_pos = 0, off_fresh_query = 0,
           off_items = 0, off_merges = 0, off_src = 0, off_cu_grp = 0, off_grp_src = 0, off_grp_slot = 0,
           device_bytes = 0;
    size_t workspace_bytes = 0;

    // set by kvlink_plan_upload
    bool uploaded = false;
    double theta = 0.0;
    void* d_buf = nullptr;
    kvlink::DevicePlan dev{};
};

namespace kvlink {
// Host plan builder (kvlink_plan.cpp).  num_sms must be resolved (> 0).
int build_plan(const kvlink_batch_desc_t* desc, int32_t num_sms, kvlink_plan* plan,
               std::string* why);
}  // namespace kvlink
