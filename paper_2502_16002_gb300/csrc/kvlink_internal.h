// Internal types shared by the host plan builder and the CUDA kernels.
#pragma once

#include <stdint.h>
#include <cuda_runtime.h>
#include <vector_types.h>

#include <atomic>
#include <string>
#include <utility>
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
// over a range of the query's key tiles (kAttnBN cache rows each, in cache-row order).
// The tiles an M-tile needs form at most two runs: rows [0, a) holding the cached
// entries (every layout), and, in the links-at-end layout, the fresh rows at the end.
// Tile v of that list is v itself for v < a_tiles, else b_tile0 + (v - a_tiles); the
// item covers list entries [kv_tile0, kv_tile1).
struct AttnItem {
    int32_t query;
    int32_t kv_head;
    int32_t tok0, tok1;          // fresh tokens [tok0, tok1) of the query (query-relative)
    int32_t kv_tile0, kv_tile1;  // entries of the tile list
    int32_t slot;                // partial-result slot, or -1: write the output directly
    int32_t min_vis;             // cache rows below min_vis are visible to every row
    int32_t owner;               // 1: the item's key range is written to the linked cache
                                 // by the one-kernel path (the last M-tile of each (query,
                                 // KV head) covers every cache row exactly once)
    int32_t a_tiles;             // tiles of the first run (rows from 0)
    int32_t b_tile0;             // first tile of the second run
};
static_assert(sizeof(AttnItem) == 44, "AttnItem layout");

// Key tile (kAttnBN rows from the query's first cache row) of entry v of an item's list.
__host__ __device__ inline int32_t item_tile(const AttnItem& it, int32_t v) {
    return v < it.a_tiles ? v : it.b_tile0 + (v - it.a_tiles);
}

// fresh_row0 of a query without a fresh region at the end (interleaved layout)
constexpr int32_t kNoFreshRegion = 0x3fffffff;

// Runs `fn` (a kernel attribute setter) once per device: such attributes belong to the
// device's context, so a process that launches on several devices needs the call on each.
// Thread-safe; concurrent first calls may both run `fn`, which is idempotent.
template <typename Fn>
inline cudaError_t once_per_device(std::atomic<uint64_t>& done, Fn&& fn) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const uint64_t bit = dev >= 0 && dev < 64 ? (uint64_t)1 << dev : 0;
    if (bit && (done.load(std::memory_order_acquire) & bit)) return cudaSuccess;
    e = fn();
    if (e == cudaSuccess && bit) done.fetch_or(bit, std::memory_order_release);
    return e;
}

// Bounds of the re-encode and placement kernels' tables (device-side checks).
struct CopyBounds {
    int64_t ctx_rows;    // rows of the linked cache
    int64_t pool_rows;   // rows of the pool tensor
    int32_t n_fresh;     // fresh rows
    int32_t n_rope_rows; // rows of the RoPE delta table
};

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
    const CopyChunk* chunks_sorted;  // the cached chunks by source row (all-layer re-encode)
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
    const kvlink_source_t* src_row;  // [ctx_rows] the same records by linked-cache row
    // Visibility of fresh row r (query b): cache rows [0, fresh_vis[r]) and, when the query
    // keeps its fresh rows at the end, [fresh_row0[b], fresh_row0[b] + f + 1) with f the row's
    // index among the query's fresh rows (interleaved: fresh_row0 = kNoFreshRegion).
    const int32_t* fresh_vis;    // [n_fresh]
    const int32_t* fresh_row0;   // [B], query-relative
    const int32_t* fresh_dst;    // [n_fresh] batch cache row of every fresh row
    // sizes the tables index into (checked on the device by the KVLINK_DEBUG_CHECKS build)
    int32_t batch, h_kv, n_fresh, n_slots, n_rope_rows, n_items;
    int64_t ctx_rows, pool_rows;
    // Groups of 8 cache rows (8m .. 8m+7 of a query), at cu_grp[b] + m: the first source
    // row when the group's 8 rows are consecutive in one tensor (one 8-row TMA copy), else
    // -1 (rows copied one by one; also the query's last, partial group).
    const int32_t* cu_grp;       // [B+1]
    const int32_t* grp_src;      // pool row, or kGrpFresh | fresh row
    // Persistent attention: CTA c runs items sched[cu_sched[c] .. cu_sched[c+1]) in order.
    const int32_t* sched;        // [n_items] item indices
    const int32_t* cu_sched;     // [n_ctas + 1]
    // Split KV ranges merged inside the persistent attention: the merge group of every
    // partial slot, and one arrival counter per group.  A counter only ever grows (each
    // launch adds its group's n_split), so the piece that brings it to a multiple of n_split
    // is the last of its launch and merges; kvlink_plan_upload zeroes the counters.
    const int32_t* slot_group;   // [n_slots]
    unsigned long long* merge_count;   // [n_merges], in the plan buffer (written by the kernel)
    int32_t n_merges;
};
// Where the suffix attention reads the values.  cache_v non-NULL: the linked cache's value
// rows, [ctx_rows][h_kv][D].  cache_v NULL (zero-copy values): every value row where it
// already is, pool_v [pool_rows][h_kv][D] for the prefix and document positions and v_new
// [n_fresh][h_kv][D] for the fresh rows, found through the plan's source and group tables.
struct ValueSource {
    const void* cache_v;
    const void* pool_v;
    const void* v_new;
};
constexpr int32_t kGrpFresh = 1 << 30;
constexpr int32_t kGrpRowMask = kGrpFresh - 1;

}  // namespace kvlink

namespace kvlink {
// Pinned host buffer of the plan upload, reused by later uploads.  `done` is recorded on
// the upload's stream after its copy; the buffer is rewritten only once it has completed.
struct PinnedStaging {
    char* ptr = nullptr;
    size_t bytes = 0;
    cudaEvent_t done = nullptr;
    PinnedStaging() = default;
    PinnedStaging(const PinnedStaging&) = delete;
    PinnedStaging& operator=(const PinnedStaging&) = delete;
    PinnedStaging(PinnedStaging&& o) noexcept { swap(o); }
    PinnedStaging& operator=(PinnedStaging&& o) noexcept {
        swap(o);
        return *this;
    }
    ~PinnedStaging();
    void swap(PinnedStaging& o) noexcept {
        std::swap(ptr, o.ptr);
        std::swap(bytes, o.bytes);
        std::swap(done, o.done);
    }
};
// Events reused by the calls of one plan (created on first use, destroyed with the plan).
struct EventPool {
    std::vector<cudaEvent_t> ev;
    EventPool() = default;
    EventPool(const EventPool&) = delete;
    EventPool& operator=(const EventPool&) = delete;
    EventPool(EventPool&& o) noexcept { ev.swap(o.ev); }
    EventPool& operator=(EventPool&& o) noexcept {
        ev.swap(o.ev);
        return *this;
    }
    ~EventPool();
};
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
    std::vector<kvlink::CopyChunk> chunks_sorted;   // the cached chunks by source row
    int32_t n_rope_rows = 0;
    std::vector<int64_t> cu_ctx;
    std::vector<int32_t> cu_fresh;
    std::vector<int32_t> fresh_pos;
    std::vector<int32_t> fresh_query;
    std::vector<kvlink_source_t> src, src_row;
    std::vector<int32_t> fresh_vis, fresh_row0, fresh_dst;
    std::vector<int32_t> cu_grp, grp_src;
    std::vector<kvlink::AttnItem> items;
    std::vector<kvlink::MergeGroup> merges;
    std::vector<int32_t> sched, cu_sched;   // the persistent attention's item list per CTA
    std::vector<int32_t> slot_group;        // merge group of every partial slot
    int32_t n_slots = 0;
    int64_t cached_tokens = 0;
    int64_t attn_pairs = 0;

    // layout of the device buffer (byte offsets) and its total size
    size_t off_chunks_sorted = 0;
    size_t off_seg = 0, off_chunks = 0, off_rope = 0, off_pool_start = 0, off_pool_bt = 0,
           off_cu_ctx = 0, off_cu_fresh = 0, off_fresh_pos = 0, off_fresh_query = 0,
           off_items = 0, off_merges = 0, off_src = 0, off_cu_grp = 0, off_grp_src = 0, off_src_row = 0,
           off_fresh_vis = 0, off_fresh_row0 = 0, off_fresh_dst = 0, off_sched = 0, off_cu_sched = 0,
           off_slot_group = 0, off_merge_count = 0,
           device_bytes = 0;
    size_t workspace_bytes = 0;

    bool built = false;                 // holds a batch (a failed rebuild clears it)
    kvlink::PinnedStaging staging;
    kvlink::EventPool events;           // per-layer events of the overlapped all-layers calls
    kvlink::EventPool host_events;      // events of the host-path calls (kept apart from the above)
    int32_t host_chain_layers = 0;      // layers of the last host-path call (its events chain the next)

    // set by kvlink_plan_upload
    bool uploaded = false;
    double theta = 0.0;
    void* d_buf = nullptr;
    kvlink::DevicePlan dev{};
};

namespace kvlink {
// Record a failed CUDA call for kvlink_last_cuda_error() and return KVLINK_ECUDA
// (kvlink_api.cu); record_launch_error checks cudaGetLastError() the same way and returns
// KVLINK_OK when there is nothing to record.
int record_cuda_error(cudaError_t e, const char* where);
int record_launch_error(const char* where);
// Host plan builder (kvlink_plan.cpp).  num_sms must be resolved (> 0).
int build_plan(const kvlink_batch_desc_t* desc, int32_t num_sms, kvlink_plan* plan,
               std::string* why);
}  // namespace kvlink
