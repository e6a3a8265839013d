// C ABI entry points (declared in include/kvlink.h): argument validation on the
// host, plan upload, and the launches of the linked-prefill kernels.
#include <cuda_runtime.h>

#include <algorithm>
#include <cstring>
#include <new>
#include <string>
#include <vector>

#include "kvlink_internal.h"

namespace kvlink {
void launch_rope_table(const kvlink_segment_t* d_seg, int n_seg, float4* d_rope, int head_dim,
                       double theta, cudaStream_t stream);
void launch_reencode(const DevicePlan& P, int chunk_base, int n_chunks, int head_dim, int h_kv, int num_sms,
                     const void* pool_k, const void* pool_v, const void* k_new, const void* v_new, void* cache_k,
                     void* cache_v, cudaStream_t stream);
void launch_reencode_layers(const DevicePlan& P, int n_chunks, int head_dim, int h_kv, int num_sms, int n_layers,
                            const void* const* pool_k, const void* const* pool_v, void* const* cache_k,
                            void* const* cache_v, cudaStream_t stream);
void launch_reencode_host(const DevicePlan& P, int n_chunks, int head_dim, int h_kv, int num_sms,
                          const void* pool_k, const void* pool_v, void* cache_k, void* cache_v, cudaStream_t stream);
void launch_place_fresh(const int32_t* d_fresh_dst, int n_fresh, int64_t ctx_rows, int row_bytes,
                        const void* k_new, const void* v_new, void* cache_k, void* cache_v, cudaStream_t stream);
int read_copy_status(int32_t* status);
void launch_rope_fresh(const int32_t* d_fresh_pos, int n_fresh, int head_dim, double theta, void* q, int h_q,
                       void* k, int h_kv, cudaStream_t stream);
int clear_copy_status();
void launch_attention_simt(const DevicePlan& P, int n_fresh, int head_dim, int h_q, int h_kv,
                           const void* q, const void* cache_k, const void* cache_v, void* out,
                           cudaStream_t stream);
int launch_attention_tc(const DevicePlan& P, int n_items, int n_ctas, int n_merges, int n_fresh, int64_t ctx_rows,
                        int head_dim, int h_q, int h_kv, const void* q, const void* cache_k, const ValueSource& vs,
                        void* out, void* ws, cudaStream_t stream, cudaError_t* err);
int read_attention_status(int32_t* status);
int clear_attention_status();
int launch_attention_fused(const DevicePlan& P, int n_items, int n_merges, int n_fresh, int64_t pool_rows,
                           int head_dim, int h_q, int h_kv, const void* q, const void* pool_k, const void* pool_v,
                           const void* k_new, const void* v_new, void* cache_k, void* cache_v, void* out, void* ws,
                           cudaStream_t stream, cudaError_t* err);
int read_fused_status(int32_t* status);
int clear_fused_status();
int launch_wait_selftest(uint32_t limit_ms, cudaStream_t stream);
}  // namespace kvlink

using namespace kvlink;

namespace {

thread_local std::string g_last_cuda_error;

int cuda_fail(cudaError_t e, const char* where) {
    g_last_cuda_error = std::string(where) + ": " + cudaGetErrorString(e);
    return KVLINK_ECUDA;
}

int check_launch(const char* where) {
    const cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? KVLINK_OK : cuda_fail(e, where);
}

}  // namespace

namespace kvlink {
// The recorder above, for entry points defined in other translation units.
int record_cuda_error(cudaError_t e, const char* where) { return cuda_fail(e, where); }
int record_launch_error(const char* where) { return check_launch(where); }
}  // namespace kvlink

namespace {

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

int resolve_num_sms(int32_t requested) {
    if (requested > 0) return requested;
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) == cudaSuccess &&
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess && n > 0)
        return n;
    cudaGetLastError();  // no device visible: clear the sticky error, use GB300's count
    return 152;
}

int check_plan(const kvlink_plan_t* p) {
    if (!p) return KVLINK_EINVAL;
    if (!p->uploaded) return KVLINK_EINVAL;
    return KVLINK_OK;
}

}  // namespace

extern "C" {

int kvlink_version(void) { return 100; }

const char* kvlink_strerror(int code) {
    switch (code) {
        case KVLINK_OK: return "ok";
        case KVLINK_EINVAL: return "invalid argument";
        case KVLINK_EBOUNDS: return "index out of bounds";
        case KVLINK_ECAPACITY: return "buffer too small";
        case KVLINK_EUNSUPPORTED: return "unsupported shape";
        case KVLINK_ECUDA: return "CUDA error";
        case KVLINK_EDEVICE: return "device-side error recorded in the status word";
        default: return "unknown error";
    }
}

const char* kvlink_last_cuda_error(void) { return g_last_cuda_error.c_str(); }

namespace kvlink {
PinnedStaging::~PinnedStaging() {
    // errors are ignored: at process exit the runtime may already be gone
    if (done) {
        cudaEventSynchronize(done);
        cudaEventDestroy(done);
    }
    if (ptr) cudaFreeHost(ptr);
}

EventPool::~EventPool() {
    for (cudaEvent_t e : ev) cudaEventDestroy(e);
}

static int events_reserve(EventPool& pool, size_t n) {
    while (pool.ev.size() < n) {
        cudaEvent_t e = nullptr;
        cudaError_t err = cudaEventCreateWithFlags(&e, cudaEventDisableTiming);
        if (err != cudaSuccess) return cuda_fail(err, "event");
        pool.ev.push_back(e);
    }
    return KVLINK_OK;
}

// Room for `bytes` in the staging buffer, once the last copy out of it has completed.
static int staging_reserve(PinnedStaging& st, size_t bytes) {
    if (st.done) {
        cudaError_t e = cudaEventSynchronize(st.done);
        if (e != cudaSuccess) return cuda_fail(e, "kvlink_plan_upload: previous copy");
    } else {
        cudaError_t e = cudaEventCreateWithFlags(&st.done, cudaEventDisableTiming);
        if (e != cudaSuccess) return cuda_fail(e, "kvlink_plan_upload: event");
    }
    if (st.bytes >= bytes) return KVLINK_OK;
    if (st.ptr) cudaFreeHost(st.ptr);
    st.ptr = nullptr;
    st.bytes = 0;
    void* h = nullptr;
    cudaError_t e = cudaHostAlloc(&h, bytes, cudaHostAllocDefault);
    if (e != cudaSuccess) return cuda_fail(e, "kvlink_plan_upload: pinned staging");
    std::memset(h, 0, bytes);
    st.ptr = (char*)h;
    st.bytes = bytes;
    return KVLINK_OK;
}
}  // namespace kvlink

int kvlink_plan_create(const kvlink_batch_desc_t* desc, kvlink_plan_t** out) {
    if (!desc || !out) return KVLINK_EINVAL;
    *out = nullptr;
    kvlink_plan* p = new (std::nothrow) kvlink_plan();
    if (!p) return KVLINK_ECAPACITY;
    std::string why;
    int rc;
    try {
        rc = build_plan(desc, resolve_num_sms(desc->num_sms), p, &why);
    } catch (...) {
        rc = KVLINK_ECAPACITY;
    }
    if (rc != KVLINK_OK) {
        delete p;
        return rc;
    }
    p->built = true;
    *out = p;
    return KVLINK_OK;
}

int kvlink_plan_rebuild(kvlink_plan_t* p, const kvlink_batch_desc_t* desc) {
    if (!p || !desc) return KVLINK_EINVAL;
    // a fresh plan that takes over the old one's table storage (cleared, capacity kept, so
    // the tables are rebuilt in memory that is already mapped) and its staging buffer
    kvlink_plan q;
    q.staging = std::move(p->staging);
    // the events of earlier calls still order this plan's next calls after them
    q.events = std::move(p->events);
    q.host_events = std::move(p->host_events);
    q.host_chain_layers = p->host_chain_layers;
#define KVLINK_RECYCLE(m) \
    q.m.swap(p->m);       \
    q.m.clear();
    KVLINK_RECYCLE(pool_start) KVLINK_RECYCLE(pool_len) KVLINK_RECYCLE(pool_block_table) KVLINK_RECYCLE(seg)
    KVLINK_RECYCLE(chunks) KVLINK_RECYCLE(chunks_sorted) KVLINK_RECYCLE(cu_ctx) KVLINK_RECYCLE(cu_fresh)
    KVLINK_RECYCLE(fresh_pos) KVLINK_RECYCLE(fresh_query) KVLINK_RECYCLE(src) KVLINK_RECYCLE(src_row)
    KVLINK_RECYCLE(fresh_vis) KVLINK_RECYCLE(fresh_row0) KVLINK_RECYCLE(fresh_dst) KVLINK_RECYCLE(cu_grp)
    KVLINK_RECYCLE(grp_src)
    KVLINK_RECYCLE(items) KVLINK_RECYCLE(merges) KVLINK_RECYCLE(sched) KVLINK_RECYCLE(cu_sched)
    KVLINK_RECYCLE(slot_group)
#undef KVLINK_RECYCLE
    std::string why;
    int rc;
    try {
        rc = build_plan(desc, resolve_num_sms(desc->num_sms), &q, &why);
    } catch (...) {
        rc = KVLINK_ECAPACITY;
    }
    q.built = rc == KVLINK_OK;
    *p = std::move(q);
    return rc;
}

void kvlink_plan_destroy(kvlink_plan_t* plan) { delete plan; }

int kvlink_plan_get_info(const kvlink_plan_t* p, kvlink_plan_info_t* info) {
    if (!p || !info) return KVLINK_EINVAL;
    std::memset(info, 0, sizeof(*info));
    info->batch = p->batch;
    info->h_q = p->h_q;
    info->h_kv = p->h_kv;
    info->head_dim = p->head_dim;
    info->n_link = p->n_link;
    info->n_segments = (int32_t)p->seg.size();
    info->n_rope_rows = p->n_rope_rows;
    info->n_fresh = p->cu_fresh.empty() ? 0 : p->cu_fresh.back();
    info->ctx_rows = p->cu_ctx.empty() ? 0 : p->cu_ctx.back();
    info->cached_tokens = p->cached_tokens;
    info->n_copy_chunks = (int32_t)p->chunks.size();
    info->n_attn_items = (int32_t)p->items.size();
    info->n_attn_splits = p->n_slots;
    info->num_sms = p->num_sms;
    info->device_bytes = p->device_bytes;
    info->workspace_bytes = p->workspace_bytes;
    info->attn_pairs = p->attn_pairs;
    info->n_attn_ctas = p->cu_sched.empty() ? 0 : (int32_t)p->cu_sched.size() - 1;
    return KVLINK_OK;
}

int kvlink_plan_get_segments(const kvlink_plan_t* p, kvlink_segment_t* seg, int32_t cap) {
    if (!p || !seg) return KVLINK_EINVAL;
    if (cap < (int32_t)p->seg.size()) return KVLINK_ECAPACITY;
    std::memcpy(seg, p->seg.data(), p->seg.size() * sizeof(kvlink_segment_t));
    return KVLINK_OK;
}

int kvlink_plan_get_offsets(const kvlink_plan_t* p, int64_t* cu_ctx, int32_t* cu_fresh) {
    if (!p || !cu_ctx || !cu_fresh) return KVLINK_EINVAL;
    std::memcpy(cu_ctx, p->cu_ctx.data(), p->cu_ctx.size() * sizeof(int64_t));
    std::memcpy(cu_fresh, p->cu_fresh.data(), p->cu_fresh.size() * sizeof(int32_t));
    return KVLINK_OK;
}

int kvlink_plan_get_fresh_positions(const kvlink_plan_t* p, int32_t* pos, int32_t cap) {
    if (!p || !pos) return KVLINK_EINVAL;
    if (cap < (int32_t)p->fresh_pos.size()) return KVLINK_ECAPACITY;
    std::memcpy(pos, p->fresh_pos.data(), p->fresh_pos.size() * sizeof(int32_t));
    return KVLINK_OK;
}

int kvlink_plan_get_sources(const kvlink_plan_t* p, kvlink_source_t* src, int64_t cap) {
    if (!p || !src) return KVLINK_EINVAL;
    if (cap < (int64_t)p->src.size()) return KVLINK_ECAPACITY;
    std::memcpy(src, p->src.data(), p->src.size() * sizeof(kvlink_source_t));
    return KVLINK_OK;
}

static_assert(KVLINK_GROUP_FRESH == kvlink::kGrpFresh, "value-group fresh bit");
int kvlink_plan_get_value_groups(const kvlink_plan_t* p, int32_t* grp, int32_t* cu_grp, int64_t cap) {
    if (!p || !grp || !cu_grp) return KVLINK_EINVAL;
    if (cap < (int64_t)p->grp_src.size()) return KVLINK_ECAPACITY;
    std::memcpy(grp, p->grp_src.data(), p->grp_src.size() * sizeof(int32_t));
    std::memcpy(cu_grp, p->cu_grp.data(), p->cu_grp.size() * sizeof(int32_t));
    return KVLINK_OK;
}

int kvlink_plan_get_attention_items(const kvlink_plan_t* p, kvlink_attn_item_t* items, int32_t cap) {
    if (!p || !items) return KVLINK_EINVAL;
    if (cap < (int32_t)p->sched.size()) return KVLINK_ECAPACITY;
    int32_t k = 0;
    for (size_t c = 0; c + 1 < p->cu_sched.size(); ++c)
        for (int32_t s = p->cu_sched[c]; s < p->cu_sched[c + 1]; ++s) {
            const AttnItem& it = p->items[(size_t)p->sched[(size_t)s]];
            items[k++] = kvlink_attn_item_t{it.query,   it.kv_head,  it.tok0, it.tok1,       it.kv_tile0,
                                            it.kv_tile1, it.a_tiles, it.b_tile0, it.slot, (int32_t)c};
        }
    return KVLINK_OK;
}

int kvlink_plan_upload(kvlink_plan_t* p, double theta, void* d_buf, size_t bytes, kvlink_stream_t stream) {
    if (!p || !d_buf) return KVLINK_EINVAL;
    if (!(theta > 1.0)) return KVLINK_EINVAL;
    if (((uintptr_t)d_buf & 255u) != 0) return KVLINK_EINVAL;
    if (bytes < p->device_bytes) return KVLINK_ECAPACITY;
    if (!p->built) return KVLINK_EINVAL;
    int rc = staging_reserve(p->staging, p->device_bytes);
    if (rc != KVLINK_OK) return rc;
    char* host = p->staging.ptr;
    auto put = [&](size_t off, const void* src, size_t n) {
        if (n) std::memcpy(host + off, src, n);
    };
    put(p->off_seg, p->seg.data(), p->seg.size() * sizeof(kvlink_segment_t));
    put(p->off_chunks, p->chunks.data(), p->chunks.size() * sizeof(CopyChunk));
    put(p->off_chunks_sorted, p->chunks_sorted.data(), p->chunks_sorted.size() * sizeof(CopyChunk));
    put(p->off_pool_start, p->pool_start.data(), p->pool_start.size() * sizeof(int64_t));
    put(p->off_pool_bt, p->pool_block_table.data(), p->pool_block_table.size() * sizeof(int32_t));
    put(p->off_cu_ctx, p->cu_ctx.data(), p->cu_ctx.size() * sizeof(int64_t));
    put(p->off_cu_fresh, p->cu_fresh.data(), p->cu_fresh.size() * sizeof(int32_t));
    put(p->off_fresh_pos, p->fresh_pos.data(), p->fresh_pos.size() * sizeof(int32_t));
    put(p->off_fresh_query, p->fresh_query.data(), p->fresh_query.size() * sizeof(int32_t));
    put(p->off_items, p->items.data(), p->items.size() * sizeof(AttnItem));
    put(p->off_merges, p->merges.data(), p->merges.size() * sizeof(MergeGroup));
    put(p->off_src, p->src.data(), p->src.size() * sizeof(kvlink_source_t));
    put(p->off_cu_grp, p->cu_grp.data(), p->cu_grp.size() * sizeof(int32_t));
    put(p->off_grp_src, p->grp_src.data(), p->grp_src.size() * sizeof(int32_t));
    put(p->off_src_row, p->src_row.data(), p->src_row.size() * sizeof(kvlink_source_t));
    put(p->off_fresh_vis, p->fresh_vis.data(), p->fresh_vis.size() * sizeof(int32_t));
    put(p->off_fresh_row0, p->fresh_row0.data(), p->fresh_row0.size() * sizeof(int32_t));
    put(p->off_fresh_dst, p->fresh_dst.data(), p->fresh_dst.size() * sizeof(int32_t));
    put(p->off_sched, p->sched.data(), p->sched.size() * sizeof(int32_t));
    put(p->off_cu_sched, p->cu_sched.data(), p->cu_sched.size() * sizeof(int32_t));
    put(p->off_slot_group, p->slot_group.data(), p->slot_group.size() * sizeof(int32_t));
    std::memset(host + p->off_merge_count, 0, p->merges.size() * sizeof(unsigned long long));
    cudaStream_t s = (cudaStream_t)stream;
    cudaError_t e = cudaMemcpyAsync(d_buf, host, p->device_bytes, cudaMemcpyHostToDevice, s);
    if (e != cudaSuccess) return cuda_fail(e, "kvlink_plan_upload copy");
    // asynchronous: the next upload (or the plan's destruction) waits for this copy
    e = cudaEventRecord(p->staging.done, s);
    if (e != cudaSuccess) return cuda_fail(e, "kvlink_plan_upload event");
    char* b = (char*)d_buf;
    DevicePlan& d = p->dev;
    d.seg = (const kvlink_segment_t*)(b + p->off_seg);
    d.chunks = (const CopyChunk*)(b + p->off_chunks);
    d.chunks_sorted = (const CopyChunk*)(b + p->off_chunks_sorted);
    d.rope = (const float4*)(b + p->off_rope);
    d.pool_start = (const int64_t*)(b + p->off_pool_start);
    d.pool_block_table = (const int32_t*)(b + p->off_pool_bt);
    d.cu_ctx = (const int64_t*)(b + p->off_cu_ctx);
    d.cu_fresh = (const int32_t*)(b + p->off_cu_fresh);
    d.fresh_pos = (const int32_t*)(b + p->off_fresh_pos);
    d.fresh_query = (const int32_t*)(b + p->off_fresh_query);
    d.items = (const AttnItem*)(b + p->off_items);
    d.merges = (const MergeGroup*)(b + p->off_merges);
    d.src = (const kvlink_source_t*)(b + p->off_src);
    d.cu_grp = (const int32_t*)(b + p->off_cu_grp);
    d.grp_src = (const int32_t*)(b + p->off_grp_src);
    d.src_row = (const kvlink_source_t*)(b + p->off_src_row);
    d.fresh_vis = (const int32_t*)(b + p->off_fresh_vis);
    d.fresh_row0 = (const int32_t*)(b + p->off_fresh_row0);
    d.fresh_dst = (const int32_t*)(b + p->off_fresh_dst);
    d.sched = (const int32_t*)(b + p->off_sched);
    d.cu_sched = (const int32_t*)(b + p->off_cu_sched);
    d.slot_group = (const int32_t*)(b + p->off_slot_group);
    d.merge_count = (unsigned long long*)(b + p->off_merge_count);
    d.n_merges = (int32_t)p->merges.size();
    d.batch = p->batch;
    d.h_kv = p->h_kv;
    d.n_fresh = p->cu_fresh.back();
    d.n_slots = p->n_slots;
    d.n_rope_rows = p->n_rope_rows;
    d.n_items = (int32_t)p->items.size();
    d.ctx_rows = p->cu_ctx.back();
    d.pool_rows = p->pool_rows;
    launch_rope_table(d.seg, (int)p->seg.size(), (float4*)(b + p->off_rope), p->head_dim, theta, s);
    rc = check_launch("rope_table_kernel");
    if (rc != KVLINK_OK) return rc;
    p->theta = theta;
    p->d_buf = d_buf;
    p->uploaded = true;
    return KVLINK_OK;
}

int kvlink_reencode_concat(const kvlink_plan_t* p, const void* pool_k, const void* pool_v,
                           void* cache_k, void* cache_v, kvlink_stream_t stream) {
    int rc = check_plan(p);
    if (rc) return rc;
    // cache_v NULL: keys only (zero-copy values); pool_v is then not read
    if (!pool_k || !cache_k || (cache_v && !pool_v)) return KVLINK_EINVAL;
    if (!aligned16(pool_k) || !aligned16(cache_k) || (cache_v && (!aligned16(pool_v) || !aligned16(cache_v))))
        return KVLINK_EINVAL;
    launch_reencode(p->dev, 0, p->n_chunks_cached, p->head_dim, p->h_kv, p->num_sms, pool_k, pool_v, nullptr,
                    nullptr, cache_k, cache_v, (cudaStream_t)stream);
    return check_launch("reencode_kernel");
}

static bool all_aligned(int32_t n, const void* const* a) {
    for (int32_t l = 0; l < n; ++l)
        if (!a[l] || !aligned16(a[l])) return false;
    return true;
}

int kvlink_reencode_concat_layers(const kvlink_plan_t* p, int32_t n_layers, const void* const* pool_k,
                                  const void* const* pool_v, void* const* cache_k, void* const* cache_v,
                                  kvlink_stream_t stream) {
    int rc = check_plan(p);
    if (rc) return rc;
    // cache_v NULL: keys only for every layer (zero-copy values); pool_v is then not read
    if (n_layers <= 0 || !pool_k || !cache_k || (cache_v && !pool_v)) return KVLINK_EINVAL;
    if (!all_aligned(n_layers, pool_k) || !all_aligned(n_layers, (const void* const*)cache_k) ||
        (cache_v && (!all_aligned(n_layers, pool_v) || !all_aligned(n_layers, (const void* const*)cache_v))))
        return KVLINK_EINVAL;
    std::vector<const void*> no_pool_v;
    std::vector<void*> no_cache_v;
    if (!cache_v) {
        no_pool_v.assign((size_t)n_layers, nullptr);
        no_cache_v.assign((size_t)n_layers, nullptr);
        pool_v = no_pool_v.data();
        cache_v = no_cache_v.data();
    }
    launch_reencode_layers(p->dev, p->n_chunks_cached, p->head_dim, p->h_kv, p->num_sms, n_layers, pool_k, pool_v,
                           cache_k, cache_v, (cudaStream_t)stream);
    return check_launch("reencode_kernel (layers)");
}

static int place_fresh(const kvlink_plan_t* p, const void* k_new, const void* v_new, void* cache_k,
                       void* cache_v, cudaStream_t s) {
    launch_place_fresh(p->dev.fresh_dst, p->cu_fresh.back(), p->cu_ctx.back(), p->h_kv * p->head_dim * 2, k_new,
                       v_new, cache_k, cache_v, s);
    return check_launch("place_fresh_kernel");
}

// The attention's arguments (vs.cache_v NULL: zero-copy values, read from vs.pool_v and
// vs.v_new).  The entry points that launch something before the attention check them first,
// so that a call returning an error has launched nothing.
static int attention_args(const kvlink_plan_t* p, const void* q, const void* cache_k, const ValueSource& vs,
                          const void* out, const void* ws, size_t ws_bytes) {
    if (!q || !cache_k || !out) return KVLINK_EINVAL;
    if (!aligned16(q) || !aligned16(cache_k) || !aligned16(out)) return KVLINK_EINVAL;
    if (vs.cache_v ? !aligned16(vs.cache_v)
                   : (!vs.pool_v || !vs.v_new || !aligned16(vs.pool_v) || !aligned16(vs.v_new)))
        return KVLINK_EINVAL;
    if (p->workspace_bytes > 0 && (!ws || ws_bytes < p->workspace_bytes)) return KVLINK_ECAPACITY;
    if (ws && !aligned16(ws)) return KVLINK_EINVAL;
    return KVLINK_OK;
}

static int attention_common(const kvlink_plan_t* p, const void* q, void* cache_k, const ValueSource& vs,
                            void* out, void* ws, size_t ws_bytes, cudaStream_t s) {
    const int arc = attention_args(p, q, cache_k, vs, out, ws, ws_bytes);
    if (arc) return arc;
    cudaError_t err = cudaSuccess;
    const int rc = launch_attention_tc(p->dev, (int)p->items.size(), (int)p->cu_sched.size() - 1,
                                       (int)p->merges.size(), p->cu_fresh.back(),
                                       p->cu_ctx.back(), p->head_dim, p->h_q, p->h_kv, q, cache_k, vs, out,
                                       ws, s, &err);
    if (rc == KVLINK_ECUDA) return cuda_fail(err, "suffix attention launch");
    return rc;
}

// the values of the linked cache, or (cache_v NULL) where they are
static ValueSource values(void* cache_v, const void* pool_v, const void* v_new) {
    return cache_v ? ValueSource{cache_v, nullptr, nullptr} : ValueSource{nullptr, pool_v, v_new};
}

int kvlink_suffix_attention(const kvlink_plan_t* p, const void* q, const void* k_new, const void* v_new,
                            void* cache_k, void* cache_v, void* out, void* ws, size_t ws_bytes,
                            kvlink_stream_t stream) {
    int rc = check_plan(p);
    if (rc) return rc;
    if ((k_new == nullptr) != (v_new == nullptr)) return KVLINK_EINVAL;
    if (k_new && (!aligned16(k_new) || !aligned16(v_new))) return KVLINK_EINVAL;
    if (!cache_k || !cache_v) return KVLINK_EINVAL;
    rc = attention_args(p, q, cache_k, values(cache_v, nullptr, nullptr), out, ws, ws_bytes);
    if (rc) return rc;
    cudaStream_t s = (cudaStream_t)stream;
    if (k_new) {
        rc = place_fresh(p, k_new, v_new, cache_k, cache_v, s);
        if (rc) return rc;
    }
    return attention_common(p, q, cache_k, values(cache_v, nullptr, nullptr), out, ws, ws_bytes, s);
}

int kvlink_suffix_attention_pool_values(const kvlink_plan_t* p, const void* q, const void* k_new,
                                        const void* v_new, const void* pool_v, void* cache_k, void* out, void* ws,
                                        size_t ws_bytes, kvlink_stream_t stream) {
    int rc = check_plan(p);
    if (rc) return rc;
    if (!v_new || !pool_v || !cache_k) return KVLINK_EINVAL;
    if (k_new && !aligned16(k_new)) return KVLINK_EINVAL;
    rc = attention_args(p, q, cache_k, values(nullptr, pool_v, v_new), out, ws, ws_bytes);
    if (rc) return rc;
    cudaStream_t s = (cudaStream_t)stream;
    if (k_new) {
        rc = place_fresh(p, k_new, nullptr, cache_k, nullptr, s);
        if (rc) return rc;
    }
    return attention_common(p, q, cache_k, values(nullptr, pool_v, v_new), out, ws, ws_bytes, s);
}

int kvlink_suffix_attention_simt(const kvlink_plan_t* p, const void* q, const void* k_new, const void* v_new,
                                 void* cache_k, void* cache_v, void* out, kvlink_stream_t stream) {
    int rc = check_plan(p);
    if (rc) return rc;
    if ((k_new == nullptr) != (v_new == nullptr)) return KVLINK_EINVAL;
    if (k_new && (!aligned16(k_new) || !aligned16(v_new))) return KVLINK_EINVAL;
    if (!q || !cache_k || !cache_v || !out) return KVLINK_EINVAL;
    if (!aligned16(q) || !aligned16(cache_k) || !aligned16(cache_v) || !aligned16(out)) return KVLINK_EINVAL;
    cudaStream_t s = (cudaStream_t)stream;
    if (k_new) {
        rc = place_fresh(p, k_new, v_new, cache_k, cache_v, s);
        if (rc) return rc;
    }
    launch_attention_simt(p->dev, p->cu_fresh.back(), p->head_dim, p->h_q, p->h_kv, q, cache_k, cache_v, out, s);
    return check_launch("simt attention");
}

int kvlink_linked_prefill(const kvlink_plan_t* p, const void* pool_k, const void* pool_v, const void* q,
                          const void* k_new, const void* v_new, void* cache_k, void* cache_v, void* out,
                          void* ws, size_t ws_bytes, kvlink_stream_t stream) {
    int rc = check_plan(p);
    if (rc) return rc;
    // cache_v NULL: zero-copy values (keys re-encoded, values read where they are)
    if (!pool_k || !pool_v || !k_new || !v_new || !cache_k) return KVLINK_EINVAL;
    if (!aligned16(pool_k) || !aligned16(pool_v) || !aligned16(k_new) || !aligned16(v_new) ||
        (cache_v && !aligned16(cache_v)))
        return KVLINK_EINVAL;
    rc = attention_args(p, q, cache_k, values(cache_v, pool_v, v_new), out, ws, ws_bytes);
    if (rc) return rc;
    cudaStream_t s = (cudaStream_t)stream;
    launch_reencode(p->dev, 0, (int)p->chunks.size(), p->head_dim, p->h_kv, p->num_sms, pool_k, pool_v, k_new,
                    v_new, cache_k, cache_v, s);
    rc = check_launch("reencode_kernel (with the fresh rows)");
    if (rc) return rc;
    return attention_common(p, q, cache_k, values(cache_v, pool_v, v_new), out, ws, ws_bytes, s);
}

int kvlink_linked_prefill_fused(const kvlink_plan_t* p, const void* pool_k, const void* pool_v, const void* q,
                                const void* k_new, const void* v_new, void* cache_k, void* cache_v, void* out,
                                void* ws, size_t ws_bytes, kvlink_stream_t stream) {
    int rc = check_plan(p);
    if (rc) return rc;
    if (!pool_k || !pool_v || !q || !k_new || !v_new || !out) return KVLINK_EINVAL;
    if (!aligned16(pool_k) || !aligned16(pool_v) || !aligned16(q) || !aligned16(k_new) || !aligned16(v_new) ||
        !aligned16(out))
        return KVLINK_EINVAL;
    if ((cache_k && !aligned16(cache_k)) || (cache_v && !aligned16(cache_v))) return KVLINK_EINVAL;
    if (p->workspace_bytes > 0 && (!ws || ws_bytes < p->workspace_bytes)) return KVLINK_ECAPACITY;
    if (ws && !aligned16(ws)) return KVLINK_EINVAL;
    cudaError_t err = cudaSuccess;
    rc = launch_attention_fused(p->dev, (int)p->items.size(), (int)p->merges.size(), p->cu_fresh.back(),
                                p->pool_rows, p->head_dim, p->h_q, p->h_kv, q, pool_k, pool_v, k_new, v_new, cache_k,
                                cache_v, out, ws, (cudaStream_t)stream, &err);
    if (rc == KVLINK_ECUDA) return cuda_fail(err, "fused linked prefill launch");
    return rc;
}

int kvlink_linked_prefill_layers(const kvlink_plan_t* p, int32_t n_layers, const void* const* pool_k,
                                 const void* const* pool_v, const void* const* q, const void* const* k_new,
                                 const void* const* v_new, void* const* cache_k, void* const* cache_v,
                                 void* const* out, void* ws, size_t ws_bytes, kvlink_stream_t stream) {
    int rc = check_plan(p);
    if (rc) return rc;
    // cache_v NULL: zero-copy values in every layer
    if (n_layers <= 0 || !pool_k || !pool_v || !q || !k_new || !v_new || !cache_k || !out) return KVLINK_EINVAL;
    // every argument is checked before the first launch
    if (!all_aligned(n_layers, q) || !all_aligned(n_layers, k_new) || !all_aligned(n_layers, v_new) ||
        !all_aligned(n_layers, (const void* const*)out))
        return KVLINK_EINVAL;
    if (p->workspace_bytes > 0 && (!ws || ws_bytes < p->workspace_bytes)) return KVLINK_ECAPACITY;
    if (ws && !aligned16(ws)) return KVLINK_EINVAL;
    if (!all_aligned(n_layers, pool_k) || !all_aligned(n_layers, pool_v) ||
        !all_aligned(n_layers, (const void* const*)cache_k) ||
        (cache_v && !all_aligned(n_layers, (const void* const*)cache_v)))
        return KVLINK_EINVAL;
    // per layer, one re-encode launch that also places the fresh rows, then the suffix
    // attention.  (Re-encoding every layer's documents in one launch first streams at the
    // same rate and then needs a separate fresh-row launch per layer: slower.)
    for (int l = 0; l < n_layers; ++l) {
        rc = kvlink_linked_prefill(p, pool_k[l], pool_v[l], q[l], k_new[l], v_new[l], cache_k[l],
                                   cache_v ? cache_v[l] : nullptr, out[l], ws, ws_bytes, stream);
        if (rc) return rc;
    }
    return KVLINK_OK;
}

int kvlink_linked_prefill_layers_overlapped(kvlink_plan_t* p, int32_t n_layers, const void* const* pool_k,
                                            const void* const* pool_v, const void* const* q,
                                            const void* const* k_new, const void* const* v_new,
                                            void* const* cache_k, void* const* cache_v, void* const* out, void* ws,
                                            size_t ws_bytes, kvlink_stream_t stream,
                                            kvlink_stream_t reencode_stream) {
    int rc = check_plan(p);
    if (rc) return rc;
    // cache_v NULL: zero-copy values in every layer
    if (n_layers <= 0 || !pool_k || !pool_v || !q || !k_new || !v_new || !cache_k || !out) return KVLINK_EINVAL;
    if (stream == reencode_stream) return KVLINK_EINVAL;
    // every argument is checked before the first launch
    if (!all_aligned(n_layers, pool_k) || !all_aligned(n_layers, pool_v) ||
        !all_aligned(n_layers, (const void* const*)cache_k) ||
        (cache_v && !all_aligned(n_layers, (const void* const*)cache_v)) ||
        !all_aligned(n_layers, q) || !all_aligned(n_layers, k_new) || !all_aligned(n_layers, v_new) ||
        !all_aligned(n_layers, (const void* const*)out))
        return KVLINK_EINVAL;
    if (p->workspace_bytes > 0 && (!ws || ws_bytes < p->workspace_bytes)) return KVLINK_ECAPACITY;
    if (ws && !aligned16(ws)) return KVLINK_EINVAL;
    rc = events_reserve(p->events, (size_t)n_layers + 1);
    if (rc) return rc;
    cudaStream_t s = (cudaStream_t)stream, r = (cudaStream_t)reencode_stream;
    cudaEvent_t* ev = p->events.ev.data();
    // the re-encode stream starts after the work already on `stream` (the plan upload, the
    // pool), then re-encodes every layer's document caches back to back
    cudaError_t e = cudaEventRecord(ev[n_layers], s);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(r, ev[n_layers], 0);
    if (e != cudaSuccess) return cuda_fail(e, "linked_prefill_layers_overlapped: stream order");
    for (int l = 0; l < n_layers; ++l) {
        launch_reencode(p->dev, 0, p->n_chunks_cached, p->head_dim, p->h_kv, p->num_sms, pool_k[l], pool_v[l],
                        nullptr, nullptr, cache_k[l], cache_v ? cache_v[l] : nullptr, r);
        rc = check_launch("reencode_kernel (overlapped)");
        if (rc) return rc;
        e = cudaEventRecord(ev[l], r);
        if (e != cudaSuccess) return cuda_fail(e, "linked_prefill_layers_overlapped: event");
    }
    // per layer on `stream`: once its caches are in place, the fresh rows and the attention;
    // the last wait also orders every re-encode before later work on `stream`
    for (int l = 0; l < n_layers; ++l) {
        e = cudaStreamWaitEvent(s, ev[l], 0);
        if (e != cudaSuccess) return cuda_fail(e, "linked_prefill_layers_overlapped: wait");
        void* cv = cache_v ? cache_v[l] : nullptr;
        rc = place_fresh(p, k_new[l], v_new[l], cache_k[l], cv, s);
        if (rc) return rc;
        rc = attention_common(p, q[l], cache_k[l], values(cv, pool_v[l], v_new[l]), out[l], ws, ws_bytes, s);
        if (rc) return rc;
    }
    return KVLINK_OK;
}

int kvlink_linked_prefill_layers_host(kvlink_plan_t* p, int32_t n_layers, const void* const* pool_k,
                                      const void* const* pool_v, const void* const* h_q, const void* const* h_k_new,
                                      const void* const* h_v_new, void* const* q, void* const* k_new,
                                      void* const* v_new, void* const* cache_k, void* const* cache_v,
                                      void* const* out, void* const* h_out, void* ws, size_t ws_bytes,
                                      kvlink_stream_t stream, kvlink_stream_t reencode_stream,
                                      kvlink_stream_t copy_in_stream, kvlink_stream_t copy_out_stream) {
    int rc = check_plan(p);
    if (rc) return rc;
    // cache_v NULL: zero-copy values in every layer
    if (n_layers <= 0 || !pool_k || !pool_v || !h_q || !h_k_new || !h_v_new || !q || !k_new || !v_new ||
        !cache_k || !out || !h_out)
        return KVLINK_EINVAL;
    if (stream == reencode_stream || stream == copy_in_stream || stream == copy_out_stream ||
        reencode_stream == copy_in_stream || reencode_stream == copy_out_stream || copy_in_stream == copy_out_stream)
        return KVLINK_EINVAL;
    auto cv = [](void* const* a) { return (const void* const*)a; };
    if (!all_aligned(n_layers, pool_k) || !all_aligned(n_layers, pool_v) || !all_aligned(n_layers, cv(q)) ||
        !all_aligned(n_layers, cv(k_new)) || !all_aligned(n_layers, cv(v_new)) || !all_aligned(n_layers, cv(cache_k)) ||
        (cache_v && !all_aligned(n_layers, cv(cache_v))) || !all_aligned(n_layers, cv(out)))
        return KVLINK_EINVAL;
    for (int l = 0; l < n_layers; ++l)
        if (!h_q[l] || !h_k_new[l] || !h_v_new[l] || !h_out[l]) return KVLINK_EINVAL;
    if (p->workspace_bytes > 0 && (!ws || ws_bytes < p->workspace_bytes)) return KVLINK_ECAPACITY;
    if (ws && !aligned16(ws)) return KVLINK_EINVAL;
    // events (the plan's host-path pool, used by no other entry point): [0, L) caches in
    // place, [L, 2L) inputs in place, [2L, 3L) layer computed, [3L, 4L) output on the host,
    // 4L the call's start.  When the previous call had as many layers, its records of the
    // last two kinds order this call's rewrites of the same buffers after their readers,
    // layer by layer.  Otherwise this call is ordered after the whole previous call: `stream`
    // waits for its last output copy (which followed every layer it computed), and the copy
    // and re-encode streams wait for this call's start on `stream`.
    const int32_t prev_layers = p->host_chain_layers;
    const bool chained = prev_layers == n_layers;
    rc = events_reserve(p->host_events, 4 * (size_t)std::max(n_layers, prev_layers) + 1);
    if (rc) return rc;
    cudaEvent_t* ev = p->host_events.ev.data();
    cudaEvent_t *ev_re = ev, *ev_in = ev + n_layers, *ev_c = ev + 2 * n_layers, *ev_o = ev + 3 * n_layers;
    cudaStream_t s = (cudaStream_t)stream, r = (cudaStream_t)reencode_stream, ci = (cudaStream_t)copy_in_stream,
                 co = (cudaStream_t)copy_out_stream;
    const size_t n_fresh = (size_t)p->cu_fresh.back();
    const size_t q_bytes = n_fresh * p->h_q * p->head_dim * 2, kv_bytes = n_fresh * p->h_kv * p->head_dim * 2;
    cudaError_t e = cudaSuccess;
    // the previous call's last output copy: waited for before any event is recorded again
    if (!chained && prev_layers > 0) e = cudaStreamWaitEvent(s, ev[4 * prev_layers - 1], 0);
    if (e == cudaSuccess) e = cudaEventRecord(ev[4 * n_layers], s);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(r, ev[4 * n_layers], 0);
    if (e == cudaSuccess && !chained) e = cudaStreamWaitEvent(ci, ev[4 * n_layers], 0);
    if (e != cudaSuccess) return cuda_fail(e, "linked_prefill_layers_host: stream order");
    // the document caches of every layer, on the re-encode stream
    for (int l = 0; l < n_layers; ++l) {
        if (chained && (e = cudaStreamWaitEvent(r, ev_c[l], 0)) != cudaSuccess)
            return cuda_fail(e, "linked_prefill_layers_host: wait");
        launch_reencode(p->dev, 0, p->n_chunks_cached, p->head_dim, p->h_kv, p->num_sms, pool_k[l], pool_v[l],
                        nullptr, nullptr, cache_k[l], cache_v ? cache_v[l] : nullptr, r);
        rc = check_launch("reencode_kernel (host path)");
        if (rc) return rc;
        if ((e = cudaEventRecord(ev_re[l], r)) != cudaSuccess) return cuda_fail(e, "linked_prefill_layers_host");
    }
    for (int l = 0; l < n_layers; ++l) {
        // fresh rows in from the host
        if (chained && (e = cudaStreamWaitEvent(ci, ev_c[l], 0)) != cudaSuccess)
            return cuda_fail(e, "linked_prefill_layers_host: wait");
        e = cudaMemcpyAsync(q[l], h_q[l], q_bytes, cudaMemcpyHostToDevice, ci);
        if (e == cudaSuccess) e = cudaMemcpyAsync(k_new[l], h_k_new[l], kv_bytes, cudaMemcpyHostToDevice, ci);
        if (e == cudaSuccess) e = cudaMemcpyAsync(v_new[l], h_v_new[l], kv_bytes, cudaMemcpyHostToDevice, ci);
        if (e == cudaSuccess) e = cudaEventRecord(ev_in[l], ci);
        // the layer, once its inputs and caches are in place (and the previous call's output
        // of this layer has left)
        if (e == cudaSuccess) e = cudaStreamWaitEvent(s, ev_in[l], 0);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(s, ev_re[l], 0);
        if (e == cudaSuccess && chained) e = cudaStreamWaitEvent(s, ev_o[l], 0);
        if (e != cudaSuccess) return cuda_fail(e, "linked_prefill_layers_host: inputs");
        void* cvl = cache_v ? cache_v[l] : nullptr;
        rc = place_fresh(p, k_new[l], v_new[l], cache_k[l], cvl, s);
        if (rc) return rc;
        rc = attention_common(p, q[l], cache_k[l], values(cvl, pool_v[l], v_new[l]), out[l], ws, ws_bytes, s);
        if (rc) return rc;
        // the output back to the host
        e = cudaEventRecord(ev_c[l], s);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(co, ev_c[l], 0);
        if (e == cudaSuccess) e = cudaMemcpyAsync(h_out[l], out[l], q_bytes, cudaMemcpyDeviceToHost, co);
        if (e == cudaSuccess) e = cudaEventRecord(ev_o[l], co);
        if (e != cudaSuccess) return cuda_fail(e, "linked_prefill_layers_host: output");
    }
    p->host_chain_layers = n_layers;
    return KVLINK_OK;
}

// The device's address of page-locked host memory (cudaHostAlloc, cudaHostRegister): the
// kernels read the pool through it.  Pageable memory and device memory are rejected.
static int host_pool_view(const void* h, const void** d) {
    if (!h) return KVLINK_EINVAL;
    cudaPointerAttributes a;
    const cudaError_t e = cudaPointerGetAttributes(&a, h);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return KVLINK_EINVAL;
    }
    if (a.type != cudaMemoryTypeHost || !a.devicePointer || !aligned16(a.devicePointer)) return KVLINK_EINVAL;
    *d = a.devicePointer;
    return KVLINK_OK;
}

int kvlink_reencode_concat_host_pool(const kvlink_plan_t* p, const void* h_pool_k, const void* h_pool_v,
                                     void* cache_k, void* cache_v, kvlink_stream_t stream) {
    int rc = check_plan(p);
    if (rc) return rc;
    if (!cache_k || !cache_v || !aligned16(cache_k) || !aligned16(cache_v)) return KVLINK_EINVAL;
    const void *dk = nullptr, *dv = nullptr;
    if ((rc = host_pool_view(h_pool_k, &dk)) || (rc = host_pool_view(h_pool_v, &dv))) return rc;
    launch_reencode_host(p->dev, p->n_chunks_cached, p->head_dim, p->h_kv, p->num_sms, dk, dv, cache_k, cache_v,
                         (cudaStream_t)stream);
    return check_launch("reencode_host_kernel");
}

int kvlink_linked_prefill_layers_host_pool(kvlink_plan_t* p, int32_t n_layers, const void* const* h_pool_k,
                                           const void* const* h_pool_v, const void* const* q,
                                           const void* const* k_new, const void* const* v_new, void* const* cache_k,
                                           void* const* cache_v, void* const* out, void* ws, size_t ws_bytes,
                                           kvlink_stream_t stream, kvlink_stream_t load_stream) {
    int rc = check_plan(p);
    if (rc) return rc;
    if (n_layers <= 0 || !h_pool_k || !h_pool_v || !q || !k_new || !v_new || !cache_k || !cache_v || !out)
        return KVLINK_EINVAL;
    if (stream == load_stream) return KVLINK_EINVAL;
    if (!all_aligned(n_layers, (const void* const*)cache_k) || !all_aligned(n_layers, (const void* const*)cache_v) ||
        !all_aligned(n_layers, q) || !all_aligned(n_layers, k_new) || !all_aligned(n_layers, v_new) ||
        !all_aligned(n_layers, (const void* const*)out))
        return KVLINK_EINVAL;
    if (p->workspace_bytes > 0 && (!ws || ws_bytes < p->workspace_bytes)) return KVLINK_ECAPACITY;
    if (ws && !aligned16(ws)) return KVLINK_EINVAL;
    // every host pool pointer is resolved (and checked) before the first launch
    std::vector<const void*> dk((size_t)n_layers), dv((size_t)n_layers);
    for (int l = 0; l < n_layers; ++l)
        if ((rc = host_pool_view(h_pool_k[l], &dk[l])) || (rc = host_pool_view(h_pool_v[l], &dv[l]))) return rc;
    rc = events_reserve(p->events, (size_t)n_layers + 1);
    if (rc) return rc;
    cudaStream_t s = (cudaStream_t)stream, r = (cudaStream_t)load_stream;
    cudaEvent_t* ev = p->events.ev.data();
    cudaError_t e = cudaEventRecord(ev[n_layers], s);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(r, ev[n_layers], 0);
    if (e != cudaSuccess) return cuda_fail(e, "linked_prefill_layers_host_pool: stream order");
    // every layer's document caches loaded from host memory and re-encoded, back to back
    for (int l = 0; l < n_layers; ++l) {
        launch_reencode_host(p->dev, p->n_chunks_cached, p->head_dim, p->h_kv, p->num_sms, dk[l], dv[l], cache_k[l],
                             cache_v[l], r);
        rc = check_launch("reencode_host_kernel (layers)");
        if (rc) return rc;
        e = cudaEventRecord(ev[l], r);
        if (e != cudaSuccess) return cuda_fail(e, "linked_prefill_layers_host_pool: event");
    }
    for (int l = 0; l < n_layers; ++l) {
        e = cudaStreamWaitEvent(s, ev[l], 0);
        if (e != cudaSuccess) return cuda_fail(e, "linked_prefill_layers_host_pool: wait");
        rc = place_fresh(p, k_new[l], v_new[l], cache_k[l], cache_v[l], s);
        if (rc) return rc;
        rc = attention_common(p, q[l], cache_k[l], values(cache_v[l], nullptr, nullptr), out[l], ws, ws_bytes, s);
        if (rc) return rc;
    }
    return KVLINK_OK;
}

int kvlink_rope_fresh(const kvlink_plan_t* p, void* q, void* k_new, kvlink_stream_t stream) {
    int rc = check_plan(p);
    if (rc) return rc;
    if (!q || !k_new) return KVLINK_EINVAL;
    launch_rope_fresh(p->dev.fresh_pos, p->cu_fresh.back(), p->head_dim, p->theta, q, p->h_q, k_new, p->h_kv,
                      (cudaStream_t)stream);
    return check_launch("rope_fresh_kernel");
}

int kvlink_selftest_wait_timeout(uint32_t limit_ms, kvlink_stream_t stream) {
    if (limit_ms < 1 || limit_ms > 2000) return KVLINK_EINVAL;
    const int rc = launch_wait_selftest(limit_ms, (cudaStream_t)stream);
    return rc == KVLINK_OK ? KVLINK_OK : check_launch("wait_selftest_kernel");
}

int kvlink_device_status(int32_t* status) {
    if (!status) return KVLINK_EINVAL;
    int32_t a = 0, c = 0, f = 0;
    int rc = read_attention_status(&a);
    if (rc == KVLINK_OK) rc = read_copy_status(&c);
    if (rc == KVLINK_OK) rc = read_fused_status(&f);
    *status = a != 0 ? a : (c != 0 ? c : f);
    return rc;
}

int kvlink_clear_device_status(void) {
    int rc = clear_attention_status();
    if (rc == KVLINK_OK) rc = clear_copy_status();
    return rc != KVLINK_OK ? rc : clear_fused_status();
}

}  // extern "C"
