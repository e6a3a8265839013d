// kvlink_suffix_attention_noalloc: the suffix attention with its split-KV scratch in a
// fixed device array owned by this library, for callers that must not allocate.
//
// Who needs it: a serving loop that has fixed its whole memory budget at start-up
// and may not allocate on the request path (cudaMalloc can synchronise the device
// and fragments a pre-carved pool), and code that enqueues work from places where
// allocation is not allowed at all, such as a host callback.  Such callers still
// pass their own inputs and outputs; only the scratch moves here.
//
// The scratch is one file-scope __device__ array of KVLINK_NOALLOC_MAX_WORKSPACE_BYTES.
// Every GPU on which the library is loaded holds it until the process exits.  In host
// code its name only stands in for the symbol, so its device address is looked up
// with cudaGetSymbolAddress, once per device with that device current, on the first
// call made on that device; that first call should therefore come before any stream
// capture.  All calls share the array and it keeps the last call's contents: nothing
// in it needs to start at zero, because every partial slot the merge reads is written
// by the same call first.  Two calls whose work overlaps on the GPU (different streams,
// or different host threads on one device) race on the array.  The looked-up address
// stays cached for the life of the process, so resetting a device (cudaDeviceReset) after
// the first call on it is not supported: the next call would launch with a stale address.
#include <cuda_runtime.h>

#include <mutex>

#include "kvlink_internal.h"

namespace kvlink {
void launch_reencode(const DevicePlan& P, int chunk_base, int n_chunks, int head_dim, int h_kv, int num_sms,
                     const void* pool_k, const void* pool_v, const void* k_new, const void* v_new, void* cache_k,
                     void* cache_v, cudaStream_t stream);
void launch_place_fresh(const int32_t* d_fresh_dst, int n_fresh, int64_t ctx_rows, int row_bytes,
                        const void* k_new, const void* v_new, void* cache_k, void* cache_v, cudaStream_t stream);
int launch_attention_tc(const DevicePlan& P, int n_items, int n_ctas, int n_merges, int n_fresh, int64_t ctx_rows,
                        int head_dim, int h_q, int h_kv, const void* q, const void* cache_k, const ValueSource& vs,
                        void* out, void* ws, cudaStream_t stream, cudaError_t* err);
}  // namespace kvlink

static __device__ __align__(256) unsigned char g_noalloc_scratch[KVLINK_NOALLOC_MAX_WORKSPACE_BYTES];

namespace {

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of the scratch array on the current device (looked up once per device).
int scratch_on_current_device(void** addr) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return kvlink::record_cuda_error(e, "kvlink_suffix_attention_noalloc: device");
    if (dev < 0 || dev >= kMaxDevices) return KVLINK_EUNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_scratch_mu);
    if (!g_scratch_addr[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess) return kvlink::record_cuda_error(e, "kvlink_suffix_attention_noalloc: scratch address");
        if (!p)
            return kvlink::record_cuda_error(cudaErrorInvalidSymbol, "kvlink_suffix_attention_noalloc: scratch address");
        g_scratch_addr[dev] = p;
    }
    *addr = g_scratch_addr[dev];
    return KVLINK_OK;
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

}  // namespace

extern "C" int kvlink_suffix_attention_noalloc(const kvlink_plan_t* p, const void* q, const void* k_new,
                                               const void* v_new, void* cache_k, void* cache_v, void* out,
                                               kvlink_stream_t stream) {
    if (!p || !p->uploaded) return KVLINK_EINVAL;
    if ((k_new == nullptr) != (v_new == nullptr)) return KVLINK_EINVAL;
    if (!q || !cache_k || !cache_v || !out) return KVLINK_EINVAL;
    if (!aligned16(q) || !aligned16(cache_k) || !aligned16(cache_v) || !aligned16(out)) return KVLINK_EINVAL;
    if (k_new && (!aligned16(k_new) || !aligned16(v_new))) return KVLINK_EINVAL;
    if (p->workspace_bytes > (size_t)KVLINK_NOALLOC_MAX_WORKSPACE_BYTES) return KVLINK_ECAPACITY;
    void* ws = nullptr;
    int rc = scratch_on_current_device(&ws);
    if (rc != KVLINK_OK) return rc;
    cudaStream_t s = (cudaStream_t)stream;
    if (k_new) {
        kvlink::launch_place_fresh(p->dev.fresh_dst, p->cu_fresh.back(), p->cu_ctx.back(), p->h_kv * p->head_dim * 2,
                                   k_new, v_new, cache_k, cache_v, s);
        rc = kvlink::record_launch_error("place_fresh_kernel (noalloc)");
        if (rc != KVLINK_OK) return rc;
    }
    cudaError_t err = cudaSuccess;
    rc = kvlink::launch_attention_tc(p->dev, (int)p->items.size(), (int)p->cu_sched.size() - 1,
                                     (int)p->merges.size(), p->cu_fresh.back(),
                                     p->cu_ctx.back(), p->head_dim, p->h_q, p->h_kv, q, cache_k,
                                     kvlink::ValueSource{cache_v, nullptr, nullptr}, out, ws, s, &err);
    if (rc == KVLINK_ECUDA) return kvlink::record_cuda_error(err, "suffix attention launch (noalloc)");
    return rc;
}
