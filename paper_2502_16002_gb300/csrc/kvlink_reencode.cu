// RoPE delta table (Sec. 2.2, once per batch) and the re-encode + concat kernel
// (Sec. 2.2 positional re-encoding, Sec. 2.1 concatenation of the caches).
//
// The re-encode kernel is a streaming copy bound by HBM bandwidth.  Work units are
// runs of tokens whose K/V rows are contiguous in the source and in the linked
// cache (resolved on the host).  A persistent CTA per SM pipelines a contiguous range
// of units through a 3-stage shared-memory ring: one bulk (TMA) global -> shared load
// per group of consecutive units that read the same rows, document keys rotated on
// their way from shared memory to global memory, values and unrotated keys
// bulk-stored from shared memory.
//
// The rotation itself (double-float cos/sin, compensated products) is in
// kvlink_rope.cuh, shared with the fused linked-prefill kernel.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdint>

#include "kvlink_internal.h"
#include "kvlink_rope.cuh"
#include "kvlink_sm100.cuh"

namespace kvlink {

// --------------------------------------------------------------------------
// A2: cos/sin(delta * theta^(-2j/D)) for every cached document segment.
// The angle is formed and reduced in float64, so the rotation error does not
// grow with delta; cos and sin are stored as float pairs (hi, lo).
// --------------------------------------------------------------------------
__global__ void rope_table_kernel(const kvlink_segment_t* __restrict__ seg, int n_seg,
                                  float4* __restrict__ rope, int half, double theta, int head_dim) {
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= (int64_t)n_seg * half) return;
    const int s = (int)(i / half), j = (int)(i % half);
    const kvlink_segment_t sg = seg[s];
    if (sg.kind != KVLINK_SEG_DOC) return;
    const double inv_freq = pow(theta, -2.0 * (double)j / (double)head_dim);
    const double angle = (double)sg.pos * inv_freq;
    double sn, cs;
    sincos(angle, &sn, &cs);
    const float ch = (float)cs, sh = (float)sn;
    rope[(int64_t)sg.table * half + j] = make_float4(ch, (float)(cs - (double)ch), sh, (float)(sn - (double)sh));
}

void launch_rope_table(const kvlink_segment_t* d_seg, int n_seg, float4* d_rope, int head_dim,
                       double theta, cudaStream_t stream) {
    const int half = head_dim / 2;
    const int64_t n = (int64_t)n_seg * half;
    if (n == 0) return;
    const int threads = 256;
    rope_table_kernel<<<(unsigned)((n + threads - 1) / threads), threads, 0, stream>>>(
        d_seg, n_seg, d_rope, half, theta, head_dim);
}

// --------------------------------------------------------------------------
// A3 + A4: persistent re-encode/copy through a shared-memory ring.
// --------------------------------------------------------------------------
constexpr int kCopyConsumers = 256;                  // 8 warps rotate keys in shared memory
constexpr int kCopyThreads = 32 + kCopyConsumers;    // + 1 producer warp
constexpr int kCopyStages = 3;
constexpr uint64_t kCopyWaitLimitNs = 2000000000ull;
constexpr int32_t kCopyStatusWaitTimeout = 0x21;
#ifdef KVLINK_DEBUG_CHECKS
constexpr int32_t kCopyStatusBadIndex = 0x22;   // a table entry out of bounds
#endif

static __device__ int32_t g_copy_status;

// WV: a stage holds a unit's keys then its values (3 stages); keys only (zero-copy values):
// the same 192 KB as 6 stages of keys, so as many bytes stay in flight.
template <bool WV>
struct CopySmem {
    static constexpr int NST = WV ? kCopyStages : 2 * kCopyStages;
    static constexpr uint32_t STAGE = WV ? 2 * kCopyStageBytes : kCopyStageBytes;
    static constexpr uint32_t OFF_BAR = NST * STAGE;
    static constexpr uint32_t BYTES = OFF_BAR + 2 * NST * 8 + 16 + 128;
};

__device__ __forceinline__ bool copy_wait(uint64_t* bar, uint32_t parity, volatile int32_t* abort_flag) {
    if (sm100::mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = sm100::globaltimer_ns();
    while (true) {
        if (sm100::mbar_try_wait(bar, parity)) return true;
        if (*abort_flag) return false;
        if (sm100::globaltimer_ns() - t0 > kCopyWaitLimitNs) {
            *abort_flag = 1;
            atomicCAS(&g_copy_status, 0, kCopyStatusWaitTimeout);
            return false;
        }
    }
}

__device__ __forceinline__ void copy_drain(uint64_t* bar, uint32_t parity) {
    const uint64_t t0 = sm100::globaltimer_ns();
    while (!sm100::mbar_try_wait(bar, parity))
        if (sm100::globaltimer_ns() - t0 > kCopyWaitLimitNs) {
            atomicCAS(&g_copy_status, 0, kCopyStatusWaitTimeout);
            return;
        }
}

// Pool and linked-cache tensors of up to MAXL layers, passed by value.  Layer l's
// units are the plan's n_chunks units applied to pool_k[l], pool_v[l] -> cache_k[l],
// cache_v[l]; the document caches of every layer are inputs, so all layers can be
// re-encoded in one launch ahead of the per-layer attention.
template <int MAXL>
struct LayerPtrs {
    const __nv_bfloat16* pool_k[MAXL];
    const __nv_bfloat16* pool_v[MAXL];
    __nv_bfloat16* cache_k[MAXL];
    __nv_bfloat16* cache_v[MAXL];
};
constexpr int kMaxLayersPerLaunch = 64;     // 2 KB of kernel parameters

// Chunk u = layer * n_chunks + c of the flattened range.  CTA b handles the contiguous
// range [n*b/grid, n*(b+1)/grid), n = n_layers * n_chunks, in groups of consecutive
// chunks that read the same source rows (same layer, same tensor, same first row and
// length), loading each group's rows once.  The one-layer launches take the chunks in
// linked-cache order, where consecutive chunks read other rows (but for a document retrieved
// twice in a row with no link tokens between), so there a group is one chunk and the next
// chunk's entry is loaded a group ahead; the all-layer launch takes
// the document chunks sorted by pool row, so every destination of a document that
// several queries retrieved follows the first and its rows are loaded once per layer.
// (One layer is bound by the cache writes, which do not shrink; over all layers the
// saved reads pay: measured 1607 -> 1314 us for 32 layers of the Llama-8B batch-8
// workload, while grouping one layer's chunks moved its time from 50 to 53 us.)
// Producer (warp 0, one thread): bulk-loads a group's K rows and V rows into a stage.
// Consumers (warps 1-8), per chunk of the group: document keys are read from the stage,
// rotated by the chunk's delta in registers (each thread keeps a fixed (head, j0) slot
// and its eight double-float cos/sin pairs) and written with 16-byte global stores;
// one thread bulk-stores the values (and the keys of prefix and fresh chunks, which are
// not rotated) straight from the stage.  The stage is freed once the group's stores
// have read it and every consumer has passed the next group's barrier.  With zero-copy
// values (WV false, the linked cache has no value rows) only keys are loaded and stored,
// and the same shared memory holds twice as many stages.
__device__ __forceinline__ bool same_source(const CopyChunk& a, int la, const CopyChunk& b, int lb) {
    const bool fa = a.kind == KVLINK_SEG_LINK || a.kind == KVLINK_SEG_QUESTION;
    const bool fb = b.kind == KVLINK_SEG_LINK || b.kind == KVLINK_SEG_QUESTION;
    return la == lb && fa == fb && a.src_row == b.src_row && a.n == b.n;
}

template <int D, int MAXL, bool WV>
__global__ void __launch_bounds__(kCopyThreads, 1) reencode_kernel(
    const CopyChunk* __restrict__ chunks, int n_chunks, int n_layers, const float4* __restrict__ rope, int h_kv,
    const LayerPtrs<MAXL> L, const __nv_bfloat16* __restrict__ k_new, const __nv_bfloat16* __restrict__ v_new,
    const CopyBounds bounds) {
    using namespace sm100;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw_addr = smem_u32(smem_raw);
    uint8_t* smem = smem_raw + ((128u - (raw_addr & 127u)) & 127u);
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + CopySmem<WV>::OFF_BAR);
    uint64_t* empty = full + CopySmem<WV>::NST;
    volatile int32_t* abort_flag = reinterpret_cast<volatile int32_t*>(empty + CopySmem<WV>::NST);

    const int64_t n_units = (int64_t)n_chunks * n_layers;
    const int c_begin = (int)(n_units * blockIdx.x / gridDim.x);
    const int c_end = (int)(n_units * (blockIdx.x + 1) / gridDim.x);

    const int64_t row_elems = (int64_t)h_kv * D;
    const uint32_t row_bytes = (uint32_t)(row_elems * 2);
    auto layer_of = [&](int c) { return MAXL == 1 ? 0 : c / n_chunks; };
    // the end of the group that starts at chunk c
    auto group_end = [&](int c, int layer, const CopyChunk& ch) {
        int e = c + 1;
        while (e < c_end) {
            const int le = layer_of(e);
            if (!same_source(chunks[e - le * n_chunks], le, ch, layer)) break;
            ++e;
        }
        return e;
    };

    if (threadIdx.x == 0) {
        for (int i = 0; i < CopySmem<WV>::NST; ++i) {
            mbar_init(full + i, 1);
            mbar_init(empty + i, 1);
        }
        *abort_flag = *reinterpret_cast<volatile int32_t*>(&g_copy_status) != 0 ? 1 : 0;
#ifdef KVLINK_DEBUG_CHECKS
        // every unit of this CTA inside its tensors, before any copy uses one
        const int max_rows = kCopyStageBytes / (int)row_bytes;
        for (int c = c_begin; c < c_end && !*abort_flag; ++c) {
            const int layer = MAXL == 1 ? 0 : c / n_chunks;
            const CopyChunk ch = chunks[c - layer * n_chunks];
            const bool fresh = ch.kind == KVLINK_SEG_LINK || ch.kind == KVLINK_SEG_QUESTION;
            const bool ok = ch.n >= 1 && ch.n <= max_rows && ch.dst_row >= 0 && ch.dst_row + ch.n <= bounds.ctx_rows &&
                            ch.src_row >= 0 &&
                            ch.src_row + ch.n <= (fresh ? (int64_t)bounds.n_fresh : bounds.pool_rows) &&
                            (fresh ? (k_new != nullptr && v_new != nullptr) : (L.pool_k[layer] != nullptr)) &&
                            (ch.kind != KVLINK_SEG_DOC || (ch.table >= 0 && ch.table < bounds.n_rope_rows));
            if (!ok) {
                atomicCAS(&g_copy_status, 0, kCopyStatusBadIndex);
                *abort_flag = 1;
            }
        }
#endif
        fence_mbar_init();
    }
    __syncthreads();
    if (*abort_flag) return;  // uniform: written before the barrier

    if (threadIdx.x < 32) {
        // ------------------------------------------------------------ producer
        if (threadIdx.x == 0) {
            int issued = 0;
            // one-layer launches: a group is one unit, and the next unit's entry is loaded while
            // this one waits for its stage
            CopyChunk ch_next{};
            if (MAXL == 1 && c_begin < c_end) ch_next = chunks[c_begin];
            for (int c = c_begin, g = 0; c < c_end; ++g) {
                const int layer = layer_of(c);
                const CopyChunk ch = MAXL == 1 ? ch_next : chunks[c - layer * n_chunks];
                if (MAXL == 1 && c + 1 < c_end) ch_next = chunks[c + 1];
                const int st = g % CopySmem<WV>::NST;
                if (!copy_wait(empty + st, ((g / CopySmem<WV>::NST) & 1) ^ 1, abort_flag)) break;
                const bool fresh = ch.kind == KVLINK_SEG_LINK || ch.kind == KVLINK_SEG_QUESTION;
                const __nv_bfloat16* sk = (fresh ? k_new : L.pool_k[layer]) + ch.src_row * row_elems;
                const __nv_bfloat16* sv = WV ? (fresh ? v_new : L.pool_v[layer]) + ch.src_row * row_elems : nullptr;
                const uint32_t bytes = (uint32_t)ch.n * row_bytes;
                uint8_t* stage = smem + st * CopySmem<WV>::STAGE;
                mbar_arrive_expect_tx(full + st, WV ? 2 * bytes : bytes);
                bulk_load(stage, sk, bytes, full + st);
                if (WV) bulk_load(stage + kCopyStageBytes, sv, bytes, full + st);
                issued = g + 1;
                c = MAXL == 1 ? c + 1 : group_end(c, layer, ch);
            }
            // no load may still be in flight when the CTA leaves
            for (int i = issued - CopySmem<WV>::NST > 0 ? issued - CopySmem<WV>::NST : 0; i < issued; ++i)
                copy_drain(full + i % CopySmem<WV>::NST, (i / CopySmem<WV>::NST) & 1);
        }
        return;
    }

    // ---------------------------------------------------------------- consumers
    const int tc = threadIdx.x - 32;
    constexpr int UPH = D / 16;                // (lo, hi) chunk pairs per head
    const int U = h_kv * UPH;                  // pairs per token, a power of two <= 128
    const int TPP = kCopyConsumers / U;        // tokens per pass
    const int unit = tc % U;
    const int tok0 = tc / U;
    const int head = unit / UPH;
    const int j0 = (unit % UPH) * 8;
    const uint32_t lo_off = (uint32_t)(head * D + j0) * 2;
    int cur_table = -1;
    float4 cs[8];
    // one-layer launches: a group is one unit (consecutive units never read the same rows), and
    // the next unit's entry is loaded a group ahead, so its latency overlaps this group's work
    CopyChunk ch_next{};
    if (MAXL == 1 && c_begin < c_end) ch_next = chunks[c_begin];
    for (int c = c_begin, g = 0; c < c_end; ++g) {
        const int layer = layer_of(c);
        const CopyChunk ch0 = MAXL == 1 ? ch_next : chunks[c - layer * n_chunks];
        if (MAXL == 1 && c + 1 < c_end) ch_next = chunks[c + 1];
        const int c1 = MAXL == 1 ? c + 1 : group_end(c, layer, ch0);
        const int st = g % CopySmem<WV>::NST;
        const bool loaded = copy_wait(full + st, (g / CopySmem<WV>::NST) & 1, abort_flag);
        // Every consumer is done with the previous group, and all of them take one decision:
        // the producer may raise the abort flag at any moment (its own wait ran out), so each
        // consumer's read of the flag could differ; the barrier ORs them, so either all 128
        // leave the loop or none does, and no consumer is left waiting at the next barrier.
        if (named_bar_any(1, kCopyConsumers, !loaded || *abort_flag != 0)) break;
        const uint8_t* stage = smem + st * CopySmem<WV>::STAGE;
        const uint32_t bytes = (uint32_t)ch0.n * row_bytes;
        for (int cc = c; cc < c1; ++cc) {
            const CopyChunk ch = MAXL == 1 ? ch0 : chunks[cc - layer * n_chunks];
            if (ch.kind == KVLINK_SEG_DOC) {
                if (ch.table != cur_table) {
                    const float4* t = rope + (int64_t)ch.table * (D / 2) + j0;
#pragma unroll
                    for (int q = 0; q < 8; ++q) cs[q] = __ldg(t + q);
                    cur_table = ch.table;
                }
                uint8_t* dst = reinterpret_cast<uint8_t*>(L.cache_k[layer] + ch.dst_row * row_elems) + lo_off;
                for (int t = tok0; t < ch.n; t += TPP) {
                    const uint8_t* src = stage + (uint32_t)t * row_bytes + lo_off;
                    uint4 a = *reinterpret_cast<const uint4*>(src);
                    uint4 b = *reinterpret_cast<const uint4*>(src + D);
                    rotate8<!WV>(a, b, cs);
                    uint8_t* d = dst + (size_t)t * row_bytes;
                    *reinterpret_cast<uint4*>(d) = a;
                    *reinterpret_cast<uint4*>(d + D) = b;
                }
            } else if (tc == 0) {
                bulk_store(L.cache_k[layer] + ch.dst_row * row_elems, stage, bytes);
            }
            if (WV && tc == 0) bulk_store(L.cache_v[layer] + ch.dst_row * row_elems, stage + kCopyStageBytes, bytes);
        }
        if (tc == 0) {
            bulk_commit();
            bulk_wait_read<1>();  // the previous group's stores have read their stage
            if (g > 0) mbar_arrive(empty + (g - 1) % CopySmem<WV>::NST);
        }
        c = c1;
    }
    if (tc == 0) bulk_wait<0>();
}

template <int D, int MAXL, bool WV>
static void launch_reencode_wv(const CopyChunk* ch, int n_chunks, int n_layers, const float4* rope, int h_kv,
                               int num_sms, const LayerPtrs<MAXL>& L, const void* k_new, const void* v_new,
                               const CopyBounds& bounds, cudaStream_t stream) {
    // a failure here surfaces as the launch error, which the caller checks
    static std::atomic<uint64_t> attr{0};
    once_per_device(attr, [] {
        return cudaFuncSetAttribute(reencode_kernel<D, MAXL, WV>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)CopySmem<WV>::BYTES);
    });
    const int64_t n_units = (int64_t)n_chunks * n_layers;
    const int grid = n_units < num_sms ? (int)n_units : num_sms;
    reencode_kernel<D, MAXL, WV><<<grid, kCopyThreads, CopySmem<WV>::BYTES, stream>>>(
        ch, n_chunks, n_layers, rope, h_kv, L, (const __nv_bfloat16*)k_new, (const __nv_bfloat16*)v_new, bounds);
}

// values copied when the linked cache has value rows (every layer's, or none: zero-copy values)
template <int D, int MAXL>
static void launch_reencode_t(const CopyChunk* ch, int n_chunks, int n_layers, const float4* rope, int h_kv,
                              int num_sms, const LayerPtrs<MAXL>& L, const void* k_new, const void* v_new,
                              const CopyBounds& bounds, cudaStream_t stream) {
    if (L.cache_v[0] != nullptr)
        launch_reencode_wv<D, MAXL, true>(ch, n_chunks, n_layers, rope, h_kv, num_sms, L, k_new, v_new, bounds, stream);
    else
        launch_reencode_wv<D, MAXL, false>(ch, n_chunks, n_layers, rope, h_kv, num_sms, L, k_new, v_new, bounds,
                                           stream);
}

void launch_reencode(const DevicePlan& P, int chunk_base, int n_chunks, int head_dim, int h_kv, int num_sms,
                     const void* pool_k, const void* pool_v, const void* k_new, const void* v_new, void* cache_k,
                     void* cache_v, cudaStream_t stream) {
    if (n_chunks <= 0) return;
    using bf = __nv_bfloat16;
    LayerPtrs<1> L{{(const bf*)pool_k}, {(const bf*)pool_v}, {(bf*)cache_k}, {(bf*)cache_v}};
    const CopyChunk* ch = P.chunks + chunk_base;
    const CopyBounds bounds{P.ctx_rows, P.pool_rows, P.n_fresh, P.n_rope_rows};
    if (head_dim == 128)
        launch_reencode_t<128, 1>(ch, n_chunks, 1, P.rope, h_kv, num_sms, L, k_new, v_new, bounds, stream);
    else
        launch_reencode_t<64, 1>(ch, n_chunks, 1, P.rope, h_kv, num_sms, L, k_new, v_new, bounds, stream);
}

// The document chunks (sorted by source) of n_layers layers, kMaxLayersPerLaunch layers per launch.
void launch_reencode_layers(const DevicePlan& P, int n_chunks, int head_dim, int h_kv, int num_sms, int n_layers,
                            const void* const* pool_k, const void* const* pool_v, void* const* cache_k,
                            void* const* cache_v, cudaStream_t stream) {
    if (n_chunks <= 0) return;
    using bf = __nv_bfloat16;
    // unit indices stay below 2^31
    const int per_launch = (int)std::min<int64_t>(kMaxLayersPerLaunch, INT32_MAX / n_chunks);
    for (int l0 = 0; l0 < n_layers; l0 += per_launch) {
        const int nl = std::min(n_layers - l0, per_launch);
        LayerPtrs<kMaxLayersPerLaunch> L{};
        for (int l = 0; l < nl; ++l) {
            L.pool_k[l] = (const bf*)pool_k[l0 + l];
            L.pool_v[l] = (const bf*)pool_v[l0 + l];
            L.cache_k[l] = (bf*)cache_k[l0 + l];
            L.cache_v[l] = (bf*)cache_v[l0 + l];
        }
        const CopyBounds bounds{P.ctx_rows, P.pool_rows, P.n_fresh, P.n_rope_rows};
        if (head_dim == 128)
            launch_reencode_t<128, kMaxLayersPerLaunch>(P.chunks_sorted, n_chunks, nl, P.rope, h_kv, num_sms, L,
                                                        nullptr, nullptr, bounds, stream);
        else
            launch_reencode_t<64, kMaxLayersPerLaunch>(P.chunks_sorted, n_chunks, nl, P.rope, h_kv, num_sms, L,
                                                       nullptr, nullptr, bounds, stream);
    }
}

// --------------------------------------------------------------------------
// A3 with the document caches in host memory (Sec. 3.3: the caches start in CPU memory and
// are loaded for every request).  On GB300 the SMs reach page-locked Grace memory over
// NVLink-C2C, so the rows are loaded straight from the host pool by the re-encode itself
// and written once, rotated, to the linked cache in HBM: no staging copy.  Plain 16-byte
// loads (the bulk-copy path of reencode_kernel is kept to device memory).  One warp per
// work unit at a time; a lane owns (head, j0) pairs of the row (elements j0..j0+7 and
// j0+D/2..j0+D/2+7 of one head) and issues the loads of two token rows before any store, so
// each lane keeps eight 16-byte host loads in flight.  The rotation is the one of
// reencode_kernel (rotate8), so the cache bits are identical.
// --------------------------------------------------------------------------
constexpr int kHostWarps = 8;
constexpr int kHostPairsPerLane = 2;        // rows of up to 64 pairs (the 8B shape) in one pass

template <int D>
__global__ void __launch_bounds__(32 * kHostWarps) reencode_host_kernel(
    const CopyChunk* __restrict__ chunks, int n_chunks, const float4* __restrict__ rope, int h_kv,
    const uint4* __restrict__ pool_k, const uint4* __restrict__ pool_v, uint4* __restrict__ cache_k,
    uint4* __restrict__ cache_v, const CopyBounds bounds) {
    if (*reinterpret_cast<volatile int32_t*>(&g_copy_status) != 0) return;   // a recorded failure
    constexpr int PAIRS_PER_HEAD = D / 16;
    constexpr int PAIRS_PER_PASS = 32 * kHostPairsPerLane;
    const int U = h_kv * PAIRS_PER_HEAD;              // (lo, hi) pairs of 16-byte words per row
    const int row_vec = h_kv * D / 8;                 // 16-byte words per row
    const int lane = threadIdx.x % 32;
    // CTA b walks the contiguous range [n*b/grid, n*(b+1)/grid) of the units sorted by source
    // row, its warps on neighbouring units: the host rows in flight at any time lie in a few
    // short runs per CTA instead of all over the pool
    const int c_begin = (int)((int64_t)n_chunks * blockIdx.x / gridDim.x);
    const int c_end = (int)((int64_t)n_chunks * (blockIdx.x + 1) / gridDim.x);
    for (int c = c_begin + (int)threadIdx.x / 32; c < c_end; c += kHostWarps) {
        const CopyChunk ch = chunks[c];
#ifdef KVLINK_DEBUG_CHECKS
        if (ch.n < 1 || ch.dst_row < 0 || ch.dst_row + ch.n > bounds.ctx_rows || ch.src_row < 0 ||
            ch.src_row + ch.n > bounds.pool_rows ||
            (ch.kind == KVLINK_SEG_DOC && (ch.table < 0 || ch.table >= bounds.n_rope_rows))) {
            if (lane == 0) atomicCAS(&g_copy_status, 0, kCopyStatusBadIndex);
            continue;
        }
#endif
        const bool rot = ch.kind == KVLINK_SEG_DOC;
        for (int p0 = 0; p0 < U; p0 += PAIRS_PER_PASS) {     // one pass for rows of <= 64 pairs
            int lo_idx[kHostPairsPerLane];
            bool has[kHostPairsPerLane];
            float4 cs[kHostPairsPerLane][8];
#pragma unroll
            for (int i = 0; i < kHostPairsPerLane; ++i) {
                const int p = p0 + lane + 32 * i;
                has[i] = p < U;
                lo_idx[i] = (p / PAIRS_PER_HEAD) * (D / 8) + p % PAIRS_PER_HEAD;
                if (rot && has[i]) {
                    const float4* t = rope + (int64_t)ch.table * (D / 2) + (p % PAIRS_PER_HEAD) * 8;
#pragma unroll
                    for (int q = 0; q < 8; ++q) cs[i][q] = __ldg(t + q);
                }
            }
            for (int t0 = 0; t0 < ch.n; t0 += 2) {
                uint4 k[2][kHostPairsPerLane][2], v[2][kHostPairsPerLane][2];
#pragma unroll
                for (int u = 0; u < 2; ++u) {
                    const int64_t src = (ch.src_row + t0 + u) * row_vec;
#pragma unroll
                    for (int i = 0; i < kHostPairsPerLane; ++i)
                        if (has[i] && t0 + u < ch.n) {
                            k[u][i][0] = pool_k[src + lo_idx[i]];
                            k[u][i][1] = pool_k[src + lo_idx[i] + D / 16];
                            v[u][i][0] = pool_v[src + lo_idx[i]];
                            v[u][i][1] = pool_v[src + lo_idx[i] + D / 16];
                        }
                }
#pragma unroll
                for (int u = 0; u < 2; ++u) {
                    const int64_t dst = (ch.dst_row + t0 + u) * row_vec;
#pragma unroll
                    for (int i = 0; i < kHostPairsPerLane; ++i)
                        if (has[i] && t0 + u < ch.n) {
                            if (rot) rotate8<false>(k[u][i][0], k[u][i][1], cs[i]);
                            cache_k[dst + lo_idx[i]] = k[u][i][0];
                            cache_k[dst + lo_idx[i] + D / 16] = k[u][i][1];
                            cache_v[dst + lo_idx[i]] = v[u][i][0];
                            cache_v[dst + lo_idx[i] + D / 16] = v[u][i][1];
                        }
                }
            }
        }
    }
}

// The cached chunks of one layer from a device-accessible host pool.
void launch_reencode_host(const DevicePlan& P, int n_chunks, int head_dim, int h_kv, int num_sms,
                          const void* pool_k, const void* pool_v, void* cache_k, void* cache_v, cudaStream_t stream) {
    if (n_chunks <= 0) return;
    const CopyBounds bounds{P.ctx_rows, P.pool_rows, P.n_fresh, P.n_rope_rows};
    const int grid = std::max(1, std::min((n_chunks + kHostWarps - 1) / kHostWarps, 2 * num_sms));
    // the cached units sorted by source row (the same set as the plan's cached units)
    if (head_dim == 128)
        reencode_host_kernel<128><<<grid, 32 * kHostWarps, 0, stream>>>(
            P.chunks_sorted, n_chunks, P.rope, h_kv, (const uint4*)pool_k, (const uint4*)pool_v, (uint4*)cache_k,
            (uint4*)cache_v, bounds);
    else
        reencode_host_kernel<64><<<grid, 32 * kHostWarps, 0, stream>>>(
            P.chunks_sorted, n_chunks, P.rope, h_kv, (const uint4*)pool_k, (const uint4*)pool_v, (uint4*)cache_k,
            (uint4*)cache_v, bounds);
}

// --------------------------------------------------------------------------
// A4: the fresh link/question rows to their cache rows (bit copies).  A few MB per layer
// on the path of the attention that follows, so the copy is built for latency: one warp
// per row and 16-byte accesses, all of a lane's loads issued before its stores.
// --------------------------------------------------------------------------
constexpr int kPlaceWarps = 8;

__global__ void __launch_bounds__(32 * kPlaceWarps) place_fresh_kernel(const int32_t* __restrict__ fresh_dst,
                                                                       int n_fresh, int64_t ctx_rows, int row_vec,
                                                                       const uint4* __restrict__ k_new,
                                                                       const uint4* __restrict__ v_new,
                                                                       uint4* __restrict__ cache_k,
                                                                       uint4* __restrict__ cache_v) {
    // the attention launched after this kernel may start its prologue now (it waits for this
    // kernel's writes before reading them)
    asm volatile("griddepcontrol.launch_dependents;");
    // after a recorded failure, later launches skip their work
    if (*reinterpret_cast<volatile int32_t*>(&g_copy_status) != 0) return;
    const int row = blockIdx.x * kPlaceWarps + threadIdx.x / 32, lane = threadIdx.x % 32;
    if (row >= n_fresh) return;
#ifdef KVLINK_DEBUG_CHECKS
    if (fresh_dst[row] < 0 || fresh_dst[row] >= ctx_rows) {
        if (lane == 0) atomicCAS(&g_copy_status, 0, kCopyStatusBadIndex);
        return;
    }
#endif
    const int64_t src = (int64_t)row * row_vec, dst = (int64_t)fresh_dst[row] * row_vec;
    const bool with_v = cache_v != nullptr;   // NULL: zero-copy values (the attention reads v_new)
    for (int i0 = lane; i0 < row_vec; i0 += 4 * 32) {
        uint4 k[4], v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int i = i0 + u * 32;
            if (i < row_vec) {
                k[u] = __ldg(k_new + src + i);
                if (with_v) v[u] = __ldg(v_new + src + i);
            }
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int i = i0 + u * 32;
            if (i < row_vec) {
                cache_k[dst + i] = k[u];
                if (with_v) cache_v[dst + i] = v[u];
            }
        }
    }
}

void launch_place_fresh(const int32_t* d_fresh_dst, int n_fresh, int64_t ctx_rows, int row_bytes, const void* k_new,
                        const void* v_new, void* cache_k, void* cache_v, cudaStream_t stream) {
    if (n_fresh <= 0) return;
    const int blocks = (n_fresh + kPlaceWarps - 1) / kPlaceWarps;
    place_fresh_kernel<<<blocks, 32 * kPlaceWarps, 0, stream>>>(d_fresh_dst, n_fresh, ctx_rows, row_bytes / 16,
                                                                (const uint4*)k_new, (const uint4*)v_new,
                                                                (uint4*)cache_k, (uint4*)cache_v);
}

// --------------------------------------------------------------------------
// RoPE of the fresh rows at their global positions (Sec. 2.2: a token at position i
// carries R_i).  One thread per (fresh row, j < D/2): the angle pos * theta^(-2j/D) is
// formed in float64, cos/sin are split into float pairs, and pair (j, j + D/2) of every
// query head and KV head of the row is rotated in place with the compensated products
// of the re-encode, so each output is within one bf16 ulp of the fp64 rotation.
// --------------------------------------------------------------------------
__global__ void rope_fresh_kernel(const int32_t* __restrict__ fresh_pos, int n_fresh, int head_dim, double theta,
                                  __nv_bfloat16* __restrict__ q, int h_q, __nv_bfloat16* __restrict__ k, int h_kv) {
    const int half = head_dim / 2;
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= (int64_t)n_fresh * half) return;
    const int r = (int)(i / half), j = (int)(i % half);
    const double angle = (double)fresh_pos[r] * pow(theta, -2.0 * (double)j / (double)head_dim);
    double sn, cs;
    sincos(angle, &sn, &cs);
    const float ch = (float)cs, cl = (float)(cs - (double)ch), sh = (float)sn, sl = (float)(sn - (double)sh);
    auto rot = [&](__nv_bfloat16* row) {
        const float x = __bfloat162float(row[j]), y = __bfloat162float(row[j + half]);
        row[j] = __float2bfloat16_rn(rot_first(x, y, ch, cl, sh, sl));
        row[j + half] = __float2bfloat16_rn(rot_second(x, y, ch, cl, sh, sl));
    };
    for (int h = 0; h < h_q; ++h) rot(q + ((int64_t)r * h_q + h) * head_dim);
    for (int h = 0; h < h_kv; ++h) rot(k + ((int64_t)r * h_kv + h) * head_dim);
}

void launch_rope_fresh(const int32_t* d_fresh_pos, int n_fresh, int head_dim, double theta, void* q, int h_q,
                       void* k, int h_kv, cudaStream_t stream) {
    const int64_t n = (int64_t)n_fresh * (head_dim / 2);
    if (n == 0) return;
    const int threads = 256;
    rope_fresh_kernel<<<(unsigned)((n + threads - 1) / threads), threads, 0, stream>>>(
        d_fresh_pos, n_fresh, head_dim, theta, (__nv_bfloat16*)q, h_q, (__nv_bfloat16*)k, h_kv);
}

int read_copy_status(int32_t* status) {
    return cudaMemcpyFromSymbol(status, g_copy_status, sizeof(int32_t)) == cudaSuccess ? KVLINK_OK : KVLINK_ECUDA;
}

int clear_copy_status() {
    const int32_t z = 0;
    return cudaMemcpyToSymbol(g_copy_status, &z, sizeof(int32_t)) == cudaSuccess ? KVLINK_OK : KVLINK_ECUDA;
}

}  // namespace kvlink
