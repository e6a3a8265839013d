// Suffix attention on the tcgen05 tensor cores (Sec. 2.3, "inference").
//
// Work item = one M-tile of up to 128 rows (up to 128/G fresh tokens x the G
// query heads that share one KV head) of one query, over a range of 128-key
// tiles of that query's linked cache (cache-row order; in the links-at-end layout the
// cached rows and the fresh rows at the end form two runs).  Rows are (token, head)
// pairs, so the G heads of a GQA group share every K/V tile load.
//
// Warp roles (256 threads, one CTA per SM, 512 TMEM columns):
//   warps 0-3  softmax + epilogue; thread r owns row r = TMEM lane r
//   warp 4     TMA: Q once, then K tiles into an NK-stage ring
//   warp 5     TMEM allocation and the thread issuing the S = Q K^T MMAs
//   warp 6     TMA: V tiles into an NV-stage ring
//   warp 7     the thread issuing the O += P V MMAs
// Per KV tile j (TMEM: three S/P buffers of 128 columns, then O):
//   S_j = Q K_j^T           tcgen05.mma SMEM x SMEM -> S buffer j%3
//   P_j = exp2(S_j c - m)   softmax warps: TMEM -> registers -> bf16 P written back
//                           over the first 64 columns of the same buffer
//   O  += P_j V_j           tcgen05.mma TMEM x SMEM (P from TMEM, V read MN-major)
// S_j is issued only after PV_{j-3} has finished reading the buffer, so up to
// three tiles are in flight and the softmax never waits on a PV except to
// rescale O.  S and PV come from two issuing threads (see mma_s_role).  The running max m is raised only when it grows by more than 2^8,
// so that rescale is rare.  The mask keeps the cache rows holding positions up to
// the row's own (a threshold pair per row, see softmax_role) and is evaluated only on
// tiles that reach past the rows every row of the tile sees.  Items whose KV range was split write
// unnormalised partials (O, m, l) to the workspace; attn_merge_kernel combines them.
//
// Every mbarrier wait is bounded in time.  On expiry the kernel records
// kAttnStatusWaitTimeout in its status word, the other roles leave their loops,
// the producer and MMA threads wait (bounded) for their own in-flight copies and
// MMAs, TMEM is freed and the CTA returns.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include "kvlink_attention_common.cuh"
#include "kvlink_internal.h"
#include "kvlink_sm100.cuh"

namespace kvlink {
using namespace sm100;

static __device__ int32_t g_attn_status;

constexpr int kTcThreads = 256;
constexpr int kPvWarp = 7;
constexpr int kSoftmaxWarps = 4;
constexpr int kTmaKWarp = 4;
constexpr int kMmaWarp = 5;
constexpr int kTmaVWarp = 6;


template <int D, int G>
__global__ void __launch_bounds__(kTcThreads, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                   const __grid_constant__ CUtensorMap tm_v, DevicePlan P, __nv_bfloat16* __restrict__ out,
                   float* __restrict__ ws, int h_q, float scale_log2) {
    using C = TcCfg<D>;
    constexpr int NK = C::NK, NV = C::NV, NB = C::NB;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw_addr = smem_u32(smem_raw);
    uint8_t* smem = smem_raw + ((1024u - (raw_addr & 1023u)) & 1023u);

    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);
    uint64_t* bar_q_full = bars;
    uint64_t* bar_k_full = bar_q_full + 1;
    uint64_t* bar_k_empty = bar_k_full + NK;
    uint64_t* bar_v_full = bar_k_empty + NK;
    uint64_t* bar_v_empty = bar_v_full + NV;
    uint64_t* bar_s_full = bar_v_empty + NV;
    uint64_t* bar_p_full = bar_s_full + NB;
    uint64_t* bar_o_done = bar_p_full + NB;
    uint64_t* bar_drain = bar_o_done + NB;
    uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(bars + C::N_BARS);
    volatile int32_t* abort_flag = reinterpret_cast<volatile int32_t*>(tmem_holder + 1);

    const AttnItem it = P.items[blockIdx.x];
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int n_tiles = it.kv_tile1 - it.kv_tile0;

    if (threadIdx.x == 0) {
        for (int i = 0; i < C::N_BARS; ++i) {
            const bool p_full = bars + i >= bar_p_full && bars + i < bar_p_full + NB;
            mbar_init(bars + i, p_full ? kSoftmaxWarps : 1);
        }
        // after a recorded failure, later launches skip their work instead of waiting out their bounds
        *abort_flag = *reinterpret_cast<volatile int32_t*>(&g_attn_status) != 0 ? 1 : 0;
#ifdef KVLINK_DEBUG_CHECKS
        if (!*abort_flag && !item_in_bounds(it, P)) {
            atomicCAS(&g_attn_status, 0, kAttnStatusBadIndex);
            *abort_flag = 1;
        }
#endif
        fence_mbar_init();
    }
    if (warp == kMmaWarp) {
        tmem_alloc(tmem_holder, kTmemCols);
        tmem_relinquish();
    }
    if (warp == kTmaKWarp && lane == 0) {
        prefetch_tensormap(&tm_q);
        prefetch_tensormap(&tm_k);
        prefetch_tensormap(&tm_v);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_holder;
    const bool skip = *abort_flag != 0;  // written before the barrier: uniform across the CTA
    const int ctx0 = skip ? 0 : (int)P.cu_ctx[it.query];

    if (skip) {
        // nothing issued: fall through to the teardown
    } else if (warp == kTmaKWarp) {
        // ------------------------------------------------------------ Q, then the K ring
        if (lane == 0) {
            const int q_row0 = P.cu_fresh[it.query] + it.tok0;
            mbar_arrive_expect_tx(bar_q_full, C::Q_BYTES);
#pragma unroll
            for (int a = 0; a < C::ATOMS; ++a)
                tma_load_3d(smem + C::OFF_Q + a * C::ATOM_BYTES, &tm_q, a * 64, it.kv_head * G, q_row0, bar_q_full);
            produce_ring<NK, C::ATOMS>(smem + C::OFF_K, C::KV_BYTES, &tm_k, bar_k_full, bar_k_empty, n_tiles, it,
                                       ctx0, abort_flag, &g_attn_status);
            drain_bar(bar_q_full, 0, &g_attn_status);
        }
    } else if (warp == kTmaVWarp) {
        // ------------------------------------------------------------ the V ring
        if (lane == 0)
            produce_ring<NV, C::ATOMS>(smem + C::OFF_V, C::KV_BYTES, &tm_v, bar_v_full, bar_v_empty, n_tiles, it,
                                       ctx0, abort_flag, &g_attn_status);
    } else if (warp == kMmaWarp) {
        if (lane == 0)
            mma_s_role<D, NK, NB>(smem, C::OFF_Q, C::OFF_K, C::KV_BYTES, C::ATOM_BYTES, tmem + C::TMEM_S, n_tiles,
                                  bar_q_full, bar_k_full, bar_k_empty, bar_s_full, bar_o_done, bar_drain, abort_flag,
                                  &g_attn_status);
    } else if (warp == kPvWarp) {
        if (lane == 0)
            mma_pv_role<D, NV, NB>(smem, C::OFF_V, C::KV_BYTES, C::ATOM_BYTES, tmem + C::TMEM_S, tmem + C::TMEM_O,
                                   n_tiles, bar_v_full, bar_v_empty, bar_p_full, bar_o_done, bar_drain + 1,
                                   abort_flag, &g_attn_status);
    } else {
        // ------------------------------------------------------------ softmax + epilogue (warps 0-3)
        softmax_role<D, G, NB>(it, P, tmem + C::TMEM_S, tmem + C::TMEM_O, n_tiles, bar_s_full, bar_p_full,
                               bar_o_done, abort_flag, &g_attn_status, out, ws, h_q, scale_log2);
    }

    tc_fence_before();
    __syncthreads();
    if (warp == kMmaWarp) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

// Combine the partial results of split KV ranges: O = sum_s O_s 2^(m_s - M) / sum_s l_s 2^(m_s - M).
template <int D>
__global__ void __launch_bounds__(256) attn_merge_kernel(DevicePlan P, const float* __restrict__ ws,
                                                         __nv_bfloat16* __restrict__ out, int h_q, int G) {
    const MergeGroup mg = P.merges[blockIdx.x];
#ifdef KVLINK_DEBUG_CHECKS
    if (mg.query < 0 || mg.query >= P.batch || mg.kv_head < 0 || mg.kv_head >= P.h_kv || mg.tok0 < 0 ||
        mg.tok1 < mg.tok0 || mg.tok1 > P.cu_fresh[mg.query + 1] - P.cu_fresh[mg.query] || mg.slot0 < 0 ||
        mg.n_split < 1 || mg.slot0 + mg.n_split > P.n_slots) {
        if (threadIdx.x == 0) atomicCAS(&g_attn_status, 0, kAttnStatusBadIndex);
        return;
    }
#endif
    const int n_rows = (mg.tok1 - mg.tok0) * G;
    const int f0 = P.cu_fresh[mg.query];
    const int64_t slot_floats = (int64_t)kAttnBM * (D + 2);
    for (int idx = threadIdx.x; idx < n_rows * D; idx += blockDim.x) {
        const int r = idx / D, d = idx % D;
        float M = -INFINITY;
        for (int s = 0; s < mg.n_split; ++s) M = fmaxf(M, ws[(mg.slot0 + s) * slot_floats + kAttnBM * D + r]);
        float L = 0.f, O = 0.f;
        for (int s = 0; s < mg.n_split; ++s) {
            const float* w = ws + (mg.slot0 + s) * slot_floats;
            const float ms = w[kAttnBM * D + r];
            const float f = (ms == -INFINITY) ? 0.f : ex2_approx(ms - M);
            L += w[kAttnBM * D + kAttnBM + r] * f;
            O += w[r * D + d] * f;
        }
        const int frow = f0 + mg.tok0 + r / G;
        out[((int64_t)frow * h_q + mg.kv_head * G + (r % G)) * D + d] = __float2bfloat16_rn(O / L);
    }
}

// ------------------------------------------------------------------ host side

static PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    }
    return fn;
}

// bf16 tensor [d2][d1][d0] (d0 contiguous), box {b0, b1, b2}, 128-byte swizzle
bool make_map_3d(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1, uint64_t d2, uint32_t b0,
                        uint32_t b1, uint32_t b2) {
    auto fn = encode_fn();
    if (!fn) return false;
    const cuuint64_t dims[3] = {d0, d1, d2};
    const cuuint64_t strides[2] = {d0 * 2, d0 * d1 * 2};
    const cuuint32_t box[3] = {b0, b1, b2};
    const cuuint32_t es[3] = {1, 1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, es,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int D, int G>
static cudaError_t launch_tc_dg(const CUtensorMap& mq, const CUtensorMap& mk, const CUtensorMap& mv,
                                const DevicePlan& P, int n_items, int n_merges, void* out, float* ws, int h_q,
                                float scale_log2, cudaStream_t stream) {
    using C = TcCfg<D>;
    static std::atomic<uint64_t> attr_set{0};
    cudaError_t ea = once_per_device(attr_set, [] {
        return cudaFuncSetAttribute(attn_tc_kernel<D, G>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)C::SMEM_BYTES);
    });
    if (ea != cudaSuccess) return ea;
    if (n_items > 0)
        attn_tc_kernel<D, G><<<n_items, kTcThreads, C::SMEM_BYTES, stream>>>(
            mq, mk, mv, P, (__nv_bfloat16*)out, ws, h_q, scale_log2);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    if (n_merges > 0) attn_merge_kernel<D><<<n_merges, 256, 0, stream>>>(P, ws, (__nv_bfloat16*)out, h_q, G);
    return cudaGetLastError();
}

// Merge launch shared with the fused kernel: one CTA per merge group.
cudaError_t launch_attn_merge(const DevicePlan& P, int n_merges, const float* ws, void* out, int h_q, int G,
                              int head_dim, cudaStream_t stream) {
    if (n_merges <= 0) return cudaSuccess;
    if (head_dim == 128)
        attn_merge_kernel<128><<<n_merges, 256, 0, stream>>>(P, ws, (__nv_bfloat16*)out, h_q, G);
    else
        attn_merge_kernel<64><<<n_merges, 256, 0, stream>>>(P, ws, (__nv_bfloat16*)out, h_q, G);
    return cudaGetLastError();
}

// Returns 0, or KVLINK_ECUDA / KVLINK_EUNSUPPORTED.
int launch_attention_tc(const DevicePlan& P, int n_items, int n_merges, int n_fresh, int64_t ctx_rows,
                        int head_dim, int h_q, int h_kv, const void* q, const void* cache_k, const void* cache_v,
                        void* out, void* ws, cudaStream_t stream, cudaError_t* err) {
    const int G = h_q / h_kv;
    CUtensorMap mq, mk, mv;
    const uint32_t box_tok = (uint32_t)(kAttnBM / G);
    if (!make_map_3d(&mq, q, (uint64_t)head_dim, (uint64_t)h_q, (uint64_t)n_fresh, 64, (uint32_t)G, box_tok) ||
        !make_map_3d(&mk, cache_k, (uint64_t)head_dim, (uint64_t)h_kv, (uint64_t)ctx_rows, 64, 1, kAttnBN) ||
        !make_map_3d(&mv, cache_v, (uint64_t)head_dim, (uint64_t)h_kv, (uint64_t)ctx_rows, 64, 1, kAttnBN))
        return KVLINK_EUNSUPPORTED;
    const float sl2 = 1.4426950408889634f / sqrtf((float)head_dim);
    float* w = (float*)ws;
    cudaError_t e = cudaErrorInvalidValue;
#define KVLINK_TC_CASE(DD, GG)                                                                         \
    if (head_dim == DD && G == GG) e = launch_tc_dg<DD, GG>(mq, mk, mv, P, n_items, n_merges, out, w, h_q, sl2, \
                                                            stream);
    KVLINK_TC_CASE(128, 1) KVLINK_TC_CASE(128, 2) KVLINK_TC_CASE(128, 4) KVLINK_TC_CASE(128, 8)
    KVLINK_TC_CASE(128, 16) KVLINK_TC_CASE(64, 1) KVLINK_TC_CASE(64, 2) KVLINK_TC_CASE(64, 4)
    KVLINK_TC_CASE(64, 8) KVLINK_TC_CASE(64, 16)
#undef KVLINK_TC_CASE
    if (e != cudaSuccess) {
        *err = e;
        return KVLINK_ECUDA;
    }
    return KVLINK_OK;
}

// Failure-path self-test: one thread waits, through the kernels' bounded wait, on an
// mbarrier that nothing arrives at.  The wait runs out after limit_ns and records
// kAttnStatusWaitTimeout in the attention status word, exactly as a stalled pipeline would.
__global__ void wait_selftest_kernel(uint64_t limit_ns) {
    __shared__ __align__(8) uint64_t bar;
    __shared__ int32_t abort_flag;
    if (threadIdx.x != 0) return;
    mbar_init(&bar, 1);
    abort_flag = 0;
    fence_mbar_init();
    wait_bar(&bar, 0, &abort_flag, &g_attn_status, limit_ns);
}

int launch_wait_selftest(uint32_t limit_ms, cudaStream_t stream) {
    wait_selftest_kernel<<<1, 32, 0, stream>>>((uint64_t)limit_ms * 1000000ull);
    return cudaGetLastError() == cudaSuccess ? KVLINK_OK : KVLINK_ECUDA;
}

int read_attention_status(int32_t* status) {
    return cudaMemcpyFromSymbol(status, g_attn_status, sizeof(int32_t)) == cudaSuccess ? KVLINK_OK : KVLINK_ECUDA;
}

int clear_attention_status() {
    const int32_t z = 0;
    return cudaMemcpyToSymbol(g_attn_status, &z, sizeof(int32_t)) == cudaSuccess ? KVLINK_OK : KVLINK_ECUDA;
}

}  // namespace kvlink
