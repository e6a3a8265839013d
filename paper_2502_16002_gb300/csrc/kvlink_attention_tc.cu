// Suffix attention on the tcgen05 tensor cores (Sec. 2.3, "inference").
//
// Work item = one M-tile of 128 rows (128/G fresh tokens x the G query heads
// that share one KV head) of one query, over a range of 128-key tiles of that
// query's linked cache.  Rows are (token, head) pairs, so the G heads of a
// GQA group share every K/V tile load.
//
// Warp roles (192 threads, one CTA per SM, 512 TMEM columns):
//   warps 0-3  softmax + epilogue; thread r owns row r = TMEM lane r
//   warp 4     TMA producer: Q once, then K and V tiles into an NS-stage ring
//   warp 5     TMEM allocation and the single MMA-issuing thread
// Per KV tile j:
//   S_j = Q K_j^T          tcgen05.mma, SMEM x SMEM -> TMEM (double-buffered S)
//   P_j = exp2(S_j*c - m)  softmax warps: TMEM -> registers -> bf16 P in SMEM
//   O  += P_j V_j          tcgen05.mma, SMEM x SMEM -> TMEM (V read MN-major)
// The running max m is only raised when it grows by more than 2^8, so the O
// accumulator in TMEM is rescaled rarely; m, l stay per thread in registers.
// The mask keeps key slot j for a row at global position p iff j <= p, and is
// only evaluated on tiles that reach past the tile's smallest row position.
// Items whose KV range was split write unnormalised partials (O, m, l) to the
// workspace; attn_merge_kernel combines them.
//
// Every mbarrier wait is bounded in time.  On expiry the kernel records
// kAttnStatusWaitTimeout in its status word, the other roles leave their loops,
// the producer and MMA threads wait (bounded) for their own in-flight copies and
// MMAs, TMEM is freed and the CTA returns.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include "kvlink_internal.h"
#include "kvlink_sm100.cuh"

namespace kvlink {
using namespace sm100;

static __device__ int32_t g_attn_status;

constexpr int kTcThreads = 192;
constexpr int kSoftmaxWarps = 4;
constexpr int kTmaWarp = 4;
constexpr int kMmaWarp = 5;
constexpr uint32_t kTmemCols = 512;
constexpr uint64_t kWaitLimitNs = 2000000000ull;  // 2 s
constexpr int32_t kAttnStatusWaitTimeout = 0x41;
constexpr float kRescaleThreshold = 8.0f;         // log2 units: rescale O when the max grows by > 2^8

template <int D>
struct TcCfg {
    static constexpr int ATOMS = D / 64;                 // 128-byte swizzle atoms along head_dim
    static constexpr int NS = (D == 128) ? 2 : 4;        // K/V ring stages
    static constexpr uint32_t ATOM_BYTES = 128 * 128;    // [128 rows][64 bf16]
    static constexpr uint32_t Q_BYTES = ATOMS * ATOM_BYTES;
    static constexpr uint32_t KV_BYTES = ATOMS * ATOM_BYTES;
    static constexpr uint32_t P_BYTES = 2 * ATOM_BYTES;  // [128 rows][128 keys] bf16
    static constexpr uint32_t OFF_Q = 0;
    static constexpr uint32_t OFF_K = OFF_Q + Q_BYTES;
    static constexpr uint32_t OFF_V = OFF_K + NS * KV_BYTES;
    static constexpr uint32_t OFF_P = OFF_V + NS * KV_BYTES;
    static constexpr uint32_t OFF_BAR = OFF_P + P_BYTES;
    // q_full, k_full[NS], v_full[NS], kv_empty[NS], s_full[2], s_free[2], p_full, o_done, drain
    static constexpr int N_BARS = 1 + 3 * NS + 4 + 3;
    static constexpr uint32_t SMEM_BYTES = OFF_BAR + N_BARS * 8 + 16 + 1024;
    static constexpr uint32_t TMEM_S0 = 0, TMEM_S1 = 128, TMEM_O = 256;
};

// Wait for phase `parity` of `bar`; false if another role aborted or the time limit passed.
__device__ __forceinline__ bool wait_bar(uint64_t* bar, uint32_t parity, volatile int32_t* abort_flag) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = globaltimer_ns();
    while (true) {
        if (mbar_try_wait(bar, parity)) return true;
        if (*abort_flag) return false;
        if (globaltimer_ns() - t0 > kWaitLimitNs) {
            *abort_flag = 1;
            atomicCAS(&g_attn_status, 0, kAttnStatusWaitTimeout);
            return false;
        }
    }
}

// Same, but ignores the abort flag: used to drain this thread's own async work.
__device__ __forceinline__ void drain_bar(uint64_t* bar, uint32_t parity) {
    const uint64_t t0 = globaltimer_ns();
    while (!mbar_try_wait(bar, parity)) {
        if (globaltimer_ns() - t0 > kWaitLimitNs) {
            atomicCAS(&g_attn_status, 0, kAttnStatusWaitTimeout);
            return;
        }
    }
}

// All lanes wait; the warp proceeds only if every lane saw the phase complete.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int32_t* abort_flag) {
    const bool ok = wait_bar(bar, parity, abort_flag);
    return __all_sync(0xffffffffu, ok);
}

__device__ __forceinline__ uint32_t pack2_bf16(float a, float b) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<const uint32_t*>(&h);
}

__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
    asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};" ::"r"(addr), "r"(a), "r"(b), "r"(c), "r"(d) : "memory");
}

template <int D, int G>
__global__ void __launch_bounds__(kTcThreads, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                   const __grid_constant__ CUtensorMap tm_v, DevicePlan P, __nv_bfloat16* __restrict__ out,
                   float* __restrict__ ws, int h_q, float scale_log2) {
    using C = TcCfg<D>;
    constexpr int NS = C::NS;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw_addr = smem_u32(smem_raw);
    uint8_t* smem = smem_raw + ((1024u - (raw_addr & 1023u)) & 1023u);

    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);
    uint64_t* bar_q_full = bars;
    uint64_t* bar_k_full = bars + 1;
    uint64_t* bar_v_full = bars + 1 + NS;
    uint64_t* bar_kv_empty = bars + 1 + 2 * NS;
    uint64_t* bar_s_full = bars + 1 + 3 * NS;
    uint64_t* bar_s_free = bar_s_full + 2;
    uint64_t* bar_p_full = bar_s_free + 2;
    uint64_t* bar_o_done = bar_p_full + 1;
    uint64_t* bar_drain = bar_o_done + 1;
    uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(bars + C::N_BARS);
    volatile int32_t* abort_flag = reinterpret_cast<volatile int32_t*>(tmem_holder + 1);

    const AttnItem it = P.items[blockIdx.x];
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int n_tiles = it.kv_tile1 - it.kv_tile0;

    if (threadIdx.x == 0) {
        mbar_init(bar_q_full, 1);
        for (int s = 0; s < NS; ++s) {
            mbar_init(bar_k_full + s, 1);
            mbar_init(bar_v_full + s, 1);
            mbar_init(bar_kv_empty + s, 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar_s_full + i, 1);
            mbar_init(bar_s_free + i, kSoftmaxWarps);
        }
        mbar_init(bar_p_full, kSoftmaxWarps);
        mbar_init(bar_o_done, 1);
        mbar_init(bar_drain, 1);
        // after a recorded failure, later launches skip their work instead of waiting out their bounds
        *abort_flag = *reinterpret_cast<volatile int32_t*>(&g_attn_status) != 0 ? 1 : 0;
        fence_mbar_init();
    }
    if (warp == kMmaWarp) {
        tmem_alloc(tmem_holder, kTmemCols);
        tmem_relinquish();
    }
    if (warp == kTmaWarp && lane == 0) {
        prefetch_tensormap(&tm_q);
        prefetch_tensormap(&tm_k);
        prefetch_tensormap(&tm_v);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_holder;
    const bool skip = *abort_flag != 0;  // written before the barrier: uniform across the CTA

    if (skip) {
        // nothing issued: fall through to the teardown
    } else if (warp == kTmaWarp) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            const int g = it.kv_head;
            const int q_row0 = P.cu_fresh[it.query] + it.tok0;
            const int key_row0 = (int)P.cu_ctx[it.query] + it.kv_tile0 * kAttnBN;
            mbar_arrive_expect_tx(bar_q_full, C::Q_BYTES);
#pragma unroll
            for (int a = 0; a < C::ATOMS; ++a)
                tma_load_3d(smem + C::OFF_Q + a * C::ATOM_BYTES, &tm_q, a * 64, g * G, q_row0, bar_q_full);
            int issued = 0;
            for (int j = 0; j < n_tiles; ++j) {
                const int st = j % NS;
                if (!wait_bar(bar_kv_empty + st, ((j / NS) & 1) ^ 1, abort_flag)) break;
                const int key = key_row0 + j * kAttnBN;
                mbar_arrive_expect_tx(bar_k_full + st, C::KV_BYTES);
#pragma unroll
                for (int a = 0; a < C::ATOMS; ++a)
                    tma_load_3d(smem + C::OFF_K + st * C::KV_BYTES + a * C::ATOM_BYTES, &tm_k, a * 64, g, key,
                                bar_k_full + st);
                mbar_arrive_expect_tx(bar_v_full + st, C::KV_BYTES);
#pragma unroll
                for (int a = 0; a < C::ATOMS; ++a)
                    tma_load_3d(smem + C::OFF_V + st * C::KV_BYTES + a * C::ATOM_BYTES, &tm_v, a * 64, g, key,
                                bar_v_full + st);
                issued = j + 1;
            }
            // no copy may still be in flight when the CTA leaves
            drain_bar(bar_q_full, 0);
            for (int j = issued - NS > 0 ? issued - NS : 0; j < issued; ++j) {
                drain_bar(bar_k_full + j % NS, (j / NS) & 1);
                drain_bar(bar_v_full + j % NS, (j / NS) & 1);
            }
        }
    } else if (warp == kMmaWarp) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc_qk = idesc_bf16_f32(128, kAttnBN, 0, 0);
            constexpr uint32_t idesc_pv = idesc_bf16_f32(128, D, 0, 1);
            const uint32_t sQ = smem_u32(smem + C::OFF_Q);
            const uint32_t sP = smem_u32(smem + C::OFF_P);
            bool ok = wait_bar(bar_q_full, 0, abort_flag);
            auto issue_pv = [&](int i) -> bool {
                const int st = i % NS;
                if (!wait_bar(bar_p_full, i & 1, abort_flag)) return false;
                if (!wait_bar(bar_v_full + st, (i / NS) & 1, abort_flag)) return false;
                tc_fence_after();
                const uint32_t sV = smem_u32(smem + C::OFF_V + st * C::KV_BYTES);
#pragma unroll
                for (int kk = 0; kk < kAttnBN / 16; ++kk) {
                    const uint64_t a = sdesc_sw128(sP + (kk >> 2) * C::ATOM_BYTES + (kk & 3) * 32, 16, 1024);
                    const uint64_t b = sdesc_sw128(sV + kk * 16 * 128, C::ATOM_BYTES, 1024);
                    mma_bf16_ss(tmem + C::TMEM_O, a, b, idesc_pv, (i > 0 || kk > 0) ? 1u : 0u);
                }
                mma_commit(bar_o_done);
                mma_commit(bar_kv_empty + st);
                return true;
            };
            for (int j = 0; ok && j < n_tiles; ++j) {
                const int st = j % NS, sb = j & 1;
                if (!(ok = wait_bar(bar_k_full + st, (j / NS) & 1, abort_flag))) break;
                if (!(ok = wait_bar(bar_s_free + sb, ((j >> 1) & 1) ^ 1, abort_flag))) break;
                tc_fence_after();
                const uint32_t sK = smem_u32(smem + C::OFF_K + st * C::KV_BYTES);
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk) {
                    const uint32_t koff = (kk >> 2) * C::ATOM_BYTES + (kk & 3) * 32;
                    mma_bf16_ss(tmem + (sb ? C::TMEM_S1 : C::TMEM_S0), sdesc_sw128(sQ + koff, 16, 1024),
                                sdesc_sw128(sK + koff, 16, 1024), idesc_qk, kk > 0 ? 1u : 0u);
                }
                mma_commit(bar_s_full + sb);
                if (j >= 1) ok = issue_pv(j - 1);
            }
            if (ok && n_tiles > 0) ok = issue_pv(n_tiles - 1);
            mma_commit(bar_drain);  // arrives once every MMA issued above has completed
            drain_bar(bar_drain, 0);
        }
    } else {
        // ------------------------------------------------------------ softmax + epilogue
        const int r = threadIdx.x;  // tile row == TMEM lane
        const int tok = it.tok0 + r / G;
        const bool valid = tok < it.tok1;
        const int frow = P.cu_fresh[it.query] + tok;
        const int pos = valid ? P.fresh_pos[frow] : 0x7fffffff;
        const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
        const uint32_t sP = smem_u32(smem + C::OFF_P);
        float m = -INFINITY, l = 0.f;
        bool ok = true;
        for (int j = 0; j < n_tiles; ++j) {
            const int sb = j & 1;
            if (!(ok = warp_wait(bar_s_full + sb, (j >> 1) & 1, abort_flag))) break;
            tc_fence_after();
            uint32_t s[128];
            const uint32_t s_col = tmem + lane_base + (sb ? C::TMEM_S1 : C::TMEM_S0);
            tmem_ld32(s_col + 0, *reinterpret_cast<uint32_t(*)[32]>(s + 0));
            tmem_ld32(s_col + 32, *reinterpret_cast<uint32_t(*)[32]>(s + 32));
            tmem_ld32(s_col + 64, *reinterpret_cast<uint32_t(*)[32]>(s + 64));
            tmem_ld32(s_col + 96, *reinterpret_cast<uint32_t(*)[32]>(s + 96));
            tmem_ld_wait();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_s_free + sb);

            float x[128];
            const int key0 = (it.kv_tile0 + j) * kAttnBN;
            float mt = -INFINITY;
            if (key0 + kAttnBN - 1 > it.min_pos) {
#pragma unroll
                for (int c = 0; c < 128; ++c) {
                    x[c] = (key0 + c > pos) ? -INFINITY : __uint_as_float(s[c]) * scale_log2;
                    mt = fmaxf(mt, x[c]);
                }
            } else {
#pragma unroll
                for (int c = 0; c < 128; ++c) {
                    x[c] = __uint_as_float(s[c]) * scale_log2;
                    mt = fmaxf(mt, x[c]);
                }
            }
            const float m_new = fmaxf(m, mt);
            if (j > 0) {
                // PV_{j-1} complete: P may be overwritten and O is stable
                if (!(ok = warp_wait(bar_o_done, (j - 1) & 1, abort_flag))) break;
                tc_fence_after();
            }
            const bool resc = m_new > m + kRescaleThreshold;
            float alpha = 1.f;
            if (resc) {
                alpha = ex2_approx(m - m_new);
                l *= alpha;
                m = m_new;
            }
            if (j > 0 && __any_sync(0xffffffffu, resc)) {
#pragma unroll
                for (int c4 = 0; c4 < D / 32; ++c4) {
                    uint32_t o[32];
                    const uint32_t o_col = tmem + lane_base + C::TMEM_O + c4 * 32;
                    tmem_ld32(o_col, o);
                    tmem_ld_wait();
#pragma unroll
                    for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
                    tmem_st32(o_col, o);
                }
                tmem_st_wait();
            }
            const float mu = (m == -INFINITY) ? 0.f : m;
            float rs = 0.f;
#pragma unroll
            for (int cc = 0; cc < 16; ++cc) {
                float p[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    p[e] = ex2_approx(x[cc * 8 + e] - mu);
                    rs += p[e];
                }
                const uint32_t addr = sP + (cc >> 3) * C::ATOM_BYTES + r * 128 + ((((cc & 7) ^ (r & 7))) << 4);
                st_shared_v4(addr, pack2_bf16(p[0], p[1]), pack2_bf16(p[2], p[3]), pack2_bf16(p[4], p[5]),
                             pack2_bf16(p[6], p[7]));
            }
            l += rs;
            fence_proxy_async_smem();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_p_full);
        }
        if (ok && n_tiles > 0) ok = warp_wait(bar_o_done, (n_tiles - 1) & 1, abort_flag);
        if (ok) {
            tc_fence_after();
            if (it.slot < 0) {
                const float inv = 1.f / l;
                __nv_bfloat16* orow = out + ((int64_t)frow * h_q + it.kv_head * G + (r % G)) * D;
#pragma unroll
                for (int c4 = 0; c4 < D / 32; ++c4) {
                    uint32_t o[32];
                    tmem_ld32(tmem + lane_base + C::TMEM_O + c4 * 32, o);
                    tmem_ld_wait();
                    if (valid) {
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            uint4 w;
                            w.x = pack2_bf16(__uint_as_float(o[8 * q + 0]) * inv, __uint_as_float(o[8 * q + 1]) * inv);
                            w.y = pack2_bf16(__uint_as_float(o[8 * q + 2]) * inv, __uint_as_float(o[8 * q + 3]) * inv);
                            w.z = pack2_bf16(__uint_as_float(o[8 * q + 4]) * inv, __uint_as_float(o[8 * q + 5]) * inv);
                            w.w = pack2_bf16(__uint_as_float(o[8 * q + 6]) * inv, __uint_as_float(o[8 * q + 7]) * inv);
                            *reinterpret_cast<uint4*>(orow + c4 * 32 + 8 * q) = w;
                        }
                    }
                }
            } else {
                float* wo = ws + (int64_t)it.slot * kAttnBM * (D + 2);
#pragma unroll
                for (int c4 = 0; c4 < D / 32; ++c4) {
                    uint32_t o[32];
                    tmem_ld32(tmem + lane_base + C::TMEM_O + c4 * 32, o);
                    tmem_ld_wait();
#pragma unroll
                    for (int q = 0; q < 8; ++q)
                        *reinterpret_cast<uint4*>(wo + r * D + c4 * 32 + 4 * q) =
                            make_uint4(o[4 * q], o[4 * q + 1], o[4 * q + 2], o[4 * q + 3]);
                }
                wo[kAttnBM * D + r] = m;
                wo[kAttnBM * D + kAttnBM + r] = l;
            }
        }
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
static bool make_map_3d(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1, uint64_t d2, uint32_t b0,
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
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(attn_tc_kernel<D, G>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)C::SMEM_BYTES);
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    if (n_items > 0)
        attn_tc_kernel<D, G><<<n_items, kTcThreads, C::SMEM_BYTES, stream>>>(
            mq, mk, mv, P, (__nv_bfloat16*)out, ws, h_q, scale_log2);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    if (n_merges > 0) attn_merge_kernel<D><<<n_merges, 256, 0, stream>>>(P, ws, (__nv_bfloat16*)out, h_q, G);
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

int read_attention_status(int32_t* status) {
    return cudaMemcpyFromSymbol(status, g_attn_status, sizeof(int32_t)) == cudaSuccess ? KVLINK_OK : KVLINK_ECUDA;
}

int clear_attention_status() {
    const int32_t z = 0;
    return cudaMemcpyToSymbol(g_attn_status, &z, sizeof(int32_t)) == cudaSuccess ? KVLINK_OK : KVLINK_ECUDA;
}

}  // namespace kvlink
