// Suffix attention on the tcgen05 tensor cores (Sec. 2.3, "inference").
//
// Work item = one M-tile of up to 128 rows (up to 128/G fresh tokens x the G
// query heads that share one KV head) of one query, over a range of 128-key
// tiles of that query's linked cache.  Rows are (token, head) pairs, so the G
// heads of a GQA group share every K/V tile load.
//
// Warp roles (224 threads, one CTA per SM, 512 TMEM columns):
//   warps 0-3  softmax + epilogue; thread r owns row r = TMEM lane r
//   warp 4     TMA: Q once, then K tiles into an NK-stage ring
//   warp 5     TMEM allocation and the single MMA-issuing thread
//   warp 6     TMA: V tiles into an NV-stage ring
// Per KV tile j (TMEM: three S/P buffers of 128 columns, then O):
//   S_j = Q K_j^T           tcgen05.mma SMEM x SMEM -> S buffer j%3
//   P_j = exp2(S_j c - m)   softmax warps: TMEM -> registers -> bf16 P written back
//                           over the first 64 columns of the same buffer
//   O  += P_j V_j           tcgen05.mma TMEM x SMEM (P from TMEM, V read MN-major)
// S_j is issued only after PV_{j-3} has finished reading the buffer, so up to
// three tiles are in flight and the softmax never waits on a PV except to
// rescale O.  The running max m is raised only when it grows by more than 2^8,
// so that rescale is rare.  The mask keeps key slot j for a row at global
// position p iff j <= p, and is evaluated only on tiles that reach past the
// tile's smallest row position.  Items whose KV range was split write
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

#include "kvlink_internal.h"
#include "kvlink_sm100.cuh"

namespace kvlink {
using namespace sm100;

static __device__ int32_t g_attn_status;

constexpr int kTcThreads = 224;
constexpr int kSoftmaxWarps = 4;
constexpr int kTmaKWarp = 4;
constexpr int kMmaWarp = 5;
constexpr int kTmaVWarp = 6;
constexpr uint32_t kTmemCols = 512;
constexpr uint64_t kWaitLimitNs = 2000000000ull;  // 2 s
constexpr int32_t kAttnStatusWaitTimeout = 0x41;
constexpr float kRescaleThreshold = 8.0f;         // log2 units: rescale O when the max grows by > 2^8
#ifndef KVLINK_EXP_POLY_FROM
#define KVLINK_EXP_POLY_FROM 8                     // column pairs c with (c % 8) >= this use exp2_poly2
#endif
#ifndef KVLINK_PRODUCER_BACKOFF_NS
#define KVLINK_PRODUCER_BACKOFF_NS 0               // sleep between polls of the TMA producers' waits
#endif

template <int D>
struct TcCfg {
    static constexpr int ATOMS = D / 64;                 // 128-byte swizzle atoms along head_dim
    static constexpr int NK = (D == 128) ? 3 : 5;        // K ring stages
    static constexpr int NV = (D == 128) ? 3 : 5;        // V ring stages
    static constexpr int NB = 3;                         // S/P buffers in TMEM
    static constexpr uint32_t ATOM_BYTES = 128 * 128;    // [128 rows][64 bf16]
    static constexpr uint32_t Q_BYTES = ATOMS * ATOM_BYTES;
    static constexpr uint32_t KV_BYTES = ATOMS * ATOM_BYTES;
    static constexpr uint32_t OFF_Q = 0;
    static constexpr uint32_t OFF_K = OFF_Q + Q_BYTES;
    static constexpr uint32_t OFF_V = OFF_K + NK * KV_BYTES;
    static constexpr uint32_t OFF_BAR = OFF_V + NV * KV_BYTES;
    // q_full, k_full[NK], k_empty[NK], v_full[NV], v_empty[NV], s_full[NB], p_full[NB], o_done[NB], drain
    static constexpr int N_BARS = 1 + 2 * NK + 2 * NV + 3 * NB + 1;
    static constexpr uint32_t SMEM_BYTES = OFF_BAR + N_BARS * 8 + 16 + 1024;
    // TMEM columns: S/P buffers then the O accumulator
    static constexpr uint32_t TMEM_S = 0;                // buffer b at b * 128
    static constexpr uint32_t TMEM_O = NB * kAttnBN;
    static_assert(TMEM_O + D <= kTmemCols, "TMEM budget");
    static_assert(SMEM_BYTES <= 232448, "shared memory budget");
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

// wait_bar with a short sleep between polls, for roles off the critical path
__device__ __forceinline__ bool wait_bar_backoff(uint64_t* bar, uint32_t parity, volatile int32_t* abort_flag) {
    if (KVLINK_PRODUCER_BACKOFF_NS == 0) return wait_bar(bar, parity, abort_flag);
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = globaltimer_ns();
    while (true) {
        __nanosleep(KVLINK_PRODUCER_BACKOFF_NS);
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

// 2^x for a pair of floats on the FMA pipe: x = n + f with n = rint(x) (taken from the
// mantissa of x + 1.5*2^23) and f in [-1/2, 1/2]; 2^f from a degree-3 minimax polynomial
// (Remez exchange on relative error, max relative error 7.5e-5, far below the bf16
// quantum of P); 2^n added into the exponent field.  Inputs are clamped at kExpFloor =
// -126 so that the exponent field never wraps (p >= 2^-1/2 keeps it >= 0): anything at
// or below the floor comes out as a non-negative value under 2^-125, i.e. nothing
// against any unmasked term.
__device__ __forceinline__ uint64_t exp2_poly2(uint64_t x2) {
    constexpr float kC0 = 0.99992806f, kC1 = 0.69326097f, kC2 = 0.24261113f, kC3 = 0.05517167f;
    constexpr float kRound = 12582912.0f;  // 1.5 * 2^23
    constexpr float kExpFloor = -126.0f;
    float a, b;
    f2_unpack(x2, a, b);
    const uint64_t x = f2_pack(fmaxf(a, kExpFloor), fmaxf(b, kExpFloor));
    const uint64_t t = fadd2(x, f2_pack(kRound, kRound));
    const uint64_t n = fadd2(t, f2_pack(-kRound, -kRound));
    const uint64_t f = ffma2(n, f2_pack(-1.f, -1.f), x);
    uint64_t p = ffma2(f, f2_pack(kC3, kC3), f2_pack(kC2, kC2));
    p = ffma2(p, f, f2_pack(kC1, kC1));
    p = ffma2(p, f, f2_pack(kC0, kC0));
    float pa, pb, ta, tb;
    f2_unpack(p, pa, pb);
    f2_unpack(t, ta, tb);
    const float ra = __int_as_float(__float_as_int(pa) + (int)((uint32_t)__float_as_int(ta) << 23));
    const float rb = __int_as_float(__float_as_int(pb) + (int)((uint32_t)__float_as_int(tb) << 23));
    return f2_pack(ra, rb);
}

// TMA producer loop for one ring (K or V): tiles j = 0..n-1 of the item's key range.
template <int STAGES, int ATOMS>
__device__ __forceinline__ void produce_ring(uint8_t* ring, uint32_t stage_bytes, const CUtensorMap* map,
                                             uint64_t* full, uint64_t* empty, int n, int g, int key_row0,
                                             volatile int32_t* abort_flag) {
    int issued = 0;
    for (int j = 0; j < n; ++j) {
        const int st = j % STAGES;
        if (!wait_bar_backoff(empty + st, ((j / STAGES) & 1) ^ 1, abort_flag)) break;
        mbar_arrive_expect_tx(full + st, stage_bytes);
#pragma unroll
        for (int a = 0; a < ATOMS; ++a)
            tma_load_3d(ring + st * stage_bytes + a * (128 * 128), map, a * 64, g, key_row0 + j * kAttnBN, full + st);
        issued = j + 1;
    }
    // no copy may still be in flight when the CTA leaves
    for (int j = issued - STAGES > 0 ? issued - STAGES : 0; j < issued; ++j) drain_bar(full + j % STAGES, (j / STAGES) & 1);
}

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
    const int key_row0 = (int)P.cu_ctx[it.query] + it.kv_tile0 * kAttnBN;

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
            produce_ring<NK, C::ATOMS>(smem + C::OFF_K, C::KV_BYTES, &tm_k, bar_k_full, bar_k_empty, n_tiles,
                                       it.kv_head, key_row0, abort_flag);
            drain_bar(bar_q_full, 0);
        }
    } else if (warp == kTmaVWarp) {
        // ------------------------------------------------------------ the V ring
        if (lane == 0)
            produce_ring<NV, C::ATOMS>(smem + C::OFF_V, C::KV_BYTES, &tm_v, bar_v_full, bar_v_empty, n_tiles,
                                       it.kv_head, key_row0, abort_flag);
    } else if (warp == kMmaWarp) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc_qk = idesc_bf16_f32(128, kAttnBN, 0, 0);
            constexpr uint32_t idesc_pv = idesc_bf16_f32(128, D, 0, 1);
            const uint32_t sQ = smem_u32(smem + C::OFF_Q);
            bool ok = wait_bar(bar_q_full, 0, abort_flag);
            // O += P_i V_i, P_i (bf16) read from its S buffer in TMEM
            auto issue_pv = [&](int i) -> bool {
                const int b = i % NB, sv = i % NV;
                if (!wait_bar(bar_p_full + b, (i / NB) & 1, abort_flag)) return false;
                if (!wait_bar(bar_v_full + sv, (i / NV) & 1, abort_flag)) return false;
                tc_fence_after();
                const uint32_t sV = smem_u32(smem + C::OFF_V + sv * C::KV_BYTES);
                const uint32_t pcol = tmem + C::TMEM_S + b * kAttnBN;
#pragma unroll
                for (int kk = 0; kk < kAttnBN / 16; ++kk)
                    mma_bf16_ts(tmem + C::TMEM_O, pcol + kk * 8, sdesc_sw128(sV + kk * 16 * 128, C::ATOM_BYTES, 1024),
                                idesc_pv, (i > 0 || kk > 0) ? 1u : 0u);
                mma_commit(bar_o_done + b);
                mma_commit(bar_v_empty + sv);
                return true;
            };
            for (int j = 0; ok && j < n_tiles; ++j) {
                const int sk = j % NK, b = j % NB;
                if (!(ok = wait_bar(bar_k_full + sk, (j / NK) & 1, abort_flag))) break;
                // buffer b last held P_{j-NB}: its PV must have finished reading it
                if (j >= NB && !(ok = wait_bar(bar_o_done + b, ((j - NB) / NB) & 1, abort_flag))) break;
                tc_fence_after();
                const uint32_t sK = smem_u32(smem + C::OFF_K + sk * C::KV_BYTES);
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk) {
                    const uint32_t koff = (kk >> 2) * C::ATOM_BYTES + (kk & 3) * 32;
                    mma_bf16_ss(tmem + C::TMEM_S + b * kAttnBN, sdesc_sw128(sQ + koff, 16, 1024),
                                sdesc_sw128(sK + koff, 16, 1024), idesc_qk, kk > 0 ? 1u : 0u);
                }
                mma_commit(bar_s_full + b);
                mma_commit(bar_k_empty + sk);
                if (j >= 1) ok = issue_pv(j - 1);
            }
            if (ok && n_tiles > 0) ok = issue_pv(n_tiles - 1);
            mma_commit(bar_drain);  // arrives once every MMA issued above has completed
            drain_bar(bar_drain, 0);
        }
    } else {
        // ------------------------------------------------------------ softmax + epilogue (warps 0-3)
        const int r = threadIdx.x;  // tile row == TMEM lane
        const int tok = it.tok0 + r / G;
        const bool valid = tok < it.tok1;
        const int frow = P.cu_fresh[it.query] + tok;
        const int pos = valid ? P.fresh_pos[frow] : 0x7fffffff;
        const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
        float m = -INFINITY, l = 0.f;
        bool ok = true;
        for (int j = 0; j < n_tiles; ++j) {
            const int b = j % NB;
            if (!(ok = warp_wait(bar_s_full + b, (j / NB) & 1, abort_flag))) break;
            tc_fence_after();
            uint32_t s[128];
            const uint32_t s_col = tmem + lane_base + C::TMEM_S + b * kAttnBN;
            tmem_ld32(s_col + 0, *reinterpret_cast<uint32_t(*)[32]>(s + 0));
            tmem_ld32(s_col + 32, *reinterpret_cast<uint32_t(*)[32]>(s + 32));
            tmem_ld32(s_col + 64, *reinterpret_cast<uint32_t(*)[32]>(s + 64));
            tmem_ld32(s_col + 96, *reinterpret_cast<uint32_t(*)[32]>(s + 96));
            tmem_ld_wait();

            // raw row max (scale > 0 commutes with max); masked slots become -inf.  Eight
            // independent running maxima keep the dependency chain short.
            const int key0 = (it.kv_tile0 + j) * kAttnBN;
            float mx8[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) mx8[e] = -INFINITY;
            if (key0 + kAttnBN - 1 > it.min_pos) {
#pragma unroll
                for (int c = 0; c < 128; ++c) {
                    if (key0 + c > pos) s[c] = __float_as_uint(-INFINITY);
                    mx8[c & 7] = fmaxf(mx8[c & 7], __uint_as_float(s[c]));
                }
            } else {
#pragma unroll
                for (int c = 0; c < 128; ++c) mx8[c & 7] = fmaxf(mx8[c & 7], __uint_as_float(s[c]));
            }
            const float mx = fmaxf(fmaxf(fmaxf(mx8[0], mx8[1]), fmaxf(mx8[2], mx8[3])),
                                   fmaxf(fmaxf(mx8[4], mx8[5]), fmaxf(mx8[6], mx8[7])));
            const float m_new = fmaxf(m, mx * scale_log2);
            const bool resc = m_new > m + kRescaleThreshold;
            float alpha = 1.f;
            if (resc) {
                alpha = ex2_approx(m - m_new);
                l *= alpha;
                m = m_new;
            }
            if (j > 0 && __any_sync(0xffffffffu, resc)) {
                // O is touched only while no PV is in flight: PV_{j-1} done, PV_j not yet issued
                if (!(ok = warp_wait(bar_o_done + (j - 1) % NB, ((j - 1) / NB) & 1, abort_flag))) break;
                tc_fence_after();
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
            }
            // p = exp2(s * scale - m) on column pairs (packed f32x2 arithmetic); three pairs
            // in eight go to the FMA pipe (exp2_poly2), the rest to MUFU, to balance the two
            const float mu = (m == -INFINITY) ? 0.f : m;
            const uint64_t sc2 = f2_pack(scale_log2, scale_log2);
            const uint64_t nmu2 = f2_pack(-mu, -mu);
            uint64_t acc[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) acc[e] = f2_pack(0.f, 0.f);
            uint32_t pk[64];
#pragma unroll
            for (int c = 0; c < 64; ++c) {
                const uint64_t x2 = ffma2(f2_pack(__uint_as_float(s[2 * c]), __uint_as_float(s[2 * c + 1])), sc2, nmu2);
                uint64_t p2;
                if ((c & 7) >= KVLINK_EXP_POLY_FROM) {
                    p2 = exp2_poly2(x2);
                } else {
                    float a, b;
                    f2_unpack(x2, a, b);
                    p2 = f2_pack(ex2_approx(a), ex2_approx(b));
                }
                acc[c & 3] = fadd2(acc[c & 3], p2);
                float p0, p1;
                f2_unpack(p2, p0, p1);
                pk[c] = pack2_bf16(p0, p1);
            }
            float rs0, rs1;
            f2_unpack(fadd2(fadd2(acc[0], acc[1]), fadd2(acc[2], acc[3])), rs0, rs1);
            const float rs = rs0 + rs1;
            l += rs;
            // P_j (bf16) over the first 64 columns of its S buffer, read there by the PV MMA
            tmem_st32(s_col + 0, *reinterpret_cast<uint32_t(*)[32]>(pk + 0));
            tmem_st32(s_col + 32, *reinterpret_cast<uint32_t(*)[32]>(pk + 32));
            tmem_st_wait();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_p_full + b);
        }
        if (ok && n_tiles > 0) ok = warp_wait(bar_o_done + (n_tiles - 1) % NB, ((n_tiles - 1) / NB) & 1, abort_flag);
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
