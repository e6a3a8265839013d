// Suffix attention on the tcgen05 tensor cores (Sec. 2.3, "inference").
//
// Work item = one M-tile of up to 128 rows (up to 128/G fresh tokens x the G query heads
// that share one KV head) of one query, over a range of 128-key tiles of that query's linked
// cache (cache-row order; in the links-at-end layout the cached rows and the fresh rows at
// the end form two runs).  Rows are (token, head) pairs, so the G heads of a GQA group share
// every K/V tile load.  The kernel is persistent: one CTA per SM runs the list of items the
// plan gave it (see the comment before PtCfg for the warp roles).
//
// Per KV tile j (TMEM: three S/P buffers of 128 columns, then O):
//   S_j = Q K_j^T           tcgen05.mma SMEM x SMEM -> S buffer j%3
//   P_j = exp2(S_j c - m)   softmax warps: TMEM -> registers -> bf16 P written back
//                           over the first 64 columns of the same buffer
//   O  += P_j V_j           tcgen05.mma TMEM x SMEM (P from TMEM, V read MN-major)
// S_j is issued only after PV_{j-3} has finished reading the buffer, so up to three tiles
// are in flight and the softmax never waits on a PV except to rescale O.  S and PV come from
// two issuing threads: a thread that waits on an mbarrier right after its own tcgen05.commit
// was seen to stall until its MMAs had drained.  The running max m is raised only when it
// grows by more than 2^8, so the rescale is rare.  The mask keeps the cache rows holding
// positions up to the row's own and is evaluated only on tiles that reach past the rows every
// row of the tile sees.
//
// Every mbarrier wait is bounded in time.  On expiry the kernel records
// kAttnStatusWaitTimeout in its status word, the other roles leave their loops, the producer
// and MMA threads wait (bounded) for their own in-flight copies and MMAs, TMEM is freed and
// the CTA returns.
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

constexpr int kPvWarp = 7;
constexpr int kSoftmaxWarps = 4;
constexpr int kTmaKWarp = 4;
constexpr int kMmaWarp = 5;
constexpr int kTmaVWarp = 6;


// ------------------------------------------------------------------------------------------
// Persistent form: one CTA per SM runs its list of items (the plan's per-CTA schedule) back to
// back.  Every role walks the same list on its own and keeps its ring slots, TMEM buffers and
// barrier phases going across items, so an item's start (Q, the first key tiles) and finish
// (reading O out of TMEM, normalising, storing) overlap the neighbouring items' tile loops
// instead of idling the tensor cores, and no CTA is launched per item.
//   warps 0-3   softmax (softmax_item); at the end of an item its m and l go to shared memory
//   warp 4      TMA: Q of each item into one of two Q buffers (so it lands while the previous
//               item runs), and the K tiles into the NK-stage ring
//   warp 5      TMEM allocation; the thread issuing S = Q K^T
//   warp 6      TMA: V tiles into the NV-stage ring
//   warp 7      the thread issuing O += P V; an item's first PV waits until the epilogue has
//               read the previous item's O
//   warps 8-11  epilogue: once an item's last PV has finished, O is read out of TMEM (the
//               accumulator is then free for the next item) and normalised and stored from
//               registers.  A piece of a split KV range stores its partial (O, m, l); the
//               piece that completes its group (a per-group arrival counter in the plan
//               buffer) merges the group's partials into the output, so no merge launch follows
// Registers: launched at 168 per thread (384 x 168 <= 64K); the TMA/MMA warpgroup drops to
// 56 and the softmax warpgroup rises to 240 (240 + 56 + 168 per SM sub-partition).
constexpr int kPtThreads = 384;
constexpr int kPtEpiWarp0 = 8;
constexpr uint32_t kPtSoftmaxRegs = 240, kPtIdleRegs = 56;
static_assert(kPtThreads * 168 <= 65536, "launch register budget");
static_assert(128 * (kPtSoftmaxRegs + kPtIdleRegs + 168) <= kPtThreads * 168, "register split");

// Shared memory: two Q buffers (the next item's Q lands while the current item runs), the K
// ring and the V ring (one stage shorter than the K ring for head_dim 128: a V tile is needed
// a softmax later than its K tile), m and l of one item, a flag, the barriers.
template <int D>
struct PtCfg {
    static constexpr int ATOMS = D / 64;
    static constexpr int NK = (D == 128) ? 3 : 5;
    static constexpr int NV = (D == 128) ? 2 : 4;
    static constexpr int NB = 3;
    static constexpr uint32_t ATOM_BYTES = 128 * 128;
    static constexpr uint32_t Q_BYTES = ATOMS * ATOM_BYTES, KV_BYTES = ATOMS * ATOM_BYTES;
    static constexpr uint32_t OFF_Q = 0;                                // two buffers
    static constexpr uint32_t OFF_K = OFF_Q + 2 * Q_BYTES;
    static constexpr uint32_t OFF_V = OFF_K + NK * KV_BYTES;
    static constexpr uint32_t OFF_STATS = OFF_V + NV * KV_BYTES;        // m[128], l[128] of one item
    static constexpr uint32_t OFF_FLAG = OFF_STATS + 2 * kAttnBM * 4;   // the epilogue's merge decision
    static constexpr uint32_t OFF_BAR = OFF_FLAG + 16;
    // q_full[2], q_empty[2], k_full[NK], k_empty[NK], v_full[NV], v_empty[NV], s_full[NB],
    // p_full[NB], o_done[NB], o_full, o_free, st_full, st_empty, drain x2
    static constexpr int N_BARS = 4 + 2 * NK + 2 * NV + 3 * NB + 6;
    static constexpr uint32_t SMEM_BYTES = OFF_BAR + N_BARS * 8 + 16 + 1024;
    static constexpr uint32_t TMEM_S = 0, TMEM_O = NB * kAttnBN;
    static_assert(TMEM_O + D <= kTmemCols, "TMEM budget");
    static_assert(SMEM_BYTES <= 232448, "shared memory budget");
};

// The epilogue warps' part of an item (thread r = TMEM lane r): O read out of TMEM (then the
// accumulator is free for the next item's PVs), normalised and stored; for a piece of a split
// range its partial is stored, and the piece that completes its merge group combines all the
// group's partials into the output.  The four warps take every decision together (named
// barrier 1 over their 128 threads).
template <int D, int G>
__device__ __forceinline__ void epilogue_item(const AttnItem& it, const DevicePlan& P, int r, uint32_t o_taddr,
                                              float m, float l, uint64_t* bar_o_free, volatile int32_t* flag,
                                              __nv_bfloat16* __restrict__ out, float* __restrict__ ws, int h_q) {
    uint32_t o[D];
#pragma unroll
    for (int c4 = 0; c4 < D / 32; ++c4) tmem_ld32(o_taddr + c4 * 32, *reinterpret_cast<uint32_t(*)[32]>(o + 32 * c4));
    tmem_ld_wait();
    tc_fence_before();
    __syncwarp();
    if (threadIdx.x % 32 == 0) mbar_arrive(bar_o_free);     // O may now take the next item's PVs
    store_result<D, G>(it, P, r, o, 0, D, m, l, out, ws, h_q);
    if (it.slot < 0) return;
    // a piece of a split range: the last of its group to arrive merges
    const int grp = P.slot_group[it.slot];
    const MergeGroup mg = P.merges[grp];
    // The four warps' partial stores are ordered before thread 0's arrival by the barrier, and
    // the arrival (release, cumulative) publishes them to every CTA; the arrival that completes
    // the group also acquires the other pieces' partials, which the barrier then orders before
    // this CTA's reads of them.
    named_bar_sync(1, 128);
    if (r == 0) *flag = ((atom_add_acq_rel_gpu(P.merge_count + grp, 1ull) + 1) % (unsigned long long)mg.n_split) == 0;
    named_bar_sync(1, 128);
    const bool last = *flag != 0;
    named_bar_sync(1, 128);                 // every thread has read the flag before it is reused
    if (!last) return;
    const int tok = mg.tok0 + r / G;
    if (tok >= mg.tok1) return;
    merge_row_store<D>(ws, mg.slot0, mg.n_split, r,
                       out + ((int64_t)(P.cu_fresh[mg.query] + tok) * h_q + mg.kv_head * G + (r % G)) * D);
}

template <int D, int G>
__global__ void __launch_bounds__(kPtThreads, 1)
    attn_tc_persistent_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                              const __grid_constant__ CUtensorMap tm_v, DevicePlan P,
                              __nv_bfloat16* __restrict__ out, float* __restrict__ ws, int h_q, float scale_log2) {
    using C = PtCfg<D>;
    constexpr int NK = C::NK, NV = C::NV, NB = C::NB;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw_addr = smem_u32(smem_raw);
    uint8_t* smem = smem_raw + ((1024u - (raw_addr & 1023u)) & 1023u);

    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);
    uint64_t* bar_q_full = bars;                 // [2]
    uint64_t* bar_q_empty = bar_q_full + 2;      // [2]
    uint64_t* bar_k_full = bar_q_empty + 2;
    uint64_t* bar_k_empty = bar_k_full + NK;
    uint64_t* bar_v_full = bar_k_empty + NK;
    uint64_t* bar_v_empty = bar_v_full + NV;
    uint64_t* bar_s_full = bar_v_empty + NV;
    uint64_t* bar_p_full = bar_s_full + NB;
    uint64_t* bar_o_done = bar_p_full + NB;
    uint64_t* bar_o_full = bar_o_done + NB;
    uint64_t* bar_o_free = bar_o_full + 1;
    uint64_t* bar_st_full = bar_o_free + 1;
    uint64_t* bar_st_empty = bar_st_full + 1;
    uint64_t* bar_drain = bar_st_empty + 1;
    uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(bars + C::N_BARS);
    volatile int32_t* abort_flag = reinterpret_cast<volatile int32_t*>(tmem_holder + 1);
    float* st_m = reinterpret_cast<float*>(smem + C::OFF_STATS);
    float* st_l = st_m + kAttnBM;
    volatile int32_t* merge_flag = reinterpret_cast<volatile int32_t*>(smem + C::OFF_FLAG);

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int first = P.cu_sched[blockIdx.x], n_mine = P.cu_sched[blockIdx.x + 1] - first;
    int32_t* status = &g_attn_status;

    if (threadIdx.x == 0) {
        for (int i = 0; i < C::N_BARS; ++i) {
            uint64_t* b = bars + i;
            // arrivals per phase: one per softmax / epilogue warp, else one (thread or commit)
            const bool four = (b >= bar_p_full && b < bar_p_full + NB) || b == bar_o_free || b == bar_st_full ||
                              b == bar_st_empty;
            mbar_init(b, four ? 4 : 1);
        }
        // after a recorded failure, later launches skip their work instead of waiting out their bounds
        *abort_flag = *reinterpret_cast<volatile int32_t*>(&g_attn_status) != 0 ? 1 : 0;
#ifdef KVLINK_DEBUG_CHECKS
        for (int k = 0; k < n_mine && !*abort_flag; ++k) {
            const int idx = P.sched[first + k];
            bool ok = idx >= 0 && idx < P.n_items && item_in_bounds(P.items[idx], P) &&
                      P.items[idx].kv_tile1 > P.items[idx].kv_tile0;
            if (ok && P.items[idx].slot >= 0) {
                const int grp = P.slot_group[P.items[idx].slot];
                ok = grp >= 0 && grp < P.n_merges && P.merges[grp].n_split >= 1 &&
                     P.merges[grp].slot0 >= 0 && P.merges[grp].slot0 + P.merges[grp].n_split <= P.n_slots;
            }
            if (!ok) {
                atomicCAS(&g_attn_status, 0, kAttnStatusBadIndex);
                *abort_flag = 1;
            }
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

    if (skip) {
        // nothing issued: fall through to the teardown
    } else if (warp >= kSoftmaxWarps && warp < kPtEpiWarp0) {
        setmaxnreg_dec<kPtIdleRegs>();
        if (warp == kTmaKWarp && lane == 0) {
            // ------------------------------------------------ Q of every item, and the K ring
            int g = 0, q_issued = 0;
            bool ok = true;
            for (int k = 0; ok && k < n_mine; ++k) {
                const AttnItem it = P.items[P.sched[first + k]];
                const int n = it.kv_tile1 - it.kv_tile0, ctx0 = (int)P.cu_ctx[it.query];
                // Q buffer k % 2, once the S MMAs of item k - 2 have read it
                const int qb = k & 1;
                if (!(ok = wait_bar(bar_q_empty + qb, ((k >> 1) & 1) ^ 1, abort_flag, status))) break;
                mbar_arrive_expect_tx(bar_q_full + qb, C::Q_BYTES);
#pragma unroll
                for (int a = 0; a < C::ATOMS; ++a)
                    tma_load_3d(smem + C::OFF_Q + qb * C::Q_BYTES + a * C::ATOM_BYTES, &tm_q, a * 64,
                                it.kv_head * G, P.cu_fresh[it.query] + it.tok0, bar_q_full + qb);
                ++q_issued;
                for (int j = 0; j < n; ++j, ++g) {
                    const int st = g % NK;
                    if (!(ok = wait_bar(bar_k_empty + st, ((g / NK) & 1) ^ 1, abort_flag, status))) break;
                    const int row = ctx0 + item_tile(it, it.kv_tile0 + j) * kAttnBN;
                    mbar_arrive_expect_tx(bar_k_full + st, C::KV_BYTES);
#pragma unroll
                    for (int a = 0; a < C::ATOMS; ++a)
                        tma_load_3d(smem + C::OFF_K + st * C::KV_BYTES + a * C::ATOM_BYTES, &tm_k, a * 64, it.kv_head,
                                    row, bar_k_full + st);
                }
            }
            // no copy may still be in flight when the CTA leaves
            for (int gg = g - NK > 0 ? g - NK : 0; gg < g; ++gg) drain_bar(bar_k_full + gg % NK, (gg / NK) & 1, status);
            for (int k = q_issued - 2 > 0 ? q_issued - 2 : 0; k < q_issued; ++k)
                drain_bar(bar_q_full + (k & 1), (k >> 1) & 1, status);
        } else if (warp == kTmaVWarp && lane == 0) {
            // ------------------------------------------------ the V ring
            int g = 0;
            bool ok = true;
            for (int k = 0; ok && k < n_mine; ++k) {
                const AttnItem it = P.items[P.sched[first + k]];
                const int n = it.kv_tile1 - it.kv_tile0, ctx0 = (int)P.cu_ctx[it.query];
                for (int j = 0; j < n; ++j, ++g) {
                    const int st = g % NV;
                    if (!(ok = wait_bar(bar_v_empty + st, ((g / NV) & 1) ^ 1, abort_flag, status))) break;
                    const int row = ctx0 + item_tile(it, it.kv_tile0 + j) * kAttnBN;
                    mbar_arrive_expect_tx(bar_v_full + st, C::KV_BYTES);
#pragma unroll
                    for (int a = 0; a < C::ATOMS; ++a)
                        tma_load_3d(smem + C::OFF_V + st * C::KV_BYTES + a * C::ATOM_BYTES, &tm_v, a * 64, it.kv_head,
                                    row, bar_v_full + st);
                }
            }
            for (int gg = g - NV > 0 ? g - NV : 0; gg < g; ++gg) drain_bar(bar_v_full + gg % NV, (gg / NV) & 1, status);
        } else if (warp == kMmaWarp && lane == 0) {
            // ------------------------------------------------ S = Q K^T
            constexpr uint32_t idesc_qk = idesc_bf16_f32(128, kAttnBN, 0, 0);
            int g = 0;
            bool ok = true;
            for (int k = 0; ok && k < n_mine; ++k) {
                const AttnItem it = P.items[P.sched[first + k]];
                const int n = it.kv_tile1 - it.kv_tile0;
                const int qb = k & 1;
                if (!(ok = wait_bar(bar_q_full + qb, (k >> 1) & 1, abort_flag, status))) break;
                const uint32_t sQ = smem_u32(smem + C::OFF_Q + qb * C::Q_BYTES);
                for (int j = 0; j < n; ++j, ++g) {
                    const int sk = g % NK, b = g % NB;
                    if (!(ok = wait_bar(bar_k_full + sk, (g / NK) & 1, abort_flag, status))) break;
                    // buffer b last held P of tile g - NB: its PV must have finished reading it
                    if (g >= NB && !(ok = wait_bar(bar_o_done + b, ((g - NB) / NB) & 1, abort_flag, status))) break;
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
                }
                if (ok) mma_commit(bar_q_empty + qb);   // arrives once this item's S MMAs have read Q
            }
            mma_commit(bar_drain);
            drain_bar(bar_drain, 0, status);
        } else if (warp == kPvWarp && lane == 0) {
            // ------------------------------------------------ O += P V
            constexpr uint32_t idesc_pv = idesc_bf16_f32(128, D, 0, 1);
            int g = 0;
            bool ok = true;
            for (int k = 0; ok && k < n_mine; ++k) {
                const AttnItem it = P.items[P.sched[first + k]];
                const int n = it.kv_tile1 - it.kv_tile0;
                for (int i = 0; i < n; ++i, ++g) {
                    const int b = g % NB, sv = g % NV;
                    if (!(ok = wait_bar(bar_p_full + b, (g / NB) & 1, abort_flag, status))) break;
                    if (!(ok = wait_bar(bar_v_full + sv, (g / NV) & 1, abort_flag, status))) break;
                    // the item's first PV overwrites O: the epilogue must have read the previous item's
                    if (i == 0 && k > 0 && !(ok = wait_bar(bar_o_free, (k - 1) & 1, abort_flag, status))) break;
                    tc_fence_after();
                    const uint32_t sV = smem_u32(smem + C::OFF_V + sv * C::KV_BYTES);
                    const uint32_t pcol = tmem + C::TMEM_S + b * kAttnBN;
#pragma unroll
                    for (int kk = 0; kk < kAttnBN / 16; ++kk)
                        mma_bf16_ts(tmem + C::TMEM_O, pcol + kk * 8, sdesc_sw128(sV + kk * 16 * 128, C::ATOM_BYTES, 1024),
                                    idesc_pv, (i > 0 || kk > 0) ? 1u : 0u);
                    mma_commit(bar_o_done + b);
                    mma_commit(bar_v_empty + sv);
                }
                if (ok) mma_commit(bar_o_full);    // arrives once the item's last PV has finished
            }
            mma_commit(bar_drain + 1);
            drain_bar(bar_drain + 1, 0, status);
        }
    } else if (warp < kSoftmaxWarps) {
        // ---------------------------------------------------- softmax (warps 0-3)
        setmaxnreg_inc<kPtSoftmaxRegs>();
        int g = 0;
        for (int k = 0; k < n_mine; ++k) {
            const AttnItem it = P.items[P.sched[first + k]];
            const int n = it.kv_tile1 - it.kv_tile0;
            float m, l;
            if (!softmax_item<D, G, NB>(it, P, tmem + C::TMEM_S, tmem + C::TMEM_O, n, g, bar_s_full, bar_p_full,
                                        bar_o_done, abort_flag, status, scale_log2, m, l))
                break;
            g += n;
            // the row's m and l to the epilogue, once it has taken the previous item's
            if (!warp_wait(bar_st_empty, (k & 1) ^ 1, abort_flag, status)) break;
            st_m[threadIdx.x] = m;
            st_l[threadIdx.x] = l;
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_st_full);
        }
    } else {
        // ---------------------------------------------------- epilogue (warps 8-11)
        const int r = threadIdx.x - kPtEpiWarp0 * 32;                   // tile row == TMEM lane
        const uint32_t lane_base = (uint32_t)((warp % 4) * 32) << 16;
        for (int k = 0; k < n_mine; ++k) {
            const AttnItem it = P.items[P.sched[first + k]];
            bool ok = warp_wait(bar_o_full, k & 1, abort_flag, status);
            ok = ok && warp_wait(bar_st_full, k & 1, abort_flag, status);
            // the four epilogue warps leave together (they meet at named barriers below)
            if (named_bar_any(1, 128, !ok)) break;
            const float m = st_m[r], l = st_l[r];
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_st_empty);
            tc_fence_after();
            epilogue_item<D, G>(it, P, r, lane_base + tmem + C::TMEM_O, m, l, bar_o_free, merge_flag, out, ws, h_q);
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
    for (int idx = threadIdx.x; idx < n_rows * D; idx += blockDim.x) {
        const int r = idx % n_rows, d = idx / n_rows;   // neighbouring threads: neighbouring rows
        const float M = merge_max<D>(ws, mg.slot0, mg.n_split, r);
        const float L = merge_sum<D>(ws, mg.slot0, mg.n_split, r, M);
        const int frow = f0 + mg.tok0 + r / G;
        out[((int64_t)frow * h_q + mg.kv_head * G + (r % G)) * D + d] =
            __float2bfloat16_rn(merge_value<D>(ws, mg.slot0, mg.n_split, r, d, M, L));
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
                                const DevicePlan& P, int n_ctas, void* out, float* ws, int h_q, float scale_log2,
                                cudaStream_t stream) {
    static std::atomic<uint64_t> attr_set{0};
    cudaError_t ea = once_per_device(attr_set, [] {
        return cudaFuncSetAttribute(attn_tc_persistent_kernel<D, G>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)PtCfg<D>::SMEM_BYTES);
    });
    if (ea != cudaSuccess) return ea;
    // cut ranges are merged inside the kernel: nothing follows it
    if (n_ctas > 0)
        attn_tc_persistent_kernel<D, G><<<n_ctas, kPtThreads, PtCfg<D>::SMEM_BYTES, stream>>>(
            mq, mk, mv, P, (__nv_bfloat16*)out, ws, h_q, scale_log2);
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
// The persistent kernel over the plan's per-CTA schedule (n_ctas CTAs).
int launch_attention_tc(const DevicePlan& P, int n_items, int n_ctas, int n_merges, int n_fresh, int64_t ctx_rows,
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
    if (head_dim == DD && G == GG) e = launch_tc_dg<DD, GG>(mq, mk, mv, P, n_ctas, out, w, h_q, sl2, stream);
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
