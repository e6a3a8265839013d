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
// With zero-copy values the V warp gathers rows and keeps the next tile's records, so that
// warpgroup keeps 96 (240 + 96 + 168 = 3 x 168: the whole launch budget).
constexpr uint32_t kPtSoftmaxRegs = 240, kPtIdleRegs = 56, kPtIdleRegsZv = 96;
static_assert(kPtThreads * 168 <= 65536, "launch register budget");
static_assert(128 * (kPtSoftmaxRegs + kPtIdleRegs + 168) <= kPtThreads * 168, "register split");
static_assert(128 * (kPtSoftmaxRegs + kPtIdleRegsZv + 168) <= kPtThreads * 168, "register split (zero-copy values)");

// Shared memory: two Q buffers (the next item's Q lands while the current item runs), the K
// ring and the V ring (one stage shorter than the K ring for head_dim 128: a V tile is needed
// a softmax later than its K tile), m and l of one item, a flag, the barriers.  With zero-copy
// values (ZV) the rings trade places: the value tiles come from the pool, partly row by row,
// and need the longer lead.
template <int D, bool ZV = false>
struct PtCfg {
    static constexpr int ATOMS = D / 64;
    static constexpr int NQ = 2;
    static constexpr int NK = (D == 128) ? (ZV ? 2 : 3) : (ZV ? 4 : 5);
    static constexpr int NV = (D == 128) ? (ZV ? 3 : 2) : (ZV ? 5 : 4);
    static constexpr int NB = 3;
    static constexpr uint32_t ATOM_BYTES = 128 * 128;
    static constexpr uint32_t Q_BYTES = ATOMS * ATOM_BYTES, KV_BYTES = ATOMS * ATOM_BYTES;
    static constexpr uint32_t OFF_Q = 0;                                // two buffers
    static constexpr uint32_t OFF_K = OFF_Q + NQ * Q_BYTES;
    static constexpr uint32_t OFF_V = OFF_K + NK * KV_BYTES;
    static constexpr uint32_t OFF_STATS = OFF_V + NV * KV_BYTES;        // m[128], l[128] of one item
    static constexpr uint32_t OFF_FLAG = OFF_STATS + 2 * kAttnBM * 4;   // the epilogue's merge decision
    static constexpr uint32_t OFF_BAR = OFF_FLAG + 16;
    // q_full[NQ], q_empty[NQ], k_full[NK], k_empty[NK], v_full[NV], v_empty[NV], s_full[NB],
    // p_full[NB], o_done[NB], o_full, o_free, st_full, st_empty, drain x2
    static constexpr int N_BARS = 2 * NQ + 2 * NK + 2 * NV + 3 * NB + 6;
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

// Zero-copy values: the V tiles are read where the values are (the pool's rows for the prefix
// and document positions, v_new for the fresh rows) in the cache-row order of the key tiles,
// so the linked cache needs no value rows.  The whole V warp runs it.  Per 8 cache rows the
// plan's group table says whether their sources are 8 consecutive rows of one tensor; those
// groups are TMA copies landing 1024-byte aligned in the 128-byte swizzled layout the PV MMA
// reads, a run of groups that continue one another in naturally aligned boxes of 8 to 128 rows
// (lane = group + 16 x atom; the first group of a box issues it).  The rows of the other groups
// (a segment boundary inside, or past the query's end) the warp copies 16 bytes at a time with
// cp.async (lane = 16-byte chunk of a row), or zero-fills.
// The warp keeps the tables a tile ahead: the items' entries 32 at a time (one item per lane),
// and the group entries and source records of the next tile, loaded while the current tile is
// issued and first used a tile later.  Per tile it issues the row copies first and the boxes
// second; lane 0 raises the stage's byte count for the boxes before they are issued.  A stage
// without row copies is published at once (lane 0 arrives; the boxes complete it).  A stage with
// row copies is published after the next tile has been issued, when its copies have landed:
// every lane waits for them and fences them into the async proxy, then lane 0 arrives.  That
// arrival waits for the next stage to come free, i.e. for the PV MMA NV - 1 tiles back, so the
// value ring is deeper here (NV >= 3) than with a linked value cache.  (With two stages the
// deferred arrival made each PV MMA wait for the one before it; publishing only after the
// copies' own latency left each stage a copy latency late.)
struct PoolValues {
    const __nv_bfloat16* pool_v;   // [pool_rows][h_kv][D]
    const __nv_bfloat16* v_new;    // [n_fresh][h_kv][D]
    int h_kv;
};

// Source tensors of the value copies: boxes of 8 << h rows (h = 0..4: 8 to 128 rows) over the
// pool (src 0) and v_new (src 1).  Passed as one kernel parameter.
constexpr int kVBoxSizes = 5;
struct ValueMaps {
    CUtensorMap m[2][kVBoxSizes];
};

template <int D, int NV>
__device__ __forceinline__ void pool_values_role(const DevicePlan& P, const PoolValues& V, const ValueMaps* M,
                                                 uint8_t* smem_v, int first, int n_mine, uint64_t* bar_v_full,
                                                 uint64_t* bar_v_empty, volatile int32_t* abort_flag,
                                                 int32_t* status) {
    constexpr int ATOMS = D / 64;
    constexpr uint32_t ATOM_BYTES = 128 * 128, KV_BYTES = ATOMS * ATOM_BYTES, GROUP_BYTES = ATOMS * 8 * 128;
    constexpr int N_GRP = kAttnBN / 8;      // 16 groups per tile
    constexpr int CPR = D / 8;              // 16-byte chunks per row
    constexpr int RPP = 32 / CPR;           // rows per warp pass
    constexpr int RPL = kAttnBN / 32;       // records per lane
    static_assert(N_GRP * ATOMS <= 32 && 8 % RPP == 0 && N_GRP == 16, "V warp split");
    const int lane = threadIdx.x % 32, ch = lane % CPR;
    const uint32_t v_base = smem_u32(smem_v);
    const int64_t row_elems = (int64_t)V.h_kv * D;

    // The tables of this CTA's items, one item per lane, 32 items per load: an item's entry
    // (its schedule index, then the item, then its query's offsets) is a chain of dependent
    // loads, paid once per 32 items instead of at every item change.
    int l_head = 0, l_t0 = 0, l_n = 0, l_a = 0, l_b = 0, l_npos = 0, l_gbase = 0, l_ngrp = 0;
    int64_t l_ctx0 = 0;
    auto load_items = [&](int k0) {
        const int k = k0 + lane;
        if (k < n_mine) {
            const AttnItem it = P.items[P.sched[first + k]];
            l_head = it.kv_head;
            l_t0 = it.kv_tile0;
            l_n = it.kv_tile1 - it.kv_tile0;
            l_a = it.a_tiles;
            l_b = it.b_tile0;
            l_ctx0 = P.cu_ctx[it.query];
            l_npos = (int)(P.cu_ctx[it.query + 1] - l_ctx0);
            l_gbase = P.cu_grp[it.query];
            l_ngrp = P.cu_grp[it.query + 1] - l_gbase;
        }
    };
    // the tile after the current one: tile jn of item kn, and what the warp loaded for it (raw:
    // the loads are first used a tile later, so their latency overlaps the current tile)
    int kn = 0, jn = 0;
    int headn = 0, t0n = 0, nn = 0, an = 0, bn = 0, n_posn = 0, gbasen = 0, n_grpn = 0;
    int64_t ctx0n = 0;
    int key0n = 0;
    int32_t gwn = -1;
    int2 srcn[RPL];
    auto item_info = [&](int k) {
        if (k % 32 == 0) load_items(k);
        const int src = k % 32;
        headn = __shfl_sync(0xffffffffu, l_head, src);
        t0n = __shfl_sync(0xffffffffu, l_t0, src);
        nn = __shfl_sync(0xffffffffu, l_n, src);
        an = __shfl_sync(0xffffffffu, l_a, src);
        bn = __shfl_sync(0xffffffffu, l_b, src);
        ctx0n = __shfl_sync(0xffffffffu, l_ctx0, src);
        n_posn = __shfl_sync(0xffffffffu, l_npos, src);
        gbasen = __shfl_sync(0xffffffffu, l_gbase, src);
        n_grpn = __shfl_sync(0xffffffffu, l_ngrp, src);
    };
    // group entries and source records (kind, row; row -1 past the query's end) of tile jn
    auto prefetch = [&]() {
        const int v = t0n + jn;   // the item's key-tile list entry (item_tile)
        key0n = (v < an ? v : bn + (v - an)) * kAttnBN;
        const int m0 = key0n / 8;
        gwn = -1;
        if (lane < N_GRP && m0 + lane < n_grpn) gwn = __ldg(P.grp_src + gbasen + m0 + lane);
#pragma unroll
        for (int t = 0; t < RPL; ++t) {
            const int pos = key0n + lane + 32 * t;
            srcn[t] = make_int2(0, -1);
            if (pos < n_posn) srcn[t] = __ldg(reinterpret_cast<const int2*>(P.src_row + ctx0n + pos));
        }
    };

    bool have = n_mine > 0;
    if (have) {
        item_info(0);
        prefetch();
    }
    int g = 0;                 // tiles issued
    bool pend = false;         // tile g - 1 has row copies and is not yet published
    static_assert(NV >= 3, "the deferred publication needs three value stages");
    while (have) {
        // the current tile is the prefetched one
        const int kv_head = headn;
        int32_t gw = gwn;
        int32_t rec[RPL];      // kGrpFresh | row, or -1 (zero-filled)
#pragma unroll
        for (int t = 0; t < RPL; ++t) {
            const int2 e = srcn[t];
            rec[t] = e.y < 0 ? -1 : (e.y | (e.x == KVLINK_SRC_FRESH ? kGrpFresh : 0));
#ifdef KVLINK_DEBUG_CHECKS
            if (e.y >= (e.x == KVLINK_SRC_FRESH ? (int64_t)P.n_fresh : P.pool_rows)) {
                atomicCAS(status, 0, kAttnStatusBadIndex);
                rec[t] = -1;   // zero-filled instead
            }
#endif
        }
#ifdef KVLINK_DEBUG_CHECKS
        if (gw >= 0 && (gw & kGrpRowMask) + 8 > ((gw & kGrpFresh) ? (int64_t)P.n_fresh : P.pool_rows)) {
            atomicCAS(status, 0, kAttnStatusBadIndex);
            gw = -1;   // its rows take the per-row path, whose records are checked above
        }
#endif
        // advance and start the next tile's loads
        if (++jn >= nn) {
            jn = 0;
            if (++kn < n_mine) item_info(kn);
            else have = false;
        }
        if (have) prefetch();

        const int st = g % NV;
        if (!warp_wait(bar_v_empty + st, ((g / NV) & 1) ^ 1, abort_flag, status)) break;
        const uint32_t by_tma = __ballot_sync(0xffffffffu, gw >= 0);   // lanes >= N_GRP hold -1
        const uint32_t by_row = ~by_tma & ((1u << N_GRP) - 1);
        // Runs of groups whose rows continue one another go in naturally aligned boxes of 1, 2,
        // 4, 8 or 16 groups: a block of 2^h groups starting at a multiple of 2^h is one box when
        // every group in it is a TMA group and each continues the one before.
        const int32_t prev = __shfl_up_sync(0xffffffffu, gw, 1);
        const uint32_t cont = __ballot_sync(0xffffffffu, lane < N_GRP && lane > 0 && gw >= 0 && gw == prev + 8);
        // the row copies first (one commit group per tile), then the boxes
        const uint32_t sv_addr = v_base + st * KV_BYTES;
        const int64_t col = (int64_t)kv_head * D + 8 * ch;   // this lane's chunk within a row
        for (uint32_t rest = by_row; rest != 0; rest &= rest - 1) {
            const int m = __ffs(rest) - 1;
#pragma unroll
            for (int p = 0; p < 8 / RPP; ++p) {
                const int r0 = m * 8 + p * RPP;          // a multiple of RPP: the rows' records
                const int t = r0 / 32;                   // sit in slot t of every lane
                int32_t mine = rec[0];
#pragma unroll
                for (int u = 1; u < RPL; ++u)
                    if (t == u) mine = rec[u];
                const int r = r0 + lane / CPR;
                const int32_t e = __shfl_sync(0xffffffffu, mine, r % 32);
                const uint32_t dst =
                    sv_addr + (uint32_t)(ch >> 3) * ATOM_BYTES + (uint32_t)r * 128u + ((uint32_t)((ch & 7) ^ (r & 7)) << 4);
                if (e >= 0)
                    cp_async16(dst, ((e & kGrpFresh) ? V.v_new : V.pool_v) + (int64_t)(e & kGrpRowMask) * row_elems + col);
                else
                    st_shared_zero16(dst);
            }
        }
        cp_async_commit();
        uint8_t* sv = smem_v + st * KV_BYTES;
        if (lane == 0) mbar_expect_tx(bar_v_full + st, (uint32_t)__popc(by_tma) * GROUP_BYTES);
        __syncwarp();
        {
            const int m = lane % N_GRP, a = lane / N_GRP;
            // the largest whole block holding group m
            int h = 0;
#pragma unroll
            for (int hh = 1; hh < kVBoxSizes; ++hh) {
                const int n = 1 << hh, b0 = m & ~(n - 1);
                const uint32_t blk = ((1u << n) - 1u) << b0;
                const uint32_t inner = blk & ~(1u << b0);         // groups that must continue
                if ((by_tma & blk) == blk && (cont & inner) == inner) h = hh;
            }
            const int32_t gm = __shfl_sync(0xffffffffu, gw, m);
            if (a < ATOMS && gm >= 0 && (m & ((1 << h) - 1)) == 0)
                tma_load_3d(sv + a * ATOM_BYTES + m * 8 * 128, &M->m[(gm & kGrpFresh) ? 1 : 0][h], a * 64, kv_head,
                            gm & kGrpRowMask, bar_v_full + st);
        }
        // The previous tile's row copies have had this tile's issue time to land: publish that
        // stage (fence into the async proxy, lane 0 arrives); a tile without row copies is
        // published at once.  With NV >= 3 stages the deferred arrival waits only for the PV MMA
        // NV - 1 tiles back, which its own PV follows anyway.
        if (pend) {
            cp_async_wait<1>();
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_v_full + (g - 1) % NV);
        }
        pend = by_row != 0;
        if (!pend) {
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_v_full + st);
        }
        ++g;
    }
    if (pend) {
        cp_async_wait<0>();
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(bar_v_full + (g - 1) % NV);
    }
    // no copy may still be in flight when the CTA leaves
    if (lane == 0)
        for (int gg = g - NV > 0 ? g - NV : 0; gg < g; ++gg) drain_bar(bar_v_full + gg % NV, (gg / NV) & 1, status);
}

template <int D, int G, bool ZV>
__global__ void __launch_bounds__(kPtThreads, 1)
    attn_tc_persistent_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                              const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ ValueMaps vmaps,
                              DevicePlan P, const PoolValues V, __nv_bfloat16* __restrict__ out,
                              float* __restrict__ ws, int h_q, float scale_log2) {
    using C = PtCfg<D, ZV>;
    constexpr int NK = C::NK, NV = C::NV, NB = C::NB;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw_addr = smem_u32(smem_raw);
    uint8_t* smem = smem_raw + ((1024u - (raw_addr & 1023u)) & 1023u);

    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);
    constexpr int NQ = C::NQ;
    uint64_t* bar_q_full = bars;                 // [NQ]
    uint64_t* bar_q_empty = bar_q_full + NQ;     // [NQ]
    uint64_t* bar_k_full = bar_q_empty + NQ;
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
        if (ZV)
            for (int i = 0; i < 2 * kVBoxSizes; ++i) prefetch_tensormap(&vmaps.m[i / kVBoxSizes][i % kVBoxSizes]);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_holder;
    // Launched as a programmatic dependent of the kernel before it on the stream (the fresh-row
    // placement in the step): the prologue above overlaps that kernel; nothing it writes is read
    // before this wait.
    asm volatile("griddepcontrol.wait;" ::: "memory");
    const bool skip = *abort_flag != 0;  // written before the barrier: uniform across the CTA

    if (skip) {
        // nothing issued: fall through to the teardown
    } else if (warp >= kSoftmaxWarps && warp < kPtEpiWarp0) {
        setmaxnreg_dec<ZV ? kPtIdleRegsZv : kPtIdleRegs>();
        if (warp == kTmaKWarp && lane == 0) {
            // ------------------------------------------------ Q of every item, and the K ring
            int g = 0, q_issued = 0;
            bool ok = true;
            for (int k = 0; ok && k < n_mine; ++k) {
                const AttnItem it = P.items[P.sched[first + k]];
                const int n = it.kv_tile1 - it.kv_tile0, ctx0 = (int)P.cu_ctx[it.query];
                // Q buffer k % NQ, once the S MMAs of item k - NQ have read it
                const int qb = k % NQ;
                if (!(ok = wait_bar(bar_q_empty + qb, ((k / NQ) & 1) ^ 1, abort_flag, status))) break;
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
            for (int k = q_issued - NQ > 0 ? q_issued - NQ : 0; k < q_issued; ++k)
                drain_bar(bar_q_full + k % NQ, (k / NQ) & 1, status);
        } else if (warp == kTmaVWarp && ZV) {
            // ------------------------------------------------ the V ring, values where they are
            if constexpr (ZV)
                pool_values_role<D, NV>(P, V, &vmaps, smem + C::OFF_V, first, n_mine, bar_v_full, bar_v_empty,
                                        abort_flag, status);
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
                const int qb = k % NQ;
                if (!(ok = wait_bar(bar_q_full + qb, (k / NQ) & 1, abort_flag, status))) break;
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

template <int D, int G, bool ZV>
static cudaError_t launch_tc_dg(const CUtensorMap& mq, const CUtensorMap& mk, const CUtensorMap& mv,
                                const ValueMaps& vm, const DevicePlan& P, const PoolValues& V, int n_ctas, void* out,
                                float* ws, int h_q, float scale_log2, cudaStream_t stream) {
    static std::atomic<uint64_t> attr_set{0};
    cudaError_t ea = once_per_device(attr_set, [] {
        return cudaFuncSetAttribute(attn_tc_persistent_kernel<D, G, ZV>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)PtCfg<D, ZV>::SMEM_BYTES);
    });
    if (ea != cudaSuccess) return ea;
    // cut ranges are merged inside the kernel: nothing follows it.  Programmatic stream
    // serialization: the launch may begin while the kernel before it finishes (the kernel waits
    // for it with griddepcontrol.wait after its prologue): 431.2 -> 429.7 us/query on the
    // 32-layer step of the Llama-8B batch-8 workload, 416.2 -> 406.7 with zero-copy values.
    if (n_ctas > 0) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3((unsigned)n_ctas);
        cfg.blockDim = dim3(kPtThreads);
        cfg.dynamicSmemBytes = PtCfg<D, ZV>::SMEM_BYTES;
        cfg.stream = stream;
        cudaLaunchAttribute at[1];
        at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        at[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = at;
        cfg.numAttrs = 1;
        const cudaError_t le = cudaLaunchKernelEx(&cfg, attn_tc_persistent_kernel<D, G, ZV>, mq, mk, mv, vm, P, V,
                                                  (__nv_bfloat16*)out, ws, h_q, scale_log2);
        if (le != cudaSuccess) return le;
    }
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
// The persistent kernel over the plan's per-CTA schedule (n_ctas CTAs); values from the linked
// cache (vs.cache_v), or where they are (vs.cache_v NULL: vs.pool_v and vs.v_new, through
// 8-row TMA boxes).
int launch_attention_tc(const DevicePlan& P, int n_items, int n_ctas, int n_merges, int n_fresh, int64_t ctx_rows,
                        int head_dim, int h_q, int h_kv, const void* q, const void* cache_k, const ValueSource& vs,
                        void* out, void* ws, cudaStream_t stream, cudaError_t* err) {
    const int G = h_q / h_kv;
    const bool zv = vs.cache_v == nullptr;
    CUtensorMap mq, mk, mv;      // values: the linked cache (zero-copy values: vm)
    ValueMaps vm{};              // zero-copy values: pool / v_new in boxes of 8 .. 128 rows
    const uint32_t box_tok = (uint32_t)(kAttnBM / G);
    if (!make_map_3d(&mq, q, (uint64_t)head_dim, (uint64_t)h_q, (uint64_t)n_fresh, 64, (uint32_t)G, box_tok) ||
        !make_map_3d(&mk, cache_k, (uint64_t)head_dim, (uint64_t)h_kv, (uint64_t)ctx_rows, 64, 1, kAttnBN))
        return KVLINK_EUNSUPPORTED;
    if (!zv) {
        if (!make_map_3d(&mv, vs.cache_v, (uint64_t)head_dim, (uint64_t)h_kv, (uint64_t)ctx_rows, 64, 1, kAttnBN))
            return KVLINK_EUNSUPPORTED;
    } else {
        mv = mk;   // unused
        const uint64_t D = (uint64_t)head_dim, H = (uint64_t)h_kv;
        const uint64_t rows[2] = {(uint64_t)P.pool_rows, (uint64_t)n_fresh};
        const void* base[2] = {vs.pool_v, vs.v_new};
        for (int src = 0; src < 2; ++src)
            for (int h = 0; h < kVBoxSizes; ++h)
                if (!make_map_3d(&vm.m[src][h], base[src], D, H, rows[src], 64, 1, 8u << h)) return KVLINK_EUNSUPPORTED;
    }
    const PoolValues V{(const __nv_bfloat16*)vs.pool_v, (const __nv_bfloat16*)vs.v_new, h_kv};
    const float sl2 = 1.4426950408889634f / sqrtf((float)head_dim);
    float* w = (float*)ws;
    cudaError_t e = cudaErrorInvalidValue;
#define KVLINK_TC_CASE(DD, GG)                                                                              \
    if (head_dim == DD && G == GG)                                                                          \
        e = zv ? launch_tc_dg<DD, GG, true>(mq, mk, mv, vm, P, V, n_ctas, out, w, h_q, sl2, stream)         \
               : launch_tc_dg<DD, GG, false>(mq, mk, mv, vm, P, V, n_ctas, out, w, h_q, sl2, stream);
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
