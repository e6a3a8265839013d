// Pieces shared by the two tensor-core attention kernels (the suffix attention over a
// materialised linked cache, and the fused linked prefill): bounded mbarrier waits,
// the softmax + epilogue role, and the FMA-pipe 2^x.
//
// The softmax role (Sec. 2.3 attention of the fresh rows; online softmax over KV
// tiles): 4 warps, thread r owns tile row r = TMEM lane r.  For every KV tile j it
// reads S_j from TMEM buffer j % NB, masks keys whose position is above the row's
// position, raises the running max (rescaling O in TMEM only when the max grew by
// more than 2^8), writes P_j = exp2(S_j c - m) as bf16 over the first half of the
// same buffer and signals the MMA thread.  Keys are visited in cache-row order.  At the end it normalises O and stores the output rows, or
// stores the unnormalised partial (O, m, l) when the item's KV range was split.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "kvlink_internal.h"
#include "kvlink_sm100.cuh"

namespace kvlink {

constexpr uint64_t kWaitLimitNs = 2000000000ull;  // 2 s
constexpr int32_t kAttnStatusWaitTimeout = 0x41;
constexpr int32_t kAttnStatusBadIndex = 0x42;    // KVLINK_DEBUG_CHECKS: a table entry out of bounds

// Whether a work item lies inside the plan's tables (checked by the KVLINK_DEBUG_CHECKS build
// before any access through the item).  Key-tile rows past a query's cache are read as zeros
// by TMA, so only the plan's own indices need checking.
__device__ __forceinline__ bool item_in_bounds(const AttnItem& it, const DevicePlan& P) {
    if (it.query < 0 || it.query >= P.batch || it.kv_head < 0 || it.kv_head >= P.h_kv) return false;
    const int n_fresh_q = P.cu_fresh[it.query + 1] - P.cu_fresh[it.query];
    if (it.tok0 < 0 || it.tok0 >= it.tok1 || it.tok1 > n_fresh_q) return false;
    if (it.kv_tile0 < 0 || it.kv_tile1 < it.kv_tile0 || it.a_tiles < 0 || it.b_tile0 < 0) return false;
    if (it.slot < -1 || it.slot >= P.n_slots) return false;
    return true;
}
constexpr float kRescaleThreshold = 8.0f;         // log2 units: rescale O when the max grows by > 2^8
#ifndef KVLINK_EXP_POLY_FROM
#define KVLINK_EXP_POLY_FROM 8                     // column pairs c with (c % 8) >= this use exp2_poly2
#endif

constexpr uint32_t kTmemCols = 512;

// Wait for phase `parity` of `bar`; false if another role aborted or the time limit passed.
__device__ __forceinline__ bool wait_bar(uint64_t* bar, uint32_t parity, volatile int32_t* abort_flag,
                                         int32_t* status, uint64_t limit_ns = kWaitLimitNs) {
    if (sm100::mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = sm100::globaltimer_ns();
    while (true) {
        if (sm100::mbar_try_wait(bar, parity)) return true;
        if (*abort_flag) return false;
        if (sm100::globaltimer_ns() - t0 > limit_ns) {
            *abort_flag = 1;
            atomicCAS(status, 0, kAttnStatusWaitTimeout);
            return false;
        }
    }
}

// Same, but ignores the abort flag: used to drain this thread's own async work.
__device__ __forceinline__ void drain_bar(uint64_t* bar, uint32_t parity, int32_t* status) {
    const uint64_t t0 = sm100::globaltimer_ns();
    while (!sm100::mbar_try_wait(bar, parity)) {
        if (sm100::globaltimer_ns() - t0 > kWaitLimitNs) {
            atomicCAS(status, 0, kAttnStatusWaitTimeout);
            return;
        }
    }
}

// All lanes wait; the warp proceeds only if every lane saw the phase complete.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int32_t* abort_flag,
                                          int32_t* status) {
    const bool ok = wait_bar(bar, parity, abort_flag, status);
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
    using namespace sm100;
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

// Softmax over the key tiles of one item, run by warps 0-3 (threadIdx.x = tile row).  TMEM
// holds NB S/P buffers of kAttnBN columns from column tmem_s and the O accumulator at tmem_o.
// g0 is the running count of key tiles before this item's first one: a kernel that runs
// several items one after another keeps its S buffers and barrier phases going across them
// (tile j of the item uses buffer (g0 + j) % NB).  O is touched only to rescale it, after the
// item's previous PV has finished.  Leaves the row's running max m (log2 units) and sum l.
template <int D, int G, int NB>
__device__ __forceinline__ bool softmax_item(const AttnItem& it, const DevicePlan& P, uint32_t tmem_s,
                                             uint32_t tmem_o, int n_tiles, int g0, uint64_t* bar_s_full,
                                             uint64_t* bar_p_full, uint64_t* bar_o_done,
                                             volatile int32_t* abort_flag, int32_t* status, float scale_log2,
                                             float& m_out, float& l_out) {
    using namespace sm100;
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int r = threadIdx.x;  // tile row == TMEM lane
    const int tok = it.tok0 + r / G;
    const bool valid = tok < it.tok1;
    const int frow = P.cu_fresh[it.query] + tok;
    // visible cache rows (query-relative): [0, vis_a) and [F, F + vis_b)
    const int vis_a = valid ? P.fresh_vis[frow] : 0x7fffffff;
    const int F = P.fresh_row0[it.query];
    const uint32_t vis_b = valid ? (uint32_t)(tok + 1) : 0u;
    const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
    float m = -INFINITY, l = 0.f;
    for (int j = 0; j < n_tiles; ++j) {
        const int g = g0 + j;
        const int b = g % NB;
        if (!warp_wait(bar_s_full + b, (g / NB) & 1, abort_flag, status)) return false;
        tc_fence_after();
        uint32_t s[128];
        const uint32_t s_col = lane_base + tmem_s + b * kAttnBN;
        tmem_ld32(s_col + 0, *reinterpret_cast<uint32_t(*)[32]>(s + 0));
        tmem_ld32(s_col + 32, *reinterpret_cast<uint32_t(*)[32]>(s + 32));
        tmem_ld32(s_col + 64, *reinterpret_cast<uint32_t(*)[32]>(s + 64));
        tmem_ld32(s_col + 96, *reinterpret_cast<uint32_t(*)[32]>(s + 96));
        tmem_ld_wait();

        // raw row max (scale > 0 commutes with max).  A tile lies in one run of rows (cached
        // rows, or the fresh rows at the end), where a row sees the keys below one limit, so
        // for each row the tile is fully visible, fully masked, or holds the row's limit.
        // Only the last case needs a per-column select (a compare and select per column
        // cost ~800 cycles a tile on the softmax warps), and a warp takes that path only
        // when one of its rows has its limit in the tile; a fully masked row instead drops
        // its max and gets p = 0 from an infinite exponent offset.  Only a tile holding the
        // end of the cached rows and the start of the fresh rows compares twice per column.
        const int key0 = item_tile(it, it.kv_tile0 + j) * kAttnBN;
        float mx8[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) mx8[e] = -INFINITY;
        constexpr uint32_t kNegInf = 0xff800000u;
        bool dead = false;  // the row sees no key of this tile
        bool plain = true;
        if (key0 + kAttnBN > it.min_vis) {  // some row of the tile may not see every key
            if (key0 + kAttnBN <= F || key0 >= F) {
                const int nv = (key0 >= F ? F + (int)vis_b : vis_a) - key0;  // columns [0, nv) visible
                dead = nv <= 0;
                if (__any_sync(0xffffffffu, nv > 0 && nv < kAttnBN)) {
                    plain = false;
#pragma unroll
                    for (int c = 0; c < 128; ++c) {
                        s[c] = c < nv ? s[c] : kNegInf;
                        mx8[c & 7] = fmaxf(mx8[c & 7], __uint_as_float(s[c]));
                    }
                }
            } else {
                plain = false;
#pragma unroll
                for (int c = 0; c < 128; ++c) {
                    const int kr = key0 + c;
                    if (!(kr < vis_a || (uint32_t)(kr - F) < vis_b)) s[c] = kNegInf;
                    mx8[c & 7] = fmaxf(mx8[c & 7], __uint_as_float(s[c]));
                }
            }
        }
        if (plain) {
#pragma unroll
            for (int c = 0; c < 128; ++c) mx8[c & 7] = fmaxf(mx8[c & 7], __uint_as_float(s[c]));
        }
        const float mx = dead ? -INFINITY
                              : fmaxf(fmaxf(fmaxf(mx8[0], mx8[1]), fmaxf(mx8[2], mx8[3])),
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
            if (!warp_wait(bar_o_done + (g - 1) % NB, ((g - 1) / NB) & 1, abort_flag, status)) return false;
            tc_fence_after();
#pragma unroll
            for (int c4 = 0; c4 < D / 32; ++c4) {
                uint32_t o[32];
                const uint32_t o_col = lane_base + tmem_o + c4 * 32;
                tmem_ld32(o_col, o);
                tmem_ld_wait();
#pragma unroll
                for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
                tmem_st32(o_col, o);
            }
        }
        // p = exp2(s * scale - m) on column pairs (packed f32x2 arithmetic); pairs with
        // (c % 8) >= KVLINK_EXP_POLY_FROM go to the FMA pipe (exp2_poly2), the rest to MUFU
        // a fully masked row: s * scale - inf = -inf, so every p is 0
        const float mu = dead ? INFINITY : ((m == -INFINITY) ? 0.f : m);
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
                float a, bb;
                f2_unpack(x2, a, bb);
                p2 = f2_pack(ex2_approx(a), ex2_approx(bb));
            }
            acc[c & 3] = fadd2(acc[c & 3], p2);
            float p0, p1;
            f2_unpack(p2, p0, p1);
            pk[c] = pack2_bf16(p0, p1);
        }
        float rs0, rs1;
        f2_unpack(fadd2(fadd2(acc[0], acc[1]), fadd2(acc[2], acc[3])), rs0, rs1);
        l += rs0 + rs1;
        // P_j (bf16) over the first 64 columns of its S buffer, read there by the PV MMA
        tmem_st32(s_col + 0, *reinterpret_cast<uint32_t(*)[32]>(pk + 0));
        tmem_st32(s_col + 32, *reinterpret_cast<uint32_t(*)[32]>(pk + 32));
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(bar_p_full + b);
    }
    m_out = m;
    l_out = l;
    return true;
}

// Row r of an item's result from the values o[] of its O row: the output row normalised by
// l (bf16), or, for an item whose KV range was split, the unnormalised partial (O, m, l).
template <int D, int G>
__device__ __forceinline__ void store_result(const AttnItem& it, const DevicePlan& P, int r, const uint32_t* o,
                                             int c0, int nc, float m, float l, __nv_bfloat16* __restrict__ out,
                                             float* __restrict__ ws, int h_q) {
    const int tok = it.tok0 + r / G;
    if (it.slot < 0) {
        if (tok >= it.tok1) return;
        const float inv = 1.f / l;
        const int frow = P.cu_fresh[it.query] + tok;
        __nv_bfloat16* orow = out + ((int64_t)frow * h_q + it.kv_head * G + (r % G)) * D + c0;
        for (int q = 0; q < nc / 8; ++q) {
            uint4 w;
            w.x = pack2_bf16(__uint_as_float(o[8 * q + 0]) * inv, __uint_as_float(o[8 * q + 1]) * inv);
            w.y = pack2_bf16(__uint_as_float(o[8 * q + 2]) * inv, __uint_as_float(o[8 * q + 3]) * inv);
            w.z = pack2_bf16(__uint_as_float(o[8 * q + 4]) * inv, __uint_as_float(o[8 * q + 5]) * inv);
            w.w = pack2_bf16(__uint_as_float(o[8 * q + 6]) * inv, __uint_as_float(o[8 * q + 7]) * inv);
            *reinterpret_cast<uint4*>(orow + 8 * q) = w;
        }
    } else {
        // column-major [D][kAttnBM]: the 32 rows of a warp write 128 contiguous bytes per column
        float* wo = ws + (int64_t)it.slot * kAttnBM * (D + 2);
        for (int e = 0; e < nc; ++e) wo[(c0 + e) * kAttnBM + r] = __uint_as_float(o[e]);
        if (c0 == 0) {
            wo[kAttnBM * D + r] = m;
            wo[kAttnBM * D + kAttnBM + r] = l;
        }
    }
}

// Merge of the partial results (O, m, l) of one split KV range, row r (Sec. 2.3 attention
// computed over disjoint key ranges and combined): with M = max_s m_s and f_s = 2^(m_s - M),
// out = sum_s O_s f_s * (1 / sum_s l_s f_s), summed in slot order.  O_s is column-major:
// element (r, d) of a slot at d * kAttnBM + r.  The separate merge kernel and
// the persistent attention's in-kernel merge both use these, so they give the same bits.
// Partials are read through L2 (ld.global.cg): another CTA may have written them.
template <int D>
__device__ __forceinline__ float merge_max(const float* ws, int slot0, int n, int r) {
    const int64_t slot_floats = (int64_t)kAttnBM * (D + 2);
    float M = -INFINITY;
#pragma unroll 4
    for (int s = 0; s < n; ++s) M = fmaxf(M, __ldcg(ws + (slot0 + s) * slot_floats + kAttnBM * D + r));
    return M;
}
template <int D>
__device__ __forceinline__ float merge_factor(const float* ws, int slot, int r, float M) {
    const float ms = __ldcg(ws + (int64_t)slot * kAttnBM * (D + 2) + kAttnBM * D + r);
    return (ms == -INFINITY) ? 0.f : sm100::ex2_approx(ms - M);
}
template <int D>
__device__ __forceinline__ float merge_sum(const float* ws, int slot0, int n, int r, float M) {
    float L = 0.f;
#pragma unroll 4
    for (int s = 0; s < n; ++s)
        L = __fmaf_rn(__ldcg(ws + (int64_t)(slot0 + s) * kAttnBM * (D + 2) + kAttnBM * D + kAttnBM + r),
                      merge_factor<D>(ws, slot0 + s, r, M), L);
    return L;
}
template <int D>
__device__ __forceinline__ float merge_value(const float* ws, int slot0, int n, int r, int d, float M, float L) {
    float O = 0.f;
    for (int s = 0; s < n; ++s)
        O = __fmaf_rn(__ldcg(ws + (int64_t)(slot0 + s) * kAttnBM * (D + 2) + d * kAttnBM + r),
                      merge_factor<D>(ws, slot0 + s, r, M), O);
    return __fmul_rn(O, __frcp_rn(L));
}

// Row r of a merge group's output, written as bf16 to orow, with the arithmetic of
// merge_value (the same factors, the same fused multiply-adds in slot order, the same
// reciprocal).  Built for latency: the partials are column-major, so the 32 rows of a warp
// read 128 contiguous bytes per column, and each 32-column chunk issues the loads of two
// slots (their m and 32 values each) before any arithmetic.
template <int D>
__device__ __noinline__ void merge_row_store(const float* ws, int slot0, int n, int r,
                                             __nv_bfloat16* __restrict__ orow) {
    const float M = merge_max<D>(ws, slot0, n, r);
    const float inv = __frcp_rn(merge_sum<D>(ws, slot0, n, r, M));
    const int64_t slot_floats = (int64_t)kAttnBM * (D + 2);
    for (int c0 = 0; c0 < D; c0 += 32) {
        float acc[32];
#pragma unroll
        for (int e = 0; e < 32; ++e) acc[e] = 0.f;
        for (int s0 = 0; s0 < n; s0 += 2) {
            const bool two = s0 + 1 < n;
            const float* w0 = ws + (slot0 + s0) * slot_floats;
            const float* w1 = two ? w0 + slot_floats : w0;
            const float m0 = __ldcg(w0 + kAttnBM * D + r), m1 = __ldcg(w1 + kAttnBM * D + r);
            float v0[32], v1[32];
#pragma unroll
            for (int e = 0; e < 32; ++e) {
                v0[e] = __ldcg(w0 + (c0 + e) * kAttnBM + r);
                v1[e] = __ldcg(w1 + (c0 + e) * kAttnBM + r);
            }
            const float f0 = (m0 == -INFINITY) ? 0.f : sm100::ex2_approx(m0 - M);
            const float f1 = (m1 == -INFINITY) ? 0.f : sm100::ex2_approx(m1 - M);
#pragma unroll
            for (int e = 0; e < 32; ++e) {
                acc[e] = __fmaf_rn(v0[e], f0, acc[e]);
                if (two) acc[e] = __fmaf_rn(v1[e], f1, acc[e]);
            }
        }
#pragma unroll
        for (int h = 0; h < 4; ++h) {
            uint4 w;
            w.x = pack2_bf16(__fmul_rn(acc[8 * h + 0], inv), __fmul_rn(acc[8 * h + 1], inv));
            w.y = pack2_bf16(__fmul_rn(acc[8 * h + 2], inv), __fmul_rn(acc[8 * h + 3], inv));
            w.z = pack2_bf16(__fmul_rn(acc[8 * h + 4], inv), __fmul_rn(acc[8 * h + 5], inv));
            w.w = pack2_bf16(__fmul_rn(acc[8 * h + 6], inv), __fmul_rn(acc[8 * h + 7], inv));
            *reinterpret_cast<uint4*>(orow + c0 + 8 * h) = w;
        }
    }
}

// Softmax + epilogue role of the one-item-per-CTA kernels, run by warps 0-3: the item's
// tiles, then (once its last PV has finished) its result from O in TMEM.
template <int D, int G, int NB>
__device__ __forceinline__ void softmax_role(const AttnItem& it, const DevicePlan& P, uint32_t tmem_s,
                                             uint32_t tmem_o, int n_tiles, uint64_t* bar_s_full,
                                             uint64_t* bar_p_full, uint64_t* bar_o_done,
                                             volatile int32_t* abort_flag, int32_t* status,
                                             __nv_bfloat16* __restrict__ out, float* __restrict__ ws, int h_q,
                                             float scale_log2) {
    using namespace sm100;
    float m, l;
    if (!softmax_item<D, G, NB>(it, P, tmem_s, tmem_o, n_tiles, 0, bar_s_full, bar_p_full, bar_o_done, abort_flag,
                                status, scale_log2, m, l))
        return;
    if (n_tiles > 0 &&
        !warp_wait(bar_o_done + (n_tiles - 1) % NB, ((n_tiles - 1) / NB) & 1, abort_flag, status))
        return;
    tc_fence_after();
    const int r = threadIdx.x;
    const uint32_t lane_base = (uint32_t)((threadIdx.x / 32) * 32) << 16;
#pragma unroll
    for (int c4 = 0; c4 < D / 32; ++c4) {
        uint32_t o[32];
        tmem_ld32(lane_base + tmem_o + c4 * 32, o);
        tmem_ld_wait();
        store_result<D, G>(it, P, r, o, c4 * 32, 32, m, l, out, ws, h_q);
    }
}

}  // namespace kvlink
