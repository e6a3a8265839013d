// Pieces shared by the two tensor-core attention kernels (the suffix attention over a
// materialised linked cache, and the fused linked prefill): bounded mbarrier waits,
// the softmax + epilogue role, and the FMA-pipe 2^x.
//
// The softmax role (Sec. 2.3 attention of the fresh rows; online softmax over KV
// tiles): 4 warps, thread r owns tile row r = TMEM lane r.  For every KV tile j it
// reads S_j from TMEM buffer j % NB, masks keys whose position is above the row's
// position, raises the running max (rescaling O in TMEM only when the max grew by
// more than 2^8), writes P_j = exp2(S_j c - m) as bf16 over the first half of the
// same buffer and signals the MMA thread.  Keys are visited in position order, so
// key index = position.  At the end it normalises O and stores the output rows, or
// stores the unnormalised partial (O, m, l) when the item's KV range was split.
#pragma once

#include <cuda_bf16.h>
#include <stdint.h>

#include "kvlink_internal.h"
#include "kvlink_sm100.cuh"

namespace kvlink {

constexpr uint64_t kWaitLimitNs = 2000000000ull;  // 2 s
constexpr int32_t kAttnStatusWaitTimeout = 0x41;
constexpr float kRescaleThreshold = 8.0f;         // log2 units: rescale O when the max grows by > 2^8
#ifndef KVLINK_EXP_POLY_FROM
#define KVLINK_EXP_POLY_FROM 8                     // column pairs c with (c % 8) >= this use exp2_poly2
#endif

// Wait for phase `parity` of `bar`; false if another role aborted or the time limit passed.
__device__ __forceinline__ bool wait_bar(uint64_t* bar, uint32_t parity, volatile int32_t* abort_flag,
                                         int32_t* status) {
    if (sm100::mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = sm100::globaltimer_ns();
    while (true) {
        if (sm100::mbar_try_wait(bar, parity)) return true;
        if (*abort_flag) return false;
        if (sm100::globaltimer_ns() - t0 > kWaitLimitNs) {
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

// Softmax + epilogue role, run by warps 0-3 (threadIdx.x = tile row).  TMEM holds NB
// S/P buffers of kAttnBN columns from column tmem_s and the O accumulator at tmem_o.
template <int D, int G, int NB>
__device__ __forceinline__ void softmax_role(const AttnItem& it, const DevicePlan& P, uint32_t tmem_s,
                                             uint32_t tmem_o, int n_tiles, uint64_t* bar_s_full,
                                             uint64_t* bar_p_full, uint64_t* bar_o_done,
                                             volatile int32_t* abort_flag, int32_t* status,
                                             __nv_bfloat16* __restrict__ out, float* __restrict__ ws, int h_q,
                                             float scale_log2) {
    using namespace sm100;
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
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
        if (!(ok = warp_wait(bar_s_full + b, (j / NB) & 1, abort_flag, status))) break;
        tc_fence_after();
        uint32_t s[128];
        const uint32_t s_col = lane_base + tmem_s + b * kAttnBN;
        tmem_ld32(s_col + 0, *reinterpret_cast<uint32_t(*)[32]>(s + 0));
        tmem_ld32(s_col + 32, *reinterpret_cast<uint32_t(*)[32]>(s + 32));
        tmem_ld32(s_col + 64, *reinterpret_cast<uint32_t(*)[32]>(s + 64));
        tmem_ld32(s_col + 96, *reinterpret_cast<uint32_t(*)[32]>(s + 96));
        tmem_ld_wait();

        // raw row max (scale > 0 commutes with max); masked keys become -inf.  Eight
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
            if (!(ok = warp_wait(bar_o_done + (j - 1) % NB, ((j - 1) / NB) & 1, abort_flag, status))) break;
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
    if (ok && n_tiles > 0)
        ok = warp_wait(bar_o_done + (n_tiles - 1) % NB, ((n_tiles - 1) / NB) & 1, abort_flag, status);
    if (!ok) return;
    tc_fence_after();
    if (it.slot < 0) {
        const float inv = 1.f / l;
        __nv_bfloat16* orow = out + ((int64_t)frow * h_q + it.kv_head * G + (r % G)) * D;
#pragma unroll
        for (int c4 = 0; c4 < D / 32; ++c4) {
            uint32_t o[32];
            tmem_ld32(lane_base + tmem_o + c4 * 32, o);
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
            tmem_ld32(lane_base + tmem_o + c4 * 32, o);
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

}  // namespace kvlink
