// RoPE rotation by a position delta (Sec. 2.2) on bf16 key chunks, shared by the
// re-encode kernels and the fused linked-prefill kernel so that the paths that build a
// linked value cache write the same bits for every re-encoded key (the keys-only
// re-encode takes a faster form, within the same one-ulp bound; see rotate8).
//
// Precision: a rotated component x cos a - y sin a can cancel to far below |x|,
// where the bf16 quantum is tiny; an fp32 cos/sin (relative error 2^-24) would
// then be off by many bf16 ulps.  The delta table therefore holds cos and sin as
// unevaluated float pairs hi + lo (about 48 significant bits, split from the
// fp64 values) and the products are formed with their exact FMA rounding
// errors (the error-free TwoProduct transformation of Dekker, in its FMA form as
// used by Ogita, Rump and Oishi for compensated dot products), so the fp32 result
// carries an absolute error near 2^-47 |x| and rounds to within one bf16 ulp of
// the correctly rounded fp64 rotation.  That form is only needed where the result
// cancels: rotate8 first takes a plain FMA form with an error bound and falls back
// to the compensated one where the bound does not give one ulp.
#pragma once

#include <cuda_bf16.h>
#include <stdint.h>

namespace kvlink {

__device__ __forceinline__ float bf16lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);  // round to nearest even
    return *reinterpret_cast<const uint32_t*>(&h);
}

// x c - y s and y c + x s with c = ch + cl, s = sh + sl (double-float), x, y exact.
// The leading products are rounded explicitly (no contraction) and their exact
// rounding errors recovered with FMA; the small terms are added once at the end.
__device__ __forceinline__ float rot_first(float x, float y, float ch, float cl, float sh, float sl) {
    const float p1 = __fmul_rn(x, ch), p2 = __fmul_rn(y, sh);
    const float e1 = fmaf(x, ch, -p1), e2 = fmaf(y, sh, -p2);
    const float t = __fsub_rn(p1, p2);
    const float corr = (e1 - e2) + fmaf(x, cl, -(y * sl));
    return __fadd_rn(t, corr);
}

__device__ __forceinline__ float rot_second(float x, float y, float ch, float cl, float sh, float sl) {
    const float p1 = __fmul_rn(y, ch), p2 = __fmul_rn(x, sh);
    const float e1 = fmaf(y, ch, -p1), e2 = fmaf(x, sh, -p2);
    const float t = __fadd_rn(p1, p2);
    const float corr = (e1 + e2) + fmaf(y, cl, x * sl);
    return __fadd_rn(t, corr);
}

// lo' = lo cos - hi sin ; hi' = hi cos + lo sin, for the 8 pairs (j, j + D/2) of one
// (lo, hi) chunk pair; cs[e] = (cos hi, cos lo, sin hi, sin lo) of pair j0 + e.
//
// Fast path: r = RN(x ch - RN(y sh)) (one product rounded, the other inside an FMA, the low
// parts of cos and sin left out).  With M = max(|x|, |y|) and |cos|, |sin| <= 1, its error
// against x cos - y sin is at most 2^-25 |x| + 2^-25 |y| (the dropped low parts) + 2^-24 |y|
// (the rounded product) + 2^-24 |r| (the FMA's rounding) <= 2^-23 M + 2^-24 |r|, and the same for
// the second output.  A bf16 ulp of r is at least 2^-8 |r|, so wherever |r| >= 2^-13 M the error
// is under a quarter of an ulp and r rounds to bf16 within one ulp of the correctly rounded
// fp64 rotation.  A lane with an output below that bound (cancellation), or with M under
// 2^-100 (where fp32 subnormals would void the relative bounds), takes the compensated products
// above for its whole chunk pair.  On random keys that is about one rotation in 250 per lane.
// FAST false: the compensated products for every pair.  Both forms are within one ulp; they can
// round the same key one ulp apart.  The keys-only re-encode takes the fast form (31.0 against
// 34.5 us per layer of the Llama-8B batch-8 workload); the launch that also copies the values
// is bound by its cache writes (48 us either way) and, with the fast form, made the overlapped
// 32-layer step slower (449 against 433 us/query), so it and the other kernels keep the
// compensated form.
template <bool FAST>
__device__ __forceinline__ void rotate8(uint4& lo, uint4& hi, const float4 (&cs)[8]) {
    uint32_t* a = reinterpret_cast<uint32_t*>(&lo);
    uint32_t* b = reinterpret_cast<uint32_t*>(&hi);
    float r[8], t[8];
    bool hard = !FAST;
#pragma unroll
    for (int e = 0; e < 8 && FAST; ++e) {
        const uint32_t wa = a[e / 2], wb = b[e / 2];
        const float x = (e & 1) ? bf16hi(wa) : bf16lo(wa);
        const float y = (e & 1) ? bf16hi(wb) : bf16lo(wb);
        const float4 c = cs[e];
        r[e] = fmaf(x, c.x, -__fmul_rn(y, c.z));
        t[e] = fmaf(y, c.x, __fmul_rn(x, c.z));
        const float m = fmaxf(fabsf(x), fabsf(y));
        const float lim = 0x1p-13f * m;
        hard |= (fabsf(r[e]) < lim) | (fabsf(t[e]) < lim) | (m < 0x1p-100f);
    }
    if (hard) {
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const uint32_t wa = a[e / 2], wb = b[e / 2];
            const float x = (e & 1) ? bf16hi(wa) : bf16lo(wa);
            const float y = (e & 1) ? bf16hi(wb) : bf16lo(wb);
            const float4 c = cs[e];
            r[e] = rot_first(x, y, c.x, c.y, c.z, c.w);
            t[e] = rot_second(x, y, c.x, c.y, c.z, c.w);
        }
    }
#pragma unroll
    for (int w = 0; w < 4; ++w) {
        a[w] = pack_bf16(r[2 * w], r[2 * w + 1]);
        b[w] = pack_bf16(t[2 * w], t[2 * w + 1]);
    }
}

}  // namespace kvlink
