// RoPE rotation by a position delta (Sec. 2.2) on bf16 key chunks, shared by the
// re-encode kernel and the fused linked-prefill kernel so that both write the same
// bits for every re-encoded key.
//
// Precision: a rotated component x cos a - y sin a can cancel to far below |x|,
// where the bf16 quantum is tiny; an fp32 cos/sin (relative error 2^-24) would
// then be off by many bf16 ulps.  The delta table therefore holds cos and sin as
// unevaluated float pairs hi + lo (about 48 significant bits, split from the
// fp64 values) and the products are formed with their exact FMA rounding
// errors (the error-free TwoProduct transformation of Dekker, in its FMA form as
// used by Ogita, Rump and Oishi for compensated dot products), so the fp32 result
// carries an absolute error near 2^-47 |x| and rounds to within one bf16 ulp of
// the correctly rounded fp64 rotation.
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
// (The same operations two pairs at a time in f32x2 instructions measured slower: the
// re-encode went from 34.7 to 38.6 us per layer of the Llama-8B batch-8 workload.)
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
__device__ __forceinline__ void rotate8(uint4& lo, uint4& hi, const float4 (&cs)[8]) {
    uint32_t* a = reinterpret_cast<uint32_t*>(&lo);
    uint32_t* b = reinterpret_cast<uint32_t*>(&hi);
#pragma unroll
    for (int w = 0; w < 4; ++w) {
        const float x0 = bf16lo(a[w]), x1 = bf16hi(a[w]);
        const float y0 = bf16lo(b[w]), y1 = bf16hi(b[w]);
        const float4 c0 = cs[2 * w], c1 = cs[2 * w + 1];
        const float r0 = rot_first(x0, y0, c0.x, c0.y, c0.z, c0.w);
        const float r1 = rot_first(x1, y1, c1.x, c1.y, c1.z, c1.w);
        const float t0 = rot_second(x0, y0, c0.x, c0.y, c0.z, c0.w);
        const float t1 = rot_second(x1, y1, c1.x, c1.y, c1.z, c1.w);
        a[w] = pack_bf16(r0, r1);
        b[w] = pack_bf16(t0, t1);
    }
}

}  // namespace kvlink
