// RoPE delta table (Sec. 2.2, once per batch) and the re-encode + concat kernel
// (Sec. 2.2 positional re-encoding, Sec. 2.1 concatenation of the caches).
//
// The re-encode kernel is a streaming copy bound by HBM bandwidth.  One CTA takes
// one work unit: kCopyChunk tokens of one segment.  A thread owns a fixed
// (KV head, j0) slot across the unit's tokens: it moves the 16-byte key chunks
// holding dimensions j0..j0+7 and j0+D/2..j0+D/2+7 (the two halves of the RoPE
// pairs it rotates) and the value chunks at the same offsets, so every load and
// store is a coalesced 128-bit access and the eight (cos, sin) pairs of the
// segment's delta stay in registers for the whole unit.
//
// Precision: a rotated component x cos a - y sin a can cancel to far below |x|,
// where the bf16 quantum is tiny; an fp32 cos/sin (relative error 2^-24) would
// then be off by many bf16 ulps.  The table therefore holds cos and sin as
// unevaluated float pairs hi + lo (about 48 significant bits, split from the
// fp64 values) and the kernel forms the products with their exact FMA rounding
// errors, so the fp32 result carries an absolute error near 2^-47 |x| and rounds
// to within one bf16 ulp of the correctly rounded fp64 rotation.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "kvlink_internal.h"

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
// A3 + A4: re-encode/copy one work unit per CTA.
// --------------------------------------------------------------------------
__device__ __forceinline__ uint4 ld_stream(const uint4* p) {
    uint4 r;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
                 : "l"(p));
    return r;
}

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

// lo' = lo cos - hi sin ; hi' = hi cos + lo sin, for the 8 pairs of one (lo, hi) chunk pair
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

template <int D>
__global__ void __launch_bounds__(kCopyThreads) reencode_kernel(
    DevicePlan P, int chunk_base, int h_kv, int pool_bs,
    const __nv_bfloat16* __restrict__ pool_k, const __nv_bfloat16* __restrict__ pool_v,
    const __nv_bfloat16* __restrict__ k_new, const __nv_bfloat16* __restrict__ v_new,
    __nv_bfloat16* __restrict__ cache_k, __nv_bfloat16* __restrict__ cache_v) {
    constexpr int UPH = D / 16;  // (lo, hi) chunk pairs per head
    const int U = h_kv * UPH;    // pairs per token (divides kCopyThreads)
    const int TP = kCopyThreads / U;
    const CopyChunk ch = P.chunks[chunk_base + blockIdx.x];
    const kvlink_segment_t sg = P.seg[ch.seg];
    const int n = min(kCopyChunk, sg.len - ch.t0);
    const int unit = threadIdx.x % U;
    const int tok = threadIdx.x / U;
    const int head = unit / UPH;
    const int j0 = (unit % UPH) * 8;
    const int64_t row_elems = (int64_t)h_kv * D;
    const int64_t lo_off = (int64_t)head * D + j0;
    const int64_t hi_off = lo_off + D / 2;

    const bool fresh = sg.kind == KVLINK_SEG_LINK || sg.kind == KVLINK_SEG_QUESTION;
    const bool rotate = sg.kind == KVLINK_SEG_DOC;
    const __nv_bfloat16* sk = fresh ? k_new : pool_k;
    const __nv_bfloat16* sv = fresh ? v_new : pool_v;

    float4 cs[8];
    if (rotate) {
        const float4* t = P.rope + (int64_t)sg.table * (D / 2) + j0;
#pragma unroll
        for (int q = 0; q < 8; ++q) cs[q] = __ldg(t + q);
    } else {
#pragma unroll
        for (int q = 0; q < 8; ++q) cs[q] = make_float4(1.f, 0.f, 0.f, 0.f);
    }
    const int64_t entry_start = fresh ? 0 : P.pool_start[sg.src];

    auto src_row = [&](int tt) -> int64_t {
        if (fresh) return (int64_t)sg.src + tt;
        if (pool_bs == 0) return entry_start + tt;
        return (int64_t)P.pool_block_table[entry_start + tt / pool_bs] * pool_bs + tt % pool_bs;
    };

    // two tokens per iteration: all eight 16-byte loads are issued before any store
    for (int t = tok; t < n; t += 2 * TP) {
        const int ta = ch.t0 + t;
        const bool has_b = t + TP < n;
        const int tb = ta + TP;
        const int64_t ra = src_row(ta) * row_elems;
        const int64_t rb = has_b ? src_row(tb) * row_elems : ra;
        uint4 ka0 = ld_stream(reinterpret_cast<const uint4*>(sk + ra + lo_off));
        uint4 ka1 = ld_stream(reinterpret_cast<const uint4*>(sk + ra + hi_off));
        const uint4 va0 = ld_stream(reinterpret_cast<const uint4*>(sv + ra + lo_off));
        const uint4 va1 = ld_stream(reinterpret_cast<const uint4*>(sv + ra + hi_off));
        uint4 kb0, kb1, vb0, vb1;
        if (has_b) {
            kb0 = ld_stream(reinterpret_cast<const uint4*>(sk + rb + lo_off));
            kb1 = ld_stream(reinterpret_cast<const uint4*>(sk + rb + hi_off));
            vb0 = ld_stream(reinterpret_cast<const uint4*>(sv + rb + lo_off));
            vb1 = ld_stream(reinterpret_cast<const uint4*>(sv + rb + hi_off));
        }
        if (rotate) rotate8(ka0, ka1, cs);
        const int64_t da = (sg.dst + ta) * row_elems;
        *reinterpret_cast<uint4*>(cache_k + da + lo_off) = ka0;
        *reinterpret_cast<uint4*>(cache_k + da + hi_off) = ka1;
        *reinterpret_cast<uint4*>(cache_v + da + lo_off) = va0;
        *reinterpret_cast<uint4*>(cache_v + da + hi_off) = va1;
        if (has_b) {
            if (rotate) rotate8(kb0, kb1, cs);
            const int64_t db = (sg.dst + tb) * row_elems;
            *reinterpret_cast<uint4*>(cache_k + db + lo_off) = kb0;
            *reinterpret_cast<uint4*>(cache_k + db + hi_off) = kb1;
            *reinterpret_cast<uint4*>(cache_v + db + lo_off) = vb0;
            *reinterpret_cast<uint4*>(cache_v + db + hi_off) = vb1;
        }
    }
}

void launch_reencode(const DevicePlan& P, int chunk_base, int n_chunks, int head_dim, int h_kv,
                     int pool_bs, const void* pool_k, const void* pool_v, const void* k_new,
                     const void* v_new, void* cache_k, void* cache_v, cudaStream_t stream) {
    if (n_chunks <= 0) return;
    using bf = __nv_bfloat16;
    if (head_dim == 128)
        reencode_kernel<128><<<n_chunks, kCopyThreads, 0, stream>>>(
            P, chunk_base, h_kv, pool_bs, (const bf*)pool_k, (const bf*)pool_v, (const bf*)k_new,
            (const bf*)v_new, (bf*)cache_k, (bf*)cache_v);
    else
        reencode_kernel<64><<<n_chunks, kCopyThreads, 0, stream>>>(
            P, chunk_base, h_kv, pool_bs, (const bf*)pool_k, (const bf*)pool_v, (const bf*)k_new,
            (const bf*)v_new, (bf*)cache_k, (bf*)cache_v);
}

}  // namespace kvlink
