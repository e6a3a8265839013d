// Suffix attention on the CUDA cores (Sec. 2.3, "inference"): one CTA per
// (fresh row, KV head) computes the G query heads that share the KV head, over
// the row's visible positions 0..pos (cache rows from the plan's source table, so
// any physical layout of the cache works).  Each of the four warps streams every fourth
// key with an online softmax; the warps' partial results are merged at the end.
// This is the plain, unblocked form of the computation: it reads every visible
// key once per fresh row and uses no tensor cores.  It serves head dims and
// group sizes the tensor-core kernel does not take, and as an independent GPU
// cross-check of it.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "kvlink_internal.h"

namespace kvlink {

template <int D, int G>
__global__ void __launch_bounds__(128) attn_simt_kernel(DevicePlan P, const __nv_bfloat16* __restrict__ q,
                                                        const __nv_bfloat16* __restrict__ cache_k,
                                                        const __nv_bfloat16* __restrict__ cache_v,
                                                        __nv_bfloat16* __restrict__ out, int h_q, int h_kv,
                                                        float scale_log2) {
    constexpr int DPL = D / 32;  // dims per lane
    constexpr int NW = 4;
    __shared__ float sm_m[NW][G], sm_l[NW][G];
    __shared__ float sm_acc[NW][G][D];

    const int r = blockIdx.x, g = blockIdx.y;
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int b = P.fresh_query[r];
    const int pos = P.fresh_pos[r];
    const int64_t base = P.cu_ctx[b];

    float qv[G][DPL], acc[G][DPL], m[G], l[G];
#pragma unroll
    for (int h = 0; h < G; ++h) {
        const __nv_bfloat16* qr = q + ((int64_t)r * h_q + g * G + h) * D + lane * DPL;
#pragma unroll
        for (int e = 0; e < DPL; ++e) {
            qv[h][e] = __bfloat162float(qr[e]) * scale_log2;
            acc[h][e] = 0.f;
        }
        m[h] = -INFINITY;
        l[h] = 0.f;
    }
    for (int j = warp; j <= pos; j += NW) {
        const int64_t off = ((int64_t)P.src[base + j].slot * h_kv + g) * D + lane * DPL;  // position j's row
        float kk[DPL], vv[DPL];
#pragma unroll
        for (int e = 0; e < DPL; ++e) {
            kk[e] = __bfloat162float(cache_k[off + e]);
            vv[e] = __bfloat162float(cache_v[off + e]);
        }
#pragma unroll
        for (int h = 0; h < G; ++h) {
            float s = 0.f;
#pragma unroll
            for (int e = 0; e < DPL; ++e) s = fmaf(qv[h][e], kk[e], s);
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
            const float mn = fmaxf(m[h], s);
            const float corr = exp2f(m[h] - mn);
            const float p = exp2f(s - mn);
            l[h] = l[h] * corr + p;
#pragma unroll
            for (int e = 0; e < DPL; ++e) acc[h][e] = fmaf(acc[h][e], corr, p * vv[e]);
            m[h] = mn;
        }
    }
#pragma unroll
    for (int h = 0; h < G; ++h) {
#pragma unroll
        for (int e = 0; e < DPL; ++e) sm_acc[warp][h][lane * DPL + e] = acc[h][e];
        if (lane == 0) {
            sm_m[warp][h] = m[h];
            sm_l[warp][h] = l[h];
        }
    }
    __syncthreads();
    for (int t = threadIdx.x; t < G * D; t += blockDim.x) {
        const int h = t / D, d = t % D;
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < NW; ++w) M = fmaxf(M, sm_m[w][h]);
        float L = 0.f, O = 0.f;
#pragma unroll
        for (int w = 0; w < NW; ++w) {
            const float f = sm_m[w][h] == -INFINITY ? 0.f : exp2f(sm_m[w][h] - M);
            L += sm_l[w][h] * f;
            O += sm_acc[w][h][d] * f;
        }
        out[((int64_t)r * h_q + g * G + h) * D + d] = __float2bfloat16_rn(O / L);
    }
}

template <int D>
static void launch_simt_d(const DevicePlan& P, int n_fresh, int G, const void* q, const void* ck,
                          const void* cv, void* out, int h_q, int h_kv, float sl2, cudaStream_t st) {
    using bf = __nv_bfloat16;
    const dim3 grid(n_fresh, h_kv);
    switch (G) {
#define KVLINK_SIMT_CASE(GG)                                                                   \
    case GG:                                                                                  \
        attn_simt_kernel<D, GG><<<grid, 128, 0, st>>>(P, (const bf*)q, (const bf*)ck,         \
                                                     (const bf*)cv, (bf*)out, h_q, h_kv, sl2); \
        break;
        KVLINK_SIMT_CASE(1)
        KVLINK_SIMT_CASE(2)
        KVLINK_SIMT_CASE(4)
        KVLINK_SIMT_CASE(8)
        KVLINK_SIMT_CASE(16)
#undef KVLINK_SIMT_CASE
        default:
            break;
    }
}

void launch_attention_simt(const DevicePlan& P, int n_fresh, int head_dim, int h_q, int h_kv,
                           const void* q, const void* cache_k, const void* cache_v, void* out,
                           cudaStream_t stream) {
    const float scale_log2 = 1.4426950408889634f / sqrtf((float)head_dim);
    const int G = h_q / h_kv;
    if (head_dim == 128)
        launch_simt_d<128>(P, n_fresh, G, q, cache_k, cache_v, out, h_q, h_kv, scale_log2, stream);
    else
        launch_simt_d<64>(P, n_fresh, G, q, cache_k, cache_v, out, h_q, h_kv, scale_log2, stream);
}

}  // namespace kvlink
