// Fused linked prefill on the tcgen05 tensor cores: the positional re-encoding of
// Sec. 2.2, the concatenation of the document caches (Sec. 2.1, Sec. 2.3 inference)
// and the attention of the fresh link and question rows (Sec. 2.3) in one kernel.
//
// The two-kernel path writes the whole linked cache and then reads it back for the
// attention.  Here the attention reads every key and value where it already is: pool
// rows for the prefix and the documents, k_new / v_new for the fresh rows.  Document
// keys are rotated by their delta in shared memory on their way to the tensor cores,
// and the items that own a key range also store the rows to the linked cache, so the
// cache is written once and never read back.  The rotation is the re-encode kernel's
// (kvlink_rope.cuh) and the attention arithmetic is the suffix-attention kernel's
// (kvlink_attention_common.cuh, same tiles, same MMA order), so the cache and the
// output equal the two-kernel path's bit for bit.
//
// Keys are visited in linked-cache row order, as in the suffix-attention kernel: key
// tile t of an item stands for cache rows [128 t, 128 t + 128) of its query, whose
// sources come from the plan's per-row source table, and the same per-row visibility
// mask applies, in either physical layout (interleaved, or links at the end).
//
// Warp roles (384 threads = 3 warpgroups, one CTA per SM, 512 TMEM columns):
//   warps 0-3  softmax + epilogue, thread r owns tile row r = TMEM lane r
//   warp 9     TMA: the rows of a key tile come in groups of 8 positions; a group whose
//              8 rows are consecutive in one tensor (the plan's group table) is one
//              8-row copy per 64-dim atom, landing 1024-byte aligned in the 128-byte
//              swizzled layout the MMA reads.  Runs up to NS tiles ahead.
//   warps 4-7  gather: thread (c, g) owns chunk pair (c, c + D/16) -- 16-byte chunks
//              holding dims 8c..8c+7 and the rotate-half partners D/2 + 8c.. -- of rows
//              g, g + RG, ... of every key tile, for K and for V.  Rows of the other
//              groups (a segment boundary inside, or past the query's end) it copies with
//              cp.async (or zero-fills); once the tile has landed it rotates the document
//              keys in place (the eight double-float cos/sin of its pairs stay in
//              registers while the segment does not change), stores owned rows to the
//              linked cache, and publishes.
//   warp 8     TMEM allocation, Q by TMA, the thread issuing S = Q K^T; warp 10: the
//              thread issuing O += P V; warp 11 idle (completes the third warpgroup)
// Registers: launched at 168 per thread (384 x 168 <= 64K); the third warpgroup drops
// to 56 and the softmax warpgroup rises to 232, so that on each SM sub-partition
// (one warp of each warpgroup, 512 registers per thread in all) 232 + 168 + 56 fit.
// A stage holds one K tile and one V tile: raw_full[s] completes when its TMA copies
// have landed, kv_full[s] when the four gather warps have published it, kv_empty[s]
// when the PV MMA of its tile has finished.
// The gather runs one tile ahead: copies of tile j + 1 are in flight while tile j is
// rotated.  Every wait is bounded in time as in the suffix-attention kernel; on
// expiry the CTA drains its own copies and MMAs, frees TMEM and returns.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "kvlink_attention_common.cuh"
#include "kvlink_internal.h"
#include "kvlink_rope.cuh"
#include "kvlink_sm100.cuh"

namespace kvlink {
using namespace sm100;

bool make_map_3d(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1, uint64_t d2, uint32_t b0,
                 uint32_t b1, uint32_t b2);
cudaError_t launch_attn_merge(const DevicePlan& P, int n_merges, const float* ws, void* out, int h_q, int G,
                              int head_dim, cudaStream_t stream);

static __device__ int32_t g_fused_status;

constexpr int kFusedThreads = 384;
constexpr uint32_t kLaunchRegs = 168, kSoftmaxRegs = 232, kIdleRegs = 56;
static_assert(kFusedThreads * kLaunchRegs <= 65536, "launch register budget");
static_assert(128 * (kSoftmaxRegs - kLaunchRegs) <= 128 * (kLaunchRegs - kIdleRegs), "register re-split");
static_assert(kSoftmaxRegs + kLaunchRegs + kIdleRegs <= 512, "sub-partition register budget");
constexpr int kGatherWarp0 = 4;  // warps 4-7
constexpr int kGatherThreads = 128;
constexpr int kFusedMmaWarp = 8;   // S = Q K^T issuer (and TMEM, Q)
constexpr int kFusedTmaWarp = 9;
constexpr int kFusedPvWarp = 10;   // O += P V issuer
constexpr uint32_t kFusedTmemCols = 512;

template <int D>
struct FusedCfg {
    static constexpr int ATOMS = D / 64;                   // 128-byte swizzle atoms along head_dim
    static constexpr int NS = (D == 128) ? 3 : 6;          // K+V stages
    static constexpr int NB = 3;                           // S/P buffers in TMEM
    static constexpr uint32_t ATOM_BYTES = 128 * 128;      // [128 rows][64 bf16]
    static constexpr uint32_t Q_BYTES = ATOMS * ATOM_BYTES;
    static constexpr uint32_t HALF_BYTES = ATOMS * ATOM_BYTES;  // one K (or V) tile
    static constexpr uint32_t STAGE_BYTES = 2 * HALF_BYTES;
    static constexpr uint32_t OFF_Q = 0;
    static constexpr uint32_t OFF_KV = Q_BYTES;
    static constexpr uint32_t OFF_BAR = OFF_KV + NS * STAGE_BYTES;
    // q_full, raw_full[NS], kv_full[NS], kv_empty[NS], s_full[NB], p_full[NB], o_done[NB], drain x2
    static constexpr int N_BARS = 3 + 3 * NS + 3 * NB;
    static constexpr uint32_t GROUP_TX = 8 * 128 * ATOMS * 2;  // K and V bytes of one 8-row group
    static constexpr uint32_t SMEM_BYTES = OFF_BAR + N_BARS * 8 + 16 + 1024;
    static constexpr uint32_t TMEM_S = 0;                  // buffer b at b * 128
    static constexpr uint32_t TMEM_O = NB * kAttnBN;
    static constexpr int CP = D / 16;                      // chunk pairs per row
    static constexpr int RG = kGatherThreads / CP;         // row groups
    static constexpr int RPT = kAttnBN / RG;               // rows per gather thread per tile
    static_assert(TMEM_O + D <= kFusedTmemCols, "TMEM budget");
    static_assert(SMEM_BYTES <= 232448, "shared memory budget");
    static_assert(RG * RPT == kAttnBN, "gather split");
};

// Source tensors of the 8-row TMA copies: A = pool, F = fresh rows; [rows][h_kv][D]
// bf16, box {64, 1, 8}.
struct FusedMaps {
    CUtensorMap q, ak, av, fk, fv;
};

struct FusedArgs {
    const __nv_bfloat16* pool_k;
    const __nv_bfloat16* pool_v;
    const __nv_bfloat16* k_new;
    const __nv_bfloat16* v_new;
    __nv_bfloat16* cache_k;  // side output of owner items (NULL: not written)
    __nv_bfloat16* cache_v;
    __nv_bfloat16* out;
    float* ws;
    int h_q, h_kv;
    float scale_log2;
};

// Byte offset of 16-byte chunk `ch` (dims 8ch..8ch+7) of tile row r in a 128-byte
// swizzled [atom][128 rows][64 dims] tile: the chunk index is XORed with r mod 8.
__device__ __forceinline__ uint32_t swz(int ch, int r) {
    return (uint32_t)(ch >> 3) * (128u * 128u) + (uint32_t)r * 128u + ((uint32_t)((ch & 7) ^ (r & 7)) << 4);
}

__device__ __forceinline__ kvlink_source_t load_source(const kvlink_source_t* src, int64_t i) {
    const int4 v = __ldg(reinterpret_cast<const int4*>(src) + i);
    return kvlink_source_t{v.x, v.y, v.z, v.w};
}

// TMA role (one thread): the 8-row group copies of every key tile of the item.
template <int D>
__device__ __forceinline__ void tma_role(const AttnItem& it, const DevicePlan& P, const FusedMaps& M,
                                         uint8_t* smem, uint64_t* raw_full, uint64_t* kv_empty, int n_tiles,
                                         volatile int32_t* abort_flag) {
    using C = FusedCfg<D>;
    const int32_t* grp = P.grp_src;
    const int gbase = P.cu_grp[it.query];
    const int n_grp = P.cu_grp[it.query + 1] - gbase;
    int issued = 0;
    for (int j = 0; j < n_tiles; ++j) {
        const int st = j % C::NS;
        if (!wait_bar(kv_empty + st, ((j / C::NS) & 1) ^ 1, abort_flag, &g_fused_status)) break;
        const int m0 = item_tile(it, it.kv_tile0 + j) * (kAttnBN / 8);
        int32_t gw[kAttnBN / 8];
        uint32_t n = 0;
#pragma unroll
        for (int m = 0; m < kAttnBN / 8; ++m) {
            gw[m] = m0 + m < n_grp ? __ldg(grp + gbase + m0 + m) : -1;
            n += gw[m] >= 0 ? 1u : 0u;
        }
        mbar_arrive_expect_tx(raw_full + st, n * C::GROUP_TX);
        uint8_t* sk = smem + C::OFF_KV + st * C::STAGE_BYTES;
#pragma unroll
        for (int m = 0; m < kAttnBN / 8; ++m) {
            if (gw[m] < 0) continue;
            const bool fresh = (gw[m] & kGrpFresh) != 0;
            const int row = gw[m] & kGrpRowMask;
#pragma unroll
            for (int a = 0; a < C::ATOMS; ++a) {
                const uint32_t off = a * C::ATOM_BYTES + m * 8 * 128;
                tma_load_3d(sk + off, fresh ? &M.fk : &M.ak, a * 64, it.kv_head, row, raw_full + st);
                tma_load_3d(sk + C::HALF_BYTES + off, fresh ? &M.fv : &M.av, a * 64, it.kv_head, row, raw_full + st);
            }
        }
        issued = j + 1;
    }
    // no copy may still be in flight when the CTA leaves
    for (int j = issued - C::NS > 0 ? issued - C::NS : 0; j < issued; ++j)
        drain_bar(raw_full + j % C::NS, (j / C::NS) & 1, &g_fused_status);
}

template <int D>
__device__ __forceinline__ void gather_role(const AttnItem& it, const DevicePlan& P, const FusedArgs& A,
                                            uint8_t* smem, uint64_t* raw_full, uint64_t* kv_full,
                                            uint64_t* kv_empty, int n_tiles, volatile int32_t* abort_flag) {
    using C = FusedCfg<D>;
    const int t = threadIdx.x - kGatherWarp0 * 32;
    const int lane = threadIdx.x % 32;
    const int c = t % C::CP, g = t / C::CP;
    const int64_t ctx0 = P.cu_ctx[it.query];
    const int n_pos = (int)(P.cu_ctx[it.query + 1] - ctx0);
    const int64_t row_elems = (int64_t)A.h_kv * D;
    const int64_t col0 = (int64_t)it.kv_head * D + 8 * c;  // lo chunk of this thread within a row
    const bool own_k = it.owner && A.cache_k != nullptr;
    const bool own_v = it.owner && A.cache_v != nullptr;
    const uint32_t kv_base = smem_u32(smem + C::OFF_KV);
    const int32_t* grp = P.grp_src;
    const int gbase = P.cu_grp[it.query];

    // rows of key tile j outside the TMA groups: copied row by row, or zero-filled past
    // the query's end
    auto issue = [&](int j) -> bool {
        const int st = j % C::NS;
        if (!warp_wait(kv_empty + st, ((j / C::NS) & 1) ^ 1, abort_flag, &g_fused_status)) return false;
        const uint32_t sk = kv_base + st * C::STAGE_BYTES, sv = sk + C::HALF_BYTES;
        uint8_t* gk = smem + C::OFF_KV + st * C::STAGE_BYTES;
        const int key0 = item_tile(it, it.kv_tile0 + j) * kAttnBN;
        // all of the tile's records first: one load latency, not one per row (the copies
        // below are compiler barriers for memory accesses)
        bool by_row[C::RPT];
#pragma unroll
        for (int k = 0; k < C::RPT; ++k) {
            const int pos = key0 + g + C::RG * k;
            by_row[k] = pos < n_pos && __ldg(grp + gbase + pos / 8) < 0;
        }
        kvlink_source_t es[C::RPT];
#pragma unroll
        for (int k = 0; k < C::RPT; ++k) {
            const int pos = key0 + g + C::RG * k;
            es[k] = by_row[k] ? load_source(P.src_row, ctx0 + pos) : kvlink_source_t{0, 0, 0, -1};
        }
#pragma unroll
        for (int k = 0; k < C::RPT; ++k) {
            const int r = g + C::RG * k, pos = key0 + r;
            const uint32_t o_lo = swz(c, r), o_hi = swz(c + C::CP, r);
            if (by_row[k]) {
                const kvlink_source_t& e = es[k];
                const __nv_bfloat16 *kb, *vb;
                int64_t row;
                if (e.kind == KVLINK_SRC_FRESH) {
                    kb = A.k_new, vb = A.v_new, row = e.row;
                } else {
                    kb = A.pool_k, vb = A.pool_v, row = e.row;
                }
                const int64_t off = row * row_elems + col0;
                cp_async16(sk + o_lo, kb + off);
                cp_async16(sk + o_hi, kb + off + D / 2);
                cp_async16(sv + o_lo, vb + off);
                cp_async16(sv + o_hi, vb + off + D / 2);
            } else if (pos >= n_pos) {
                const uint4 z = make_uint4(0u, 0u, 0u, 0u);
                *reinterpret_cast<uint4*>(gk + o_lo) = z;
                *reinterpret_cast<uint4*>(gk + o_hi) = z;
                *reinterpret_cast<uint4*>(gk + C::HALF_BYTES + o_lo) = z;
                *reinterpret_cast<uint4*>(gk + C::HALF_BYTES + o_hi) = z;
            }
        }
        cp_async_commit();
        return true;
    };

    int cur_table = -1;
    float4 cs[8];
    // tile j has landed (the TMA groups and this thread's copies): rotate, store owned
    // rows, publish
    auto finish = [&](int j) -> bool {
        const int st = j % C::NS;
        if (!warp_wait(raw_full + st, (j / C::NS) & 1, abort_flag, &g_fused_status)) return false;
        uint8_t* sk = smem + C::OFF_KV + st * C::STAGE_BYTES;
        uint8_t* sv = sk + C::HALF_BYTES;
        const int key0 = item_tile(it, it.kv_tile0 + j) * kAttnBN;
        kvlink_source_t es[C::RPT];
#pragma unroll
        for (int k = 0; k < C::RPT; ++k) {
            const int pos = key0 + g + C::RG * k;
            es[k] = pos < n_pos ? load_source(P.src_row, ctx0 + pos) : kvlink_source_t{0, 0, 0, -1};
        }
#pragma unroll
        for (int k = 0; k < C::RPT; ++k) {
            const int r = g + C::RG * k, pos = key0 + r;
            if (pos >= n_pos) continue;
            const kvlink_source_t& e = es[k];
            const bool rot = e.table >= 0;
            const uint32_t o_lo = swz(c, r), o_hi = swz(c + C::CP, r);
            if (rot || own_k) {
                uint4 a = *reinterpret_cast<const uint4*>(sk + o_lo);
                uint4 b = *reinterpret_cast<const uint4*>(sk + o_hi);
                if (rot) {
                    if (e.table != cur_table) {
                        const float4* tb = P.rope + (int64_t)e.table * (D / 2) + 8 * c;
#pragma unroll
                        for (int q = 0; q < 8; ++q) cs[q] = __ldg(tb + q);
                        cur_table = e.table;
                    }
                    rotate8<false>(a, b, cs);
                    *reinterpret_cast<uint4*>(sk + o_lo) = a;
                    *reinterpret_cast<uint4*>(sk + o_hi) = b;
                }
                if (own_k) {
                    __nv_bfloat16* dst = A.cache_k + (int64_t)e.slot * row_elems + col0;
                    *reinterpret_cast<uint4*>(dst) = a;
                    *reinterpret_cast<uint4*>(dst + D / 2) = b;
                }
            }
            if (own_v) {
                __nv_bfloat16* dst = A.cache_v + (int64_t)e.slot * row_elems + col0;
                *reinterpret_cast<uint4*>(dst) = *reinterpret_cast<const uint4*>(sv + o_lo);
                *reinterpret_cast<uint4*>(dst + D / 2) = *reinterpret_cast<const uint4*>(sv + o_hi);
            }
        }
        fence_proxy_async_smem();  // the MMA reads the stage through the async proxy
        __syncwarp();
        if (lane == 0) mbar_arrive(kv_full + st);
        return true;
    };

    bool ok = n_tiles > 0 && issue(0);
    for (int j = 0; ok && j < n_tiles; ++j) {
        if (j + 1 < n_tiles) {
            if (!(ok = issue(j + 1))) break;
            cp_async_wait<1>();
        } else {
            cp_async_wait<0>();
        }
        ok = finish(j);
    }
    cp_async_wait<0>();  // no copy may still be in flight when the CTA leaves
}

template <int D, int G>
__global__ void __launch_bounds__(kFusedThreads, 1)
    attn_fused_kernel(const __grid_constant__ FusedMaps M, const DevicePlan P, const FusedArgs A) {
    using C = FusedCfg<D>;
    constexpr int NS = C::NS, NB = C::NB;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw_addr = smem_u32(smem_raw);
    uint8_t* smem = smem_raw + ((1024u - (raw_addr & 1023u)) & 1023u);

    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);
    uint64_t* bar_q_full = bars;
    uint64_t* bar_raw_full = bar_q_full + 1;
    uint64_t* bar_kv_full = bar_raw_full + NS;
    uint64_t* bar_kv_empty = bar_kv_full + NS;
    uint64_t* bar_s_full = bar_kv_empty + NS;
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
            uint32_t count = 1;
            if (bars + i >= bar_kv_full && bars + i < bar_kv_full + NS) count = kGatherThreads / 32;
            if (bars + i >= bar_p_full && bars + i < bar_p_full + NB) count = 4;
            mbar_init(bars + i, count);
        }
        // after a recorded failure, later launches skip their work instead of waiting out their bounds
        *abort_flag = *reinterpret_cast<volatile int32_t*>(&g_fused_status) != 0 ? 1 : 0;
        fence_mbar_init();
    }
    if (warp == kFusedMmaWarp) {
        tmem_alloc(tmem_holder, kFusedTmemCols);
        tmem_relinquish();
        if (lane == 0) {
            prefetch_tensormap(&M.q);
            prefetch_tensormap(&M.ak);
            prefetch_tensormap(&M.av);
            prefetch_tensormap(&M.fk);
            prefetch_tensormap(&M.fv);
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_holder;
    const bool skip = *abort_flag != 0;  // written before the barrier: uniform across the CTA

    if (skip) {
        // nothing issued: fall through to the teardown
    } else if (warp >= kGatherWarp0 && warp < kGatherWarp0 + kGatherThreads / 32) {
        gather_role<D>(it, P, A, smem, bar_raw_full, bar_kv_full, bar_kv_empty, n_tiles, abort_flag);
    } else if (warp >= kFusedMmaWarp) {
        setmaxnreg_dec<kIdleRegs>();
        if (warp == kFusedMmaWarp && lane == 0) {
            constexpr uint32_t idesc_qk = idesc_bf16_f32(128, kAttnBN, 0, 0);
            const uint32_t sQ = smem_u32(smem + C::OFF_Q);
            const int q_row0 = P.cu_fresh[it.query] + it.tok0;
            mbar_arrive_expect_tx(bar_q_full, C::Q_BYTES);
#pragma unroll
            for (int a = 0; a < C::ATOMS; ++a)
                tma_load_3d(smem + C::OFF_Q + a * C::ATOM_BYTES, &M.q, a * 64, it.kv_head * G, q_row0, bar_q_full);
            bool ok = wait_bar(bar_q_full, 0, abort_flag, &g_fused_status);
            if (!ok) drain_bar(bar_q_full, 0, &g_fused_status);  // the Q copy lands before the CTA leaves
            for (int j = 0; ok && j < n_tiles; ++j) {
                const int st = j % NS, b = j % NB;
                if (!(ok = wait_bar(bar_kv_full + st, (j / NS) & 1, abort_flag, &g_fused_status))) break;
                // buffer b last held P_{j-NB}: its PV must have finished reading it
                if (j >= NB && !(ok = wait_bar(bar_o_done + b, ((j - NB) / NB) & 1, abort_flag, &g_fused_status)))
                    break;
                tc_fence_after();
                const uint32_t sK = smem_u32(smem + C::OFF_KV + st * C::STAGE_BYTES);
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk) {
                    const uint32_t koff = (kk >> 2) * C::ATOM_BYTES + (kk & 3) * 32;
                    mma_bf16_ss(tmem + C::TMEM_S + b * kAttnBN, sdesc_sw128(sQ + koff, 16, 1024),
                                sdesc_sw128(sK + koff, 16, 1024), idesc_qk, kk > 0 ? 1u : 0u);
                }
                mma_commit(bar_s_full + b);
            }
            mma_commit(bar_drain);  // arrives once every MMA issued above has completed
            drain_bar(bar_drain, 0, &g_fused_status);
        } else if (warp == kFusedPvWarp && lane == 0) {
            constexpr uint32_t idesc_pv = idesc_bf16_f32(128, D, 0, 1);
            // O += P_i V_i, P_i (bf16) read from its S buffer in TMEM; frees stage i % NS
            for (int i = 0; i < n_tiles; ++i) {
                const int b = i % NB, st = i % NS;
                if (!wait_bar(bar_p_full + b, (i / NB) & 1, abort_flag, &g_fused_status)) break;
                if (!wait_bar(bar_kv_full + st, (i / NS) & 1, abort_flag, &g_fused_status)) break;
                tc_fence_after();
                const uint32_t sV = smem_u32(smem + C::OFF_KV + st * C::STAGE_BYTES + C::HALF_BYTES);
                const uint32_t pcol = tmem + C::TMEM_S + b * kAttnBN;
#pragma unroll
                for (int kk = 0; kk < kAttnBN / 16; ++kk)
                    mma_bf16_ts(tmem + C::TMEM_O, pcol + kk * 8, sdesc_sw128(sV + kk * 16 * 128, C::ATOM_BYTES, 1024),
                                idesc_pv, (i > 0 || kk > 0) ? 1u : 0u);
                mma_commit(bar_o_done + b);
                mma_commit(bar_kv_empty + st);
            }
            mma_commit(bar_drain + 1);
            drain_bar(bar_drain + 1, 0, &g_fused_status);
        } else if (warp == kFusedTmaWarp && lane == 0) {
            tma_role<D>(it, P, M, smem, bar_raw_full, bar_kv_empty, n_tiles, abort_flag);
        }
    } else {
        setmaxnreg_inc<kSoftmaxRegs>();
        softmax_role<D, G, NB>(it, P, tmem + C::TMEM_S, tmem + C::TMEM_O, n_tiles, bar_s_full, bar_p_full,
                               bar_o_done, abort_flag, &g_fused_status, A.out, A.ws, A.h_q, A.scale_log2);
    }

    tc_fence_before();
    __syncthreads();
    if (warp == kFusedMmaWarp) {
        tc_fence_after();
        tmem_dealloc(tmem, kFusedTmemCols);
    }
}

template <int D, int G>
static cudaError_t launch_fused_dg(const FusedMaps& M, const DevicePlan& P, const FusedArgs& A, int n_items,
                                   cudaStream_t stream) {
    using C = FusedCfg<D>;
    static std::atomic<uint64_t> attr_set{0};
    cudaError_t ea = once_per_device(attr_set, [] {
        return cudaFuncSetAttribute(attn_fused_kernel<D, G>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)C::SMEM_BYTES);
    });
    if (ea != cudaSuccess) return ea;
    if (n_items > 0) attn_fused_kernel<D, G><<<n_items, kFusedThreads, C::SMEM_BYTES, stream>>>(M, P, A);
    return cudaGetLastError();
}

// Fused linked prefill: sources are the pool and the fresh rows; owner items write
// cache_k / cache_v where non-NULL.  Returns 0, KVLINK_ECUDA or KVLINK_EUNSUPPORTED.
int launch_attention_fused(const DevicePlan& P, int n_items, int n_merges, int n_fresh, int64_t pool_rows,
                           int head_dim, int h_q, int h_kv, const void* q, const void* pool_k, const void* pool_v,
                           const void* k_new, const void* v_new, void* cache_k, void* cache_v, void* out, void* ws,
                           cudaStream_t stream, cudaError_t* err) {
    const int G = h_q / h_kv;
    FusedMaps M;
    const uint64_t D = (uint64_t)head_dim, H = (uint64_t)h_kv;
    if (!make_map_3d(&M.q, q, D, (uint64_t)h_q, (uint64_t)n_fresh, 64, (uint32_t)G, (uint32_t)(kAttnBM / G)) ||
        !make_map_3d(&M.ak, pool_k, D, H, (uint64_t)pool_rows, 64, 1, 8) ||
        !make_map_3d(&M.av, pool_v, D, H, (uint64_t)pool_rows, 64, 1, 8) ||
        !make_map_3d(&M.fk, k_new, D, H, (uint64_t)n_fresh, 64, 1, 8) ||
        !make_map_3d(&M.fv, v_new, D, H, (uint64_t)n_fresh, 64, 1, 8))
        return KVLINK_EUNSUPPORTED;
    using bf = __nv_bfloat16;
    FusedArgs A{(const bf*)pool_k, (const bf*)pool_v, (const bf*)k_new, (const bf*)v_new, (bf*)cache_k,
                (bf*)cache_v, (bf*)out, (float*)ws, h_q, h_kv, 1.4426950408889634f / sqrtf((float)head_dim)};
    cudaError_t e = cudaErrorInvalidValue;
#define KVLINK_FUSED_CASE(DD, GG) \
    if (head_dim == DD && G == GG) e = launch_fused_dg<DD, GG>(M, P, A, n_items, stream);
    KVLINK_FUSED_CASE(128, 1) KVLINK_FUSED_CASE(128, 2) KVLINK_FUSED_CASE(128, 4) KVLINK_FUSED_CASE(128, 8)
    KVLINK_FUSED_CASE(128, 16) KVLINK_FUSED_CASE(64, 1) KVLINK_FUSED_CASE(64, 2) KVLINK_FUSED_CASE(64, 4)
    KVLINK_FUSED_CASE(64, 8) KVLINK_FUSED_CASE(64, 16)
#undef KVLINK_FUSED_CASE
    if (e == cudaSuccess) e = launch_attn_merge(P, n_merges, (const float*)ws, out, h_q, G, head_dim, stream);
    if (e != cudaSuccess) {
        *err = e;
        return KVLINK_ECUDA;
    }
    return KVLINK_OK;
}

int read_fused_status(int32_t* status) {
    return cudaMemcpyFromSymbol(status, g_fused_status, sizeof(int32_t)) == cudaSuccess ? KVLINK_OK : KVLINK_ECUDA;
}

int clear_fused_status() {
    const int32_t z = 0;
    return cudaMemcpyToSymbol(g_fused_status, &z, sizeof(int32_t)) == cudaSuccess ? KVLINK_OK : KVLINK_ECUDA;
}

}  // namespace kvlink
