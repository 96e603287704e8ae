// Split-KV attention of the k appended rows over [cached ; new] keys
// (Sec. 3.3, Eq. 1-3) on tcgen05 tensor cores, for head_dim 128, bf16 caches
// and up to 128 query rows per (sequence, kv head).
//
// One CTA = one work unit (split s, kv head g, sequence b), the same units and
// partial outputs as the CUDA-core kernel, so the same merge follows.  All
// R = G * k query rows of the KV head's group share every K/V tile: the GQA
// group and the k soft-prompt rows together form the M side of the MMA.
//
// Per 64-token tile i:
//   S_i  = Q K_i^T            M = 128 query rows, N = 64 tokens, K = 128 dims,
//                             Q split into bf16 hi + lo (two MMAs per step),
//                             S double-buffered in TMEM
//   softmax                   4 warps, one query row per thread; the running
//                             max only moves when a row's max grows by more
//                             than 2^8, and O is rescaled in TMEM then
//   O   += P_i V_i            P written to shared memory as bf16 (K-major A),
//                             V read in place as an MN-major B operand
// Tiles come from a 3-stage ring filled by one producer warp: TMA for whole
// cache tiles of a paged pool, cp.async for contiguous caches, plain loads for
// the tile holding the sequence end and the new keys (and for pages that fail
// the bounds check, which are zero-filled and reported).
//
// Warps 0-3: softmax + epilogue; warp 4: producer; warp 5: TMEM owner and MMA
// issuer (lane 0).  Every wait is time-limited (SP_DEV_TIMEOUT).
#include <cudaTypedefs.h>
#include <string.h>

#include "sp_common.cuh"
#include "sp_sm100.cuh"

namespace sp {

namespace {

using namespace sm100;

constexpr int DH = 128;
constexpr int TT = 64;                         // tokens per tile
constexpr int STG = 3;                         // K/V ring depth
constexpr int DEFER = STG - 2;                 // cp.async tiles in flight beyond the current
constexpr int QSUB = 128 * 64 * 2;             // one [128 rows][64] bf16 swizzled sub-tile
constexpr int KVSUB = TT * 64 * 2;             // one [64 tokens][64] sub-tile
constexpr int KV_STAGE = 4 * KVSUB;            // K (2 subs) + V (2 subs)
constexpr int OFF_QHI = 0;
constexpr int OFF_QLO = OFF_QHI + 2 * QSUB;
constexpr int OFF_KV = OFF_QLO + 2 * QSUB;
constexpr int OFF_P = OFF_KV + STG * KV_STAGE;
constexpr int MAX_SPLIT_PAGES = 1024;          // page ids of one split staged in smem
constexpr int OFF_PAGES = OFF_P + 2 * QSUB;
constexpr int OFF_BAR = OFF_PAGES + MAX_SPLIT_PAGES * 4;
constexpr int SMEM_BYTES = OFF_BAR + 256 + 1024;
constexpr int THREADS = 192;
constexpr float RESCALE_LOG2 = 8.f;            // tolerate p <= 2^8 before rescaling O
constexpr uint32_t TMEM_COLS = 256;            // S0 [0,64), S1 [64,128), O [128,256)

// byte offset of 16-byte chunk `ch` (0..7) of row `row` in a swizzled sub-tile
__device__ __forceinline__ uint32_t swz(int row, int ch) {
    return (uint32_t)(row * 128 + ((ch ^ (row & 7)) << 4));
}

__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
    __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<uint32_t *>(&v);
}

struct Bars {
    uint64_t kv_full[STG], kv_empty[STG], s_full[2], p_full[2], pv_done[2], fin;
    uint32_t tmem;
    int abort;
};

__global__ void __launch_bounds__(THREADS, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap map_k,
                   const __grid_constant__ CUtensorMap map_v, AttnArgs a) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    Bars *bars = (Bars *)(smem + OFF_BAR);
    volatile int *abort = &bars->abort;
    const int s_idx = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int R = a.R, k = a.k;

    const SeqRef sq = resolve_seq(a.seq_ids, a.seq_lens, a.lens_by_batch, b, a.kv.n_seqs,
                                  a.max_seq_len,
                                  (threadIdx.x == 0 && s_idx == 0 && g == 0) ? a.status : nullptr);
    const int L = sq.len;
    const int total = L + k;
    const int t_begin = s_idx * a.split_tokens;
    if (t_begin >= total) return;  // uniform over the CTA; the merge never reads this unit
    const int t_end = min(total, t_begin + a.split_tokens);
    const int n_tiles = (t_end - t_begin + TT - 1) / TT;
    const int act_warps = (R + 31) / 32;  // softmax warps that own real query rows
    const bool paged = a.kv.layout == SP_KV_PAGED;

    if (threadIdx.x == 0) {
        for (int i = 0; i < STG; ++i) {
            mbar_init(&bars->kv_full[i], 32);
            mbar_init(&bars->kv_empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&bars->s_full[i], 1);
            mbar_init(&bars->p_full[i], 32 * act_warps);
            mbar_init(&bars->pv_done[i], 1);
        }
        mbar_init(&bars->fin, 1);
        bars->abort = 0;
        fence_mbar_init();
        if (paged) {
            prefetch_tmap(&map_k);
            prefetch_tmap(&map_v);
        }
    }
    if (warp == 5) {
        tmem_alloc(&bars->tmem, TMEM_COLS);
        tmem_relinquish();
    }
    // Q -> bf16 hi/lo, scaled to log2 units, rows rr = hl*k + r, zero past R
    if (warp < 4) {
        for (int idx = threadIdx.x; idx < 128 * 16; idx += 128) {
            const int row = idx >> 4, c16 = idx & 15;
            const int sub = c16 >> 3, ch = c16 & 7;
            uint32_t hi[4] = {0, 0, 0, 0}, lo[4] = {0, 0, 0, 0};
            if (row < R) {
                const int hl = row / k, r = row - hl * k;
                const float4 *src = (const float4 *)(a.q + (((size_t)b * k + r) * a.Hq +
                                                             g * a.G + hl) * DH + c16 * 8);
                const float4 x0 = src[0], x1 = src[1];
                const float v[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
                float h[8], l8[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const float x = v[e] * a.scale_log2;
                    h[e] = __bfloat162float(__float2bfloat16_rn(x));
                    l8[e] = x - h[e];
                }
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    hi[e] = pack_bf16(h[2 * e], h[2 * e + 1]);
                    lo[e] = pack_bf16(l8[2 * e], l8[2 * e + 1]);
                }
            }
            st_shared_v4(smem + OFF_QHI + sub * QSUB + swz(row, ch), hi[0], hi[1], hi[2], hi[3]);
            st_shared_v4(smem + OFF_QLO + sub * QSUB + swz(row, ch), lo[0], lo[1], lo[2], lo[3]);
        }
        fence_proxy_async();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = bars->tmem;

    if (warp == 4) {
        // ------------------------------------------------------------ producer
        int issued = 0;
        bool deferred[STG] = {false, false, false};  // contiguous tiles awaiting cp.async
        int bad = 0;
        const int P = a.kv.page_size;
        const int *ptab = paged ? a.kv.page_table + (size_t)max(sq.sid, 0) * a.kv.max_pages : nullptr;
        // this split's page ids, read once (coalesced) into shared memory;
        // entries past the page-table row read as -1
        int *spages = (int *)(smem + OFF_PAGES);
        const int lp0 = paged ? t_begin / P : 0;
        const int n_lp = paged ? min(MAX_SPLIT_PAGES, ceil_div(min(t_end, L) - t_begin, P)) : 0;
        for (int j = lane; j < n_lp; j += 32)
            spages[j] = (lp0 + j < a.kv.max_pages) ? ptab[lp0 + j] : -1;
        __syncwarp();
        for (int i = 0; i < n_tiles; ++i) {
            const int st = i % STG;
            if (!mbar_wait(&bars->kv_empty[st], ((i / STG) & 1) ^ 1, abort)) break;
            const int t0 = t_begin + i * TT;
            uint8_t *K = smem + OFF_KV + st * KV_STAGE;
            uint8_t *V = K + 2 * KVSUB;
            bool pure = (t0 + TT <= L);
            if (pure && paged) {
                const int npg = TT / P;
                bool ok = true;
                const int jl = (t0 - t_begin) / P;  // index into spages
                if (lane < npg) {
                    const int lp = t0 / P + lane;
                    const int page = jl + lane < n_lp ? spages[jl + lane]
                                                      : (lp < a.kv.max_pages ? ptab[lp] : -1);
                    ok = page >= 0 && page < a.kv.n_pages;
                    if (ok && a.gathered) a.gathered[(size_t)b * a.kv.max_pages + lp] = page;
                }
                pure = __all_sync(0xffffffffu, ok);
                if (pure) {
                    if (lane == 0) {
                        mbar_arrive_expect_tx(&bars->kv_full[st], KV_STAGE);
                        for (int j = 0; j < npg; ++j) {
                            const int page = jl + j < n_lp ? spages[jl + j] : ptab[t0 / P + j];
                            const int row = (page * a.Hkv + g) * P;
                            const uint32_t off = (uint32_t)(j * P * 128);
                            tma_load_2d(K + off, &map_k, &bars->kv_full[st], 0, row);
                            tma_load_2d(K + KVSUB + off, &map_k, &bars->kv_full[st], 64, row);
                            tma_load_2d(V + off, &map_v, &bars->kv_full[st], 0, row);
                            tma_load_2d(V + KVSUB + off, &map_v, &bars->kv_full[st], 64, row);
                        }
                    } else {
                        mbar_arrive(&bars->kv_full[st]);
                    }
                }
            } else if (pure) {
                // contiguous: token-major rows of 256 B, 16-byte cp.async per chunk
                const bf16 *kb = (const bf16 *)a.kv.k_seq[sq.sid];
                const bf16 *vb = (const bf16 *)a.kv.v_seq[sq.sid];
                for (int idx = lane; idx < TT * 16; idx += 32) {
                    const int row = idx >> 4, c16 = idx & 15;
                    const size_t src = ((size_t)(t0 + row) * a.Hkv + g) * DH + c16 * 8;
                    const uint32_t dst = (c16 >> 3) * KVSUB + swz(row, c16 & 7);
                    cp_async16(K + dst, kb + src);
                    cp_async16(V + dst, vb + src);
                }
                deferred[st] = true;
            }
            if (!pure) {
                // the sequence end / new keys / a bad page: plain loads, zero fill
                for (int idx = lane; idx < TT * 16; idx += 32) {
                    const int row = idx >> 4, c16 = idx & 15;
                    const int t = t0 + row;
                    const uint32_t dst = (c16 >> 3) * KVSUB + swz(row, c16 & 7);
                    uint4 kv4 = make_uint4(0, 0, 0, 0), vv4 = make_uint4(0, 0, 0, 0);
                    if (t < L) {
                        const bf16 *ks = nullptr, *vs = nullptr;
                        if (paged) {
                            const int lp = t / P;
                            const int page = lp < a.kv.max_pages ? ptab[lp] : -1;
                            if (page >= 0 && page < a.kv.n_pages) {
                                const size_t o = (((size_t)page * a.Hkv + g) * P + t % P) * DH + c16 * 8;
                                ks = (const bf16 *)a.kv.k_pool + o;
                                vs = (const bf16 *)a.kv.v_pool + o;
                                if (c16 == 0 && a.gathered && (t % P == 0 || row == 0))
                                    a.gathered[(size_t)b * a.kv.max_pages + lp] = page;
                            } else {
                                bad = 1;
                            }
                        } else {
                            const size_t o = ((size_t)t * a.Hkv + g) * DH + c16 * 8;
                            ks = (const bf16 *)a.kv.k_seq[sq.sid] + o;
                            vs = (const bf16 *)a.kv.v_seq[sq.sid] + o;
                        }
                        if (ks) {
                            kv4 = *(const uint4 *)ks;
                            vv4 = *(const uint4 *)vs;
                        }
                    } else if (t < total) {
                        const size_t o = (((size_t)b * k + (t - L)) * a.Hkv + g) * DH + c16 * 8;
                        const float4 *kf = (const float4 *)(a.k_new + o);
                        const float4 *vf = (const float4 *)(a.v_new + o);
                        const float4 k0 = kf[0], k1 = kf[1], v0 = vf[0], v1 = vf[1];
                        kv4 = make_uint4(pack_bf16(k0.x, k0.y), pack_bf16(k0.z, k0.w),
                                         pack_bf16(k1.x, k1.y), pack_bf16(k1.z, k1.w));
                        vv4 = make_uint4(pack_bf16(v0.x, v0.y), pack_bf16(v0.z, v0.w),
                                         pack_bf16(v1.x, v1.y), pack_bf16(v1.z, v1.w));
                    }
                    st_shared_v4(K + dst, kv4.x, kv4.y, kv4.z, kv4.w);
                    st_shared_v4(V + dst, vv4.x, vv4.y, vv4.z, vv4.w);
                }
                fence_proxy_async();
                mbar_arrive(&bars->kv_full[st]);
            }
            cp_async_commit();  // one (possibly empty) group per tile
            issued = i + 1;
            // A contiguous tile is published once its copies have landed, DEFER
            // tiles later.  The MMA warp frees tile i-STG only after tile
            // i-STG+1 is published, and this loop waits for that before issuing
            // tile i+1, so DEFER must stay below STG - 1.
            cp_async_wait<DEFER>();
            const int j = i - DEFER;
            if (j >= 0 && deferred[j % STG]) {
                fence_proxy_async();
                mbar_arrive(&bars->kv_full[j % STG]);
                deferred[j % STG] = false;
            }
        }
        cp_async_wait<0>();
        for (int j = issued - DEFER; j < issued; ++j) {
            if (j >= 0 && deferred[j % STG]) {
                fence_proxy_async();
                mbar_arrive(&bars->kv_full[j % STG]);
                deferred[j % STG] = false;
            }
        }
        if (lane == 0) {
            // drain TMA writes still in flight (only possible after an abort)
            for (int j = issued > STG ? issued - STG : 0; j < issued; ++j)
                mbar_wait_drain(&bars->kv_full[j % STG], (j / STG) & 1);
        }
        bad = __any_sync(0xffffffffu, bad);
        if (bad && lane == 0 && a.status) atomicOr(a.status, SP_DEV_BAD_PAGE);
    } else if (warp == 5) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc_s = idesc_bf16_f32(128, TT);
            constexpr uint32_t idesc_o = idesc_bf16_f32_bmn(128, DH);
            const uint32_t o_tmem = tmem + 128;
            auto issue_s = [&](int i) {
                const uint8_t *K = smem + OFF_KV + (i % STG) * KV_STAGE;
                const uint32_t s_tmem = tmem + (uint32_t)((i & 1) * TT);
#pragma unroll
                for (int kk = 0; kk < DH / 16; ++kk) {
                    const int sub = kk >> 2;
                    const uint32_t off = (uint32_t)((kk & 3) * 2);  // 32 B steps along dh
                    const uint64_t bk = sw128_kmajor_desc(K + sub * KVSUB) + off;
                    mma_bf16(s_tmem, sw128_kmajor_desc(smem + OFF_QHI + sub * QSUB) + off, bk,
                             idesc_s, kk > 0 ? 1u : 0u);
                    mma_bf16(s_tmem, sw128_kmajor_desc(smem + OFF_QLO + sub * QSUB) + off, bk,
                             idesc_s, 1u);
                }
                mma_commit(&bars->s_full[i & 1]);
            };
            bool ok = mbar_wait(&bars->kv_full[0], 0, abort);
            if (ok) {
                tc_fence_after();
                issue_s(0);
            }
            for (int i = 0; ok && i < n_tiles; ++i) {
                if (i + 1 < n_tiles) {
                    ok = mbar_wait(&bars->kv_full[(i + 1) % STG], ((i + 1) / STG) & 1, abort);
                    // S buffer (i+1)&1 was last read by the softmax of tile i-1
                    if (ok && i >= 1) ok = mbar_wait(&bars->p_full[(i + 1) & 1], ((i - 1) >> 1) & 1, abort);
                    if (!ok) break;
                    tc_fence_after();
                    issue_s(i + 1);
                }
                if (!mbar_wait(&bars->p_full[i & 1], (i >> 1) & 1, abort)) break;
                tc_fence_after();
                const uint8_t *V = smem + OFF_KV + (i % STG) * KV_STAGE + 2 * KVSUB;
                const uint8_t *Pt = smem + OFF_P + (i & 1) * QSUB;
#pragma unroll
                for (int kk = 0; kk < TT / 16; ++kk) {
                    mma_bf16(o_tmem, sw128_kmajor_desc(Pt) + (uint32_t)(kk * 2),
                             sw128_mnmajor_desc(V + kk * 2048, KVSUB), idesc_o,
                             (i > 0 || kk > 0) ? 1u : 0u);
                }
                mma_commit(&bars->kv_empty[i % STG]);
                mma_commit(&bars->pv_done[i & 1]);
            }
            mma_commit(&bars->fin);  // completes when every MMA above is done
        }
        __syncwarp();
    } else if (warp < act_warps) {
        // ------------------------------------------------------------ softmax
        const int row = threadIdx.x;  // == TMEM lane
        const bool active = row < R;
        const int r_soft = row % k;
        const uint32_t lane_base = tmem + ((uint32_t)(warp * 32) << 16);
        float m = -INFINITY, l = 0.f;
        bool ok = true;
        for (int i = 0; i < n_tiles; ++i) {
            if (!mbar_wait(&bars->s_full[i & 1], (i >> 1) & 1, abort)) {
                ok = false;
                break;
            }
            tc_fence_after();
            float sv[TT];
            {
                float t32[32];
                tmem_ld32(lane_base + (uint32_t)((i & 1) * TT), t32);
#pragma unroll
                for (int j = 0; j < 32; ++j) sv[j] = t32[j];
                tmem_ld32(lane_base + (uint32_t)((i & 1) * TT + 32), t32);
#pragma unroll
                for (int j = 0; j < 32; ++j) sv[32 + j] = t32[j];
            }
            const int t0 = t_begin + i * TT;
            if (t0 + TT > L) {
                const int lim = min(total, L + r_soft + 1);  // visible: t < lim
#pragma unroll
                for (int j = 0; j < TT; ++j)
                    if (t0 + j >= lim) sv[j] = -INFINITY;
            }
            float mt = -INFINITY;
#pragma unroll
            for (int j = 0; j < TT; ++j) mt = fmaxf(mt, sv[j]);
            if (!active) mt = -INFINITY;
            const bool grow = mt > m + RESCALE_LOG2 || (m == -INFINITY && mt != -INFINITY);
            const float m_new = grow ? mt : m;
            const float alpha = (grow && m != -INFINITY) ? exp2f(m - m_new) : (grow ? 0.f : 1.f);
            if (i > 0 && __any_sync(0xffffffffu, grow)) {
                // O holds tiles < i: wait for PV_{i-1}, then rescale the rows that moved
                if (!mbar_wait(&bars->pv_done[(i - 1) & 1], ((i - 1) >> 1) & 1, abort)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
#pragma unroll 1
                for (int c0 = 0; c0 < DH; c0 += 32) {
                    float o32[32];
                    tmem_ld32(lane_base + 128 + c0, o32);
#pragma unroll
                    for (int j = 0; j < 32; ++j) o32[j] *= alpha;
                    tmem_st32(lane_base + 128 + c0, o32);
                }
            }
            l *= alpha;
            m = m_new;
            float p[TT];
            float psum = 0.f;
#pragma unroll
            for (int j = 0; j < TT; ++j) {
                p[j] = (active && sv[j] != -INFINITY) ? exp2f(sv[j] - m) : 0.f;
                psum += p[j];
            }
            l += psum;
            // P buffer i&1 was last read by PV_{i-2}
            if (i >= 2 && !mbar_wait(&bars->pv_done[i & 1], ((i - 2) >> 1) & 1, abort)) {
                ok = false;
                break;
            }
            uint8_t *Pt = smem + OFF_P + (i & 1) * QSUB;
#pragma unroll
            for (int ch = 0; ch < 8; ++ch)
                st_shared_v4(Pt + swz(row, ch), pack_bf16(p[8 * ch], p[8 * ch + 1]),
                             pack_bf16(p[8 * ch + 2], p[8 * ch + 3]),
                             pack_bf16(p[8 * ch + 4], p[8 * ch + 5]),
                             pack_bf16(p[8 * ch + 6], p[8 * ch + 7]));
            fence_proxy_async();
            tc_fence_before();
            mbar_arrive(&bars->p_full[i & 1]);
        }
        // epilogue: the unnormalised partial of this unit
        if (ok && mbar_wait(&bars->pv_done[(n_tiles - 1) & 1], ((n_tiles - 1) >> 1) & 1, abort)) {
            tc_fence_after();
            const size_t unit = ((size_t)b * a.Hkv + g) * a.n_splits + s_idx;
            float *po = a.part_o + (unit * R + row) * DH;
#pragma unroll 1
            for (int c0 = 0; c0 < DH; c0 += 32) {
                float o32[32];
                tmem_ld32(lane_base + 128 + c0, o32);
                if (active) {
#pragma unroll
                    for (int j = 0; j < 32; j += 4)
                        *(float4 *)(po + c0 + j) = make_float4(o32[j], o32[j + 1], o32[j + 2], o32[j + 3]);
                }
            }
            if (active) {
                a.part_ml[(unit * R + row) * 2] = m;
                a.part_ml[(unit * R + row) * 2 + 1] = l;
            }
        }
    }
    // every MMA must be finished before TMEM and shared memory go away
    mbar_wait_drain(&bars->fin, 0);
    tc_fence_before();
    __syncthreads();
    if (threadIdx.x == 0 && *abort && a.status) atomicOr(a.status, SP_DEV_TIMEOUT);
    if (warp == 5) tmem_dealloc(tmem, TMEM_COLS);
}

}  // namespace

bool attention_tc_supported(const AttnArgs &a) {
    return a.dh == DH && a.kv_bf16 && a.R >= 1 && a.R <= 128 && a.split_tokens % TT == 0 &&
           (a.kv.layout == SP_KV_CONTIGUOUS ||
            (a.kv.page_size == 16 || a.kv.page_size == 32 || a.kv.page_size == 64));
}

cudaError_t launch_attention_tc(const AttnArgs &a, const CUtensorMap *map_k,
                                const CUtensorMap *map_v, cudaStream_t st) {
    static bool attr = false;
    if (!attr) {
        cudaError_t e = cudaFuncSetAttribute(attn_tc_kernel,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
        if (e != cudaSuccess) return e;
        attr = true;
    }
    CUtensorMap dummy;
    memset(&dummy, 0, sizeof dummy);
    dim3 grid(a.n_splits, a.Hkv, a.B);
    attn_tc_kernel<<<grid, THREADS, SMEM_BYTES, st>>>(map_k ? *map_k : dummy,
                                                      map_v ? *map_v : dummy, a);
    return cudaGetLastError();
}

}  // namespace sp
