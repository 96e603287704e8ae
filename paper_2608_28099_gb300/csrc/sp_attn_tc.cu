// Split-KV attention of the k appended rows over [cached ; new] keys
// (Sec. 3.3, Eq. 1-3) on tcgen05 tensor cores, for head_dim 128, bf16 caches
// and up to 128 query rows per (sequence, kv head).
//
// One CTA = one work unit (split s, kv head g, sequence b), the same units and
// partial outputs as the CUDA-core kernel, so the same merge follows.  All
// R = G * k query rows of the KV head's group share every K/V tile: the GQA
// group and the k soft-prompt rows together form the M side of the MMA.
//
// Per 64-token tile i (w = i & 1):
//   S_i   = Q K_i^T           M = 128 query rows, N = 64 tokens, K = 128 dims,
//                             Q split into bf16 hi + lo held in TMEM (the
//                             MMA's A operand, two MMAs per step), into TMEM
//                             buffer S_w
//   softmax                   warpgroup w (tiles alternate between two
//                             warpgroups), one query row per thread; a row's
//                             running max only moves when its max grows by
//                             more than 2^8, and O_w is rescaled in TMEM then
//   O_w  += P_i V_i           P written as bf16 over the first half of S_w (A
//                             operand from TMEM), V read in place from shared
//                             memory as an MN-major B operand
// Each warpgroup keeps its own (max, sum, O_w); at the end warpgroup 0 folds
// warpgroup 1's state into its own (both O accumulators sit on the same TMEM
// lanes) and writes the unit's one partial.  The last unit of a (sequence, kv
// head) to finish (a counter per pair, cleared by the preceding kernel)
// combines the pair's partials in the exp2 domain and writes the output; with
// many units per pair the host leaves that to attn_merge_kernel instead.  The
// even and odd tiles form two independent pipelines, each with its own MMA
// issuing warp: one thread issuing small-N MMAs back to back leaves the tensor
// pipe idle between them, two keep it busy.
// Tiles come from a 6-stage ring: TMA for whole cache tiles of a paged pool
// (one box per (page, kv head) block of K and of V, issued by two lead warps
// taking alternate tiles), cp.async for contiguous caches, plain loads for the
// tile holding the sequence end and the new keys (and for pages that fail the
// bounds check, which are zero-filled and reported).
//
// Tile layout in shared memory (K and V alike, 64 tokens x 128 dims bf16):
// [8-token group][dim half][8 tokens][64 dims], 128-byte swizzle, so that a
// (page, head) block of 16/32/64 tokens is one TMA box and both MMAs read the
// tile with uniform strides (8-token groups 2048 B apart, dim halves 1024 B).
//
// Warps 0-3 and 4-7: the two softmax warpgroups (+ epilogue); warps 8 and 11:
// producers; warp 9: TMEM owner and MMA issuer of even tiles; warp 10: MMA
// issuer of odd tiles.  Every wait is time-limited (SP_DEV_TIMEOUT).
#include <cudaTypedefs.h>
#include <string.h>

#include "sp_common.cuh"
#include "sp_sm100.cuh"

namespace sp {

namespace {

using namespace sm100;

constexpr int DH = 128;
constexpr int TT = 64;                         // tokens per tile
constexpr int STG = 6;                         // K/V ring depth
// cp.async tiles in flight beyond the current one.  Tile j is published at
// producer iteration j + DEFER, which first waits for stage j + DEFER - STG to
// be released; the MMA warp needs tiles 0 and 1 before its first PV and tile
// i + 2 before it releases stage i + 1, so DEFER <= STG - 2 (else deadlock).
constexpr int DEFER = STG - 2;
static_assert(DEFER >= 0 && DEFER <= STG - 2, "cp.async publication depth");
constexpr int KV_TILE = TT * DH * 2;           // K or V of one tile, 16 KB
constexpr int KV_STAGE = 2 * KV_TILE;          // K then V
constexpr uint32_t GROUP_STRIDE = 2048;        // 8-token groups
constexpr uint32_t HALF_STRIDE = 1024;         // 64-dim halves within a group
constexpr int OFF_KV = 0;
constexpr int MAX_SPLIT_PAGES = 1024;          // page ids of one split staged in smem
constexpr int OFF_PAGES = OFF_KV + STG * KV_STAGE;
constexpr int OFF_BAR = OFF_PAGES + MAX_SPLIT_PAGES * 4;
constexpr int OFF_ML = OFF_BAR + 256;           // warpgroup 1's (max, sum) per row
constexpr int SMEM_BYTES = OFF_ML + 1024 + 1024;
constexpr int THREADS = 384;                   // 2 softmax warpgroups, 2 producers, 2 MMA
constexpr int PRODUCER_WARP = 8, MMA_WARP = 9, MMA_WARP1 = 10, PRODUCER_WARP1 = 11;
constexpr float RESCALE_LOG2 = 8.f;            // tolerate p <= 2^8 before rescaling O
// TMEM columns: S0 [0,64) S1 [64,128) O0 [128,256) O1 [256,384) Qhi [384,448) Qlo [448,512);
// P_w (64 bf16 per row) overwrites the first 32 columns of S_w once S_w is read.
constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t O_COL = 128, QHI_COL = 384, QLO_COL = 448;

// byte offset of 16-byte chunk c16 (0..15, 8 dims each) of token row `row`
// (0..63) in a K or V tile
__device__ __forceinline__ uint32_t kv_off(int row, int c16) {
    return (uint32_t)((row >> 3) * GROUP_STRIDE + (c16 >> 3) * HALF_STRIDE + (row & 7) * 128 +
                      (((c16 & 7) ^ (row & 7)) << 4));
}

__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
    __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<uint32_t *>(&v);
}

struct Bars {
    uint64_t kv_full[STG], kv_empty[STG], s_full[2], p_full[2], pv_done[2], fin, q_full;  // fin: 2 arrivals
    uint32_t tmem;
    int abort;
    int last;  // this CTA merges its (sequence, kv head)
};

__global__ void __launch_bounds__(THREADS, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap map_k,
                   const __grid_constant__ CUtensorMap map_v,
                   const __grid_constant__ CUtensorMap map_q, AttnArgs a) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    Bars *bars = (Bars *)(smem + OFF_BAR);
    volatile int *abort = &bars->abort;
    const int s_idx = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int R = a.R, k = a.k;
    pdl_trigger();

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
    // producers: warps 8 and 11, plus the softmax warps that own no rows (they
    // help with the cp.async and plain-load tiles; warps 8 and 11 issue TMA)
    const int n_prod = 2 + 2 * (4 - act_warps);
    const bool is_producer = warp == PRODUCER_WARP || warp == PRODUCER_WARP1 ||
                             (warp < 8 && (warp & 3) >= act_warps);
    const int pidx = warp == PRODUCER_WARP    ? 0
                     : warp == PRODUCER_WARP1 ? 1
                                              : 2 + (warp >> 2) * (4 - act_warps) + ((warp & 3) - act_warps);
    const bool paged = a.kv.layout == SP_KV_PAGED;

    if (threadIdx.x == 0) {
        for (int i = 0; i < STG; ++i) {
            mbar_init(&bars->kv_full[i], 32 * n_prod);
            mbar_init(&bars->kv_empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&bars->s_full[i], 1);
            mbar_init(&bars->p_full[i], 32 * act_warps);
            mbar_init(&bars->pv_done[i], 1);
        }
        mbar_init(&bars->fin, 2);
        mbar_init(&bars->q_full, 1);
        bars->abort = 0;
        fence_mbar_init();
        prefetch_tmap(&map_q);
        if (paged) {
            prefetch_tmap(&map_k);
            prefetch_tmap(&map_v);
        }
    }
    if (warp == MMA_WARP) {
        tmem_alloc(&bars->tmem, TMEM_COLS);
        tmem_relinquish();
    }
    // the producer stages this split's page ids while warpgroup 0 writes Q
    const int P = a.kv.page_size;
    const int *ptab = paged ? a.kv.page_table + (size_t)max(sq.sid, 0) * a.kv.max_pages : nullptr;
    int *spages = (int *)(smem + OFF_PAGES);
    const int lp0 = paged ? t_begin / P : 0;
    const int n_lp = paged ? min(MAX_SPLIT_PAGES, max(0, ceil_div(min(t_end, L) - t_begin, P))) : 0;
    pdl_wait();  // the rotated queries and new keys come from the previous kernel
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = bars->tmem;
    // one TMA brings this group's queries [k][G][128] fp32 into the first ring
    // stages (free until the pipeline starts)
    float *qs = (float *)(smem + OFF_KV);
    if (warp == PRODUCER_WARP) {
        if (lane == 0) {
            mbar_arrive_expect_tx(&bars->q_full, (uint32_t)(R * DH * 4));
            tma_load_3d(qs, &map_q, &bars->q_full, 0, g * a.G, b * k);
        }
        for (int j = lane; j < n_lp; j += 32)
            spages[j] = (lp0 + j < a.kv.max_pages) ? ptab[lp0 + j] : -1;
    }
    // Q -> bf16 hi/lo in TMEM (row rr = hl*k + r on lane rr; zero past R),
    // scaled to log2 units: 64 columns of packed pairs for hi, 64 for lo
    if (warp < 4) {
        const int row = threadIdx.x;
        const uint32_t lane_base = tmem + ((uint32_t)(warp * 32) << 16);
        const bool have_q = mbar_wait_drain(&bars->q_full, 0);
        const float4 *src = nullptr;
        if (row < R && have_q) {
            const int hl = row / k, r = row - hl * k;
            src = (const float4 *)(qs + (r * a.G + hl) * DH);
        }
#pragma unroll
        for (int half = 0; half < 2; ++half) {
            uint32_t hi[32], lo[32];
#pragma unroll
            for (int c4 = 0; c4 < 16; ++c4) {
                const float4 x = src ? src[half * 16 + c4] : make_float4(0.f, 0.f, 0.f, 0.f);
                const float v[4] = {x.x * a.scale_log2, x.y * a.scale_log2, x.z * a.scale_log2,
                                    x.w * a.scale_log2};
                float h[4], l4[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    h[e] = __bfloat162float(__float2bfloat16_rn(v[e]));
                    l4[e] = v[e] - h[e];
                }
                hi[2 * c4] = pack_bf16(h[0], h[1]);
                hi[2 * c4 + 1] = pack_bf16(h[2], h[3]);
                lo[2 * c4] = pack_bf16(l4[0], l4[1]);
                lo[2 * c4 + 1] = pack_bf16(l4[2], l4[3]);
            }
            tmem_st32u(lane_base + QHI_COL + half * 32, hi);
            tmem_st32u(lane_base + QLO_COL + half * 32, lo);
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();

    if (is_producer) {
        // ------------------------------------------------------------ producers
        const int ptid = pidx * 32 + lane, pstride = 32 * n_prod;
        const bool tma_warp = pidx < 2;  // warps 8 and 11 issue TMA for even and odd tiles
        int issued = 0;
        bool deferred[STG] = {false, false, false};  // contiguous tiles awaiting cp.async
        int bad = 0;
        for (int i = 0; i < n_tiles; ++i) {
            const int st = i % STG;
            if (!mbar_wait(&bars->kv_empty[st], ((i / STG) & 1) ^ 1, abort)) break;
            const int t0 = t_begin + i * TT;
            uint8_t *K = smem + OFF_KV + st * KV_STAGE;
            uint8_t *V = K + KV_TILE;
            const bool lead = pidx == (i & 1);
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
                pure = __all_sync(0xffffffffu, ok);  // every producer warp reaches the same verdict
                if (pure && !lead) {
                    mbar_arrive(&bars->kv_full[st]);
                } else if (pure) {
                    // one TMA box per lane: lane = 2 * page + (K, V), each the
                    // (page, head) block of P tokens; lane 0 registers the
                    // stage's bytes before any box is issued
                    if (lane == 0) mbar_arrive_expect_tx(&bars->kv_full[st], KV_STAGE);
                    __syncwarp();
                    if (lane < 2 * npg) {
                        const int j = lane >> 1, part = lane & 1;
                        const int page = jl + j < n_lp ? spages[jl + j] : ptab[t0 / P + j];
                        const int grp = (page * a.Hkv + g) * (P / 8);
                        tma_load_4d((part ? V : K) + j * P * 256, part ? &map_v : &map_k,
                                    &bars->kv_full[st], 0, 0, 0, grp);
                    }
                    if (lane != 0) mbar_arrive(&bars->kv_full[st]);
                }
            } else if (pure) {
                // contiguous: token-major rows of 256 B, 16-byte cp.async per chunk
                const bf16 *kb = (const bf16 *)a.kv.k_seq[sq.sid];
                const bf16 *vb = (const bf16 *)a.kv.v_seq[sq.sid];
                for (int idx = ptid; idx < TT * 16; idx += pstride) {
                    const int row = idx >> 4, c16 = idx & 15;
                    const size_t src = ((size_t)(t0 + row) * a.Hkv + g) * DH + c16 * 8;
                    const uint32_t dst = kv_off(row, c16);
                    cp_async16(K + dst, kb + src);
                    cp_async16(V + dst, vb + src);
                }
                deferred[st] = true;
            }
            if (!pure) {
                // the sequence end / new keys / a bad page: plain loads, zero fill
                for (int idx = ptid; idx < TT * 16; idx += pstride) {
                    const int row = idx >> 4, c16 = idx & 15;
                    const int t = t0 + row;
                    const uint32_t dst = kv_off(row, c16);
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
            // a contiguous tile is published once its copies have landed, DEFER
            // tiles later (see DEFER)
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
        if (tma_warp && lane == 0) {
            // drain TMA writes still in flight (only possible after an abort)
            for (int j = issued > STG ? issued - STG : 0; j < issued; ++j)
                if ((j & 1) == pidx) mbar_wait_drain(&bars->kv_full[j % STG], (j / STG) & 1);
        }
        bad = __any_sync(0xffffffffu, bad);
        if (bad && lane == 0 && a.status) atomicOr(a.status, SP_DEV_BAD_PAGE);
    } else if (warp == MMA_WARP || warp == MMA_WARP1) {
        // ------------------------------------------------------------ MMA issuers
        // Pipeline w = warp - MMA_WARP takes tiles i = w, w + 2, ...: S_w, then
        // per tile i: PV_i (after softmax i) and S_{i+2} (reusing S buffer w).
        // PV_i does not wait for any later tile's data, so stage i is released
        // as soon as its softmax is done.
        const int w = warp - MMA_WARP;
        if (lane == 0) {
            constexpr uint32_t idesc_s = idesc_bf16_f32(128, TT);
            constexpr uint32_t idesc_o = idesc_bf16_f32_bmn(128, DH);
            const uint32_t s_tmem = tmem + (uint32_t)(w * TT);  // S_w; P_w over its first half
            const uint32_t o_tmem = tmem + O_COL + (uint32_t)(w * DH);
            auto issue_s = [&](int i) {
                const uint8_t *K = smem + OFF_KV + (i % STG) * KV_STAGE;
#pragma unroll
                for (int kk = 0; kk < DH / 16; ++kk) {
                    // 16 dims = 32 B along a 128-byte row of dim half kk / 4
                    const uint64_t bk =
                        sw128_kmajor_desc_sbo(K + (kk >> 2) * HALF_STRIDE, GROUP_STRIDE) +
                        (uint64_t)((kk & 3) * 2);
                    // 16 dims of Q = 8 TMEM columns
                    mma_bf16_ts(s_tmem, tmem + QHI_COL + (uint32_t)(kk * 8), bk, idesc_s,
                                kk > 0 ? 1u : 0u);
                    mma_bf16_ts(s_tmem, tmem + QLO_COL + (uint32_t)(kk * 8), bk, idesc_s, 1u);
                }
                mma_commit(&bars->s_full[w]);
            };
            bool ok = true;
            if (w < n_tiles) {
                ok = mbar_wait(&bars->kv_full[w % STG], (w / STG) & 1, abort);
                if (ok) {
                    tc_fence_after();
                    issue_s(w);
                }
            }
            for (int i = w; ok && i < n_tiles; i += 2) {
                if (!mbar_wait(&bars->p_full[w], (i >> 1) & 1, abort)) break;
                tc_fence_after();
                const uint8_t *V = smem + OFF_KV + (i % STG) * KV_STAGE + KV_TILE;
#pragma unroll
                for (int kk = 0; kk < TT / 16; ++kk) {
                    // 16 tokens of P = 8 TMEM columns; 16 tokens of V = two 8-token groups
                    mma_bf16_ts(o_tmem, s_tmem + (uint32_t)(kk * 8),
                                sw128_mnmajor_desc2(V + kk * 2 * GROUP_STRIDE, HALF_STRIDE, GROUP_STRIDE),
                                idesc_o, (i >= 2 || kk > 0) ? 1u : 0u);
                }
                mma_commit(&bars->kv_empty[i % STG]);
                mma_commit(&bars->pv_done[w]);
                if (i + 2 < n_tiles) {
                    // S buffer w is free: softmax i has read it (p_full above)
                    if (!mbar_wait(&bars->kv_full[(i + 2) % STG], ((i + 2) / STG) & 1, abort)) break;
                    tc_fence_after();
                    issue_s(i + 2);
                }
            }
            mma_commit(&bars->fin);  // completes when every MMA of this issuer is done
        }
        __syncwarp();
    } else if (warp < 8 && (warp & 3) < act_warps) {
        // ------------------------------------------------------------ softmax
        const int wg = warp >> 2;       // warpgroup: tiles i with (i & 1) == wg
        const int row = threadIdx.x & 127;  // == TMEM lane
        const bool active = row < R;
        const int r_soft = row % k;
        const uint32_t lane_base = tmem + ((uint32_t)((warp & 3) * 32) << 16);
        const uint32_t s_col = (uint32_t)(wg * TT), o_col = O_COL + (uint32_t)(wg * DH);
        float m = -INFINITY, l = 0.f;
        bool ok = true;
        for (int i = wg; i < n_tiles; i += 2) {
            const uint32_t ph = (i >> 1) & 1;
            if (!mbar_wait(&bars->s_full[wg], ph, abort)) {
                ok = false;
                break;
            }
            tc_fence_after();
            float sv[TT];
            {
                float t32[32];
                tmem_ld32(lane_base + s_col, t32);
#pragma unroll
                for (int j = 0; j < 32; ++j) sv[j] = t32[j];
                tmem_ld32(lane_base + s_col + 32, t32);
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
            // tile max as an 8-way tree
            float mx[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) mx[e] = fmaxf(sv[e], sv[e + 8]);
#pragma unroll
            for (int j = 16; j < TT; j += 8)
#pragma unroll
                for (int e = 0; e < 8; ++e) mx[e] = fmaxf(mx[e], sv[j + e]);
            const float mt = fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])),
                                   fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7])));
            const bool grow = active && (mt > m + RESCALE_LOG2 || (m == -INFINITY && mt != -INFINITY));
            const float m_new = grow ? mt : m;
            const float alpha = grow ? (m == -INFINITY ? 0.f : fast_exp2(m - m_new)) : 1.f;
            // O_wg and P_wg were last used by PV_{i-2}
            if (i >= 2) {
                if (!mbar_wait(&bars->pv_done[wg], ((i - 2) >> 1) & 1, abort)) {
                    ok = false;
                    break;
                }
                if (__any_sync(0xffffffffu, grow)) {
                    tc_fence_after();
#pragma unroll 1
                    for (int c0 = 0; c0 < DH; c0 += 32) {
                        float o32[32];
                        tmem_ld32(lane_base + o_col + c0, o32);
#pragma unroll
                        for (int j = 0; j < 32; ++j) o32[j] *= alpha;
                        tmem_st32(lane_base + o_col + c0, o32);
                    }
                }
            }
            l *= alpha;
            m = m_new;
            const float mu = (m == -INFINITY) ? 0.f : m;  // a fully masked row gives p = 0
            float ps[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
            uint32_t pk[TT / 2];
#pragma unroll
            for (int j = 0; j < TT; j += 2) {
                const float p0 = fast_exp2(sv[j] - mu);
                const float p1 = fast_exp2(sv[j + 1] - mu);
                ps[(j >> 1) & 7] += p0 + p1;
                pk[j >> 1] = pack_bf16(p0, p1);
            }
            l += ((ps[0] + ps[1]) + (ps[2] + ps[3])) + ((ps[4] + ps[5]) + (ps[6] + ps[7]));
            tmem_st32u(lane_base + s_col, pk);  // P_i over the first half of S_i
            tc_fence_before();
            mbar_arrive(&bars->p_full[wg]);
        }
        // epilogue: warpgroup 1 hands its (max, sum) to warpgroup 0 through shared
        // memory; warpgroup 0 combines (max, sum, O) of both and writes the unit's
        // unnormalised partial
        float *sm_ml = (float *)(smem + OFF_ML);
        const int last0 = n_tiles >= 1 ? n_tiles - 1 - ((n_tiles - 1) & 1) : -1;  // WG0's last tile
        const int last1 = n_tiles >= 2 ? n_tiles - 1 - (n_tiles & 1) : -1;        // WG1's last tile
        if (wg == 1) {
            sm_ml[row] = last1 >= 0 ? m : -INFINITY;
            sm_ml[128 + row] = last1 >= 0 ? l : 0.f;
        }
        asm volatile("bar.sync 1, %0;" ::"r"(64 * act_warps) : "memory");
        if (wg == 0) {
            const size_t unit = ((size_t)b * a.Hkv + g) * a.n_splits + s_idx;
            float *po = a.part_o + (unit * R + row) * DH;
            const float m1 = sm_ml[row], l1 = sm_ml[128 + row];
            const float mc = fmaxf(m, m1);
            const float a0 = (m == -INFINITY) ? 0.f : fast_exp2(m - mc);
            const float a1 = (m1 == -INFINITY) ? 0.f : fast_exp2(m1 - mc);
            bool have = ok && last0 >= 0 && mbar_wait(&bars->pv_done[0], (last0 >> 1) & 1, abort);
            if (have && last1 >= 0) have = mbar_wait(&bars->pv_done[1], (last1 >> 1) & 1, abort);
            have = __all_sync(0xffffffffu, have);  // the TMEM loads below are warp-collective
            if (have) {
                tc_fence_after();
#pragma unroll 1
                for (int c0 = 0; c0 < DH; c0 += 32) {
                    float o0[32], o1[32];
                    tmem_ld32(lane_base + O_COL + c0, o0);
                    if (last1 >= 0) {
                        tmem_ld32(lane_base + O_COL + DH + c0, o1);
                    } else {
#pragma unroll
                        for (int j = 0; j < 32; ++j) o1[j] = 0.f;
                    }
                    if (active) {
#pragma unroll
                        for (int j = 0; j < 32; j += 4)
                            *(float4 *)(po + c0 + j) =
                                make_float4(a0 * o0[j] + a1 * o1[j], a0 * o0[j + 1] + a1 * o1[j + 1],
                                            a0 * o0[j + 2] + a1 * o1[j + 2], a0 * o0[j + 3] + a1 * o1[j + 3]);
                    }
                }
                if (active) {
                    a.part_ml[(unit * R + row) * 2] = mc;
                    a.part_ml[(unit * R + row) * 2 + 1] = a0 * l + a1 * l1;
                }
            }
            __threadfence();  // the partial is visible device-wide before this unit is counted
        }
    }
    // every MMA must be finished before TMEM and shared memory go away
    mbar_wait_drain(&bars->fin, 0);
    tc_fence_before();
    __syncthreads();
    if (threadIdx.x == 0 && *abort && a.status) atomicOr(a.status, SP_DEV_TIMEOUT);
    if (warp == MMA_WARP) tmem_dealloc(tmem, TMEM_COLS);

    // ---------------------------------------------------------------- merge
    if (!a.counters) return;  // merged by a separate kernel
    const int n_units = min(a.n_splits, ceil_div(total, a.split_tokens));
    int *counter = a.counters + (size_t)b * a.Hkv + g;
    if (threadIdx.x == 0) {
        bars->last = atomicAdd(counter, 1) == n_units - 1;
        __threadfence();
    }
    __syncthreads();
    if (!bars->last) return;
    // every unit of the pair has written its partial: combine them.  Pass 1: per
    // row, the normalised weight of each partial (shared memory, over the
    // free K/V ring); pass 2: per (row, 4 columns), the weighted sum.
    const size_t p0 = ((size_t)b * a.Hkv + g) * a.n_splits;
    float *wn = (float *)(smem + OFF_KV);  // [R][n_units]
    for (int rr = threadIdx.x; rr < R; rr += THREADS) {
        float mmax = -INFINITY;
#pragma unroll 8
        for (int p = 0; p < n_units; ++p) mmax = fmaxf(mmax, __ldcg(a.part_ml + ((p0 + p) * R + rr) * 2));
        float l = 0.f;
#pragma unroll 8
        for (int p = 0; p < n_units; ++p) {
            const float2 ml = __ldcg((const float2 *)(a.part_ml + ((p0 + p) * R + rr) * 2));
            const float w = (ml.x == -INFINITY) ? 0.f : exp2f(ml.x - mmax);
            wn[rr * n_units + p] = w;
            l += w * ml.y;
        }
        const float inv = l > 0.f ? 1.f / l : 0.f;
        for (int p = 0; p < n_units; ++p) wn[rr * n_units + p] *= inv;
    }
    __syncthreads();
    for (int idx = threadIdx.x; idx < R * (DH / 4); idx += THREADS) {
        const int rr = idx / (DH / 4), c = (idx % (DH / 4)) * 4;
        float4 o = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 8
        for (int p = 0; p < n_units; ++p) {
            const float w = wn[rr * n_units + p];
            const float4 op = __ldcg((const float4 *)(a.part_o + ((p0 + p) * R + rr) * DH + c));
            o.x += w * op.x;
            o.y += w * op.y;
            o.z += w * op.z;
            o.w += w * op.w;
        }
        const int hl = rr / k, r = rr - hl * k;
        const int h = g * a.G + hl;
        act_store4(a.out, (((size_t)b * k + r) * a.Hq + h) * DH + c, o);
    }
    if (threadIdx.x == 0) *counter = 0;  // ready for a launch that does not clear it
}

}  // namespace

bool attention_tc_supported(const AttnArgs &a) {
    return a.dh == DH && a.kv_bf16 && a.R >= 1 && a.R <= 128 && a.split_tokens % TT == 0 &&
           (a.kv.layout == SP_KV_CONTIGUOUS ||
            (a.kv.page_size == 16 || a.kv.page_size == 32 || a.kv.page_size == 64));
}

cudaError_t launch_attention_tc(const AttnArgs &a, const CUtensorMap *map_k,
                                const CUtensorMap *map_v, const CUtensorMap &map_q,
                                cudaStream_t st) {
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
    return launch_k(attn_tc_kernel, grid, dim3(THREADS), SMEM_BYTES, st, map_k ? *map_k : dummy,
                    map_v ? *map_v : dummy, map_q, a);
}

}  // namespace sp
