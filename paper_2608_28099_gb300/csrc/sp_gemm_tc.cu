// Tensor-core projection for the decoder layer (Sec. 3.1: Q/K/V, output,
// gate/up and down projections): Y[M][N] = X[M][K] W[N][K]^T with bf16 weights.
//
// Work: tiles of 128 weight rows x BN activation rows, each over K in k-blocks
// of 64.  Weights are the MMA's A operand (M = 128), activations its B
// operand (N = BN): the handful of rows a classify call has fill the N side of
// the instruction instead of wasting 7/8 of a 128-row M tile.  Both operands
// arrive by TMA in 128-byte swizzled K-major tiles through mbarrier rings.
//
// Activations come as two bf16 planes hi = rn(x), lo = rn(x - hi), stored one
// after the other in each stage, so [hi; lo] is a single B operand of 2 BN rows:
// one MMA of N = 2 BN per 16-wide k-step reads the weight tile once and leaves
// W hi^T in TMEM columns [0, BN) and W lo^T in [BN, 2 BN); the epilogue adds
// the halves.  The product carries ~16 bits of the activation's mantissa.
// Without the lo plane (template flag LO = false) the activations are plain
// bf16: half the MMA work and activation traffic, a deeper ring.
//
// Two schedules, fp32 partials in planes of Y that the consumers add:
//  * tile kernel: one CTA per (tile, K split); split-K when the tiles alone
//    leave SMs idle.  Roles: warp 0 lane 0 TMA, warp 1 lane 0 MMA, warp 2
//    TMEM, all eight warps the epilogue (warp w: TMEM lanes 32 (w & 3).., the
//    column chunks of half w >> 2).  A gate/up projection with one K split can
//    apply SwiGLU in the epilogue instead of writing partials.
//  * persistent stream-K kernel, for tile counts that fill the SMs badly:
//    one CTA per SM owns the contiguous (tile, k-block) units [c L, (c+1) L)
//    in tile-major order.  Its weight and activation rings run across tile
//    boundaries (the weight stream never drains) and its accumulator is
//    double-buffered in TMEM (the epilogue of one tile segment overlaps the
//    MMAs of the next).  Segment j of a tile (in CTA order) stores plane j;
//    the CTA with the tile's last segment zero-fills the planes past it, so
//    every plane is written and the sum order is fixed (no atomics).  Roles:
//    warps 0-3 epilogue, warp 4 lane 0 weights, warp 5 lane 0 activations,
//    warp 6 TMEM and MMA.
#include <cudaTypedefs.h>

#include "sp_common.cuh"
#include "sp_gemm.cuh"
#include "sp_sm100.cuh"

namespace sp {

namespace {

using namespace sm100;

constexpr int BK = 64;               // bf16 elements per 128-byte swizzle row
constexpr int A_BYTES = 128 * BK * 2;

// ---------------------------------------------------------------- tile kernel
// LO: the activations come as hi and lo planes (the MMA's N side is [hi; lo],
// 2 BN rows), else as plain bf16 (N = BN).  NT: weight tiles per CTA sharing
// each activation k-block (2: twice the weight bytes in flight per stage for
// the same activation bytes; plain bf16 only), each with its own accumulator.
template <int BN, bool LO, int NT = 1>
struct TileCfg {
    static constexpr int B_BYTES = BN * BK * 2;
    static constexpr int NB = (LO ? 2 : 1) * BN;                 // MMA N
    static constexpr int STAGE = NT * A_BYTES + (LO ? 2 : 1) * B_BYTES;
    static constexpr int STAGES = 196608 / STAGE < 10 ? 196608 / STAGE : 10;  // 192 KB ring
    static constexpr int TMEM_COLS = NT * NB < 32 ? 32 : NT * NB;  // hi and lo halves per tile
    static constexpr int OFF_POS = STAGES * STAGE + 256;  // rotation epilogue: [BN] (pos, k_new row)
    static constexpr int SMEM = STAGES * STAGE + 1024 /*align*/ + 256 /*barriers*/ + BN * 8;
    static_assert(TMEM_COLS <= 512, "TMEM");
};

struct TcArgs {
    int M, N, K;
    int kb_per_split, n_kb;
    int w_blocked;    // weights stored as contiguous [tile][k-block][128][64] blocks
    float *y;         // [split][M][N]
    size_t split_stride;
    int *status;
    // failure-path test: CTA (0, 0, 0) never loads its first k-block, so its
    // MMA warp's wait runs out; every wait of the launch gives up after wait_ns
    int inject_stall;
    unsigned long long wait_ns;
    // SwiGLU epilogue (glu_f > 0, one K split): weight tile t holds gate rows
    // 64t..64t+63 then the matching up rows, and the CTA writes
    // glu[m][64t + j] = silu(gate) * up instead of a partial plane
    int glu_f;
    ActOut glu;
    // rotation epilogue (rope.rope_cs != NULL; RopeEpi)
    RopeEpi rope;
};

constexpr int TILE_THREADS = 256;  // warps 0-2 also TMA, MMA and TMEM owner

template <int BN, bool LO, int NT>
__global__ void __launch_bounds__(TILE_THREADS, 1)
    gemm_tile_kernel(const __grid_constant__ CUtensorMap map_w,
                   const __grid_constant__ CUtensorMap map_xhi,
                   const __grid_constant__ CUtensorMap map_xlo, TcArgs g) {
    using Cfg = TileCfg<BN, LO, NT>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint64_t *full = (uint64_t *)(smem + Cfg::STAGES * Cfg::STAGE);
    uint64_t *empty = full + Cfg::STAGES;
    uint64_t *done = empty + Cfg::STAGES;
    uint32_t *tmem_slot = (uint32_t *)(done + 1);
    volatile int *abort = (volatile int *)(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int m0 = blockIdx.x * BN, t0 = blockIdx.y * NT, n0 = t0 * 128;  // first weight tile
    const int kb0 = blockIdx.z * g.kb_per_split;
    const int nkb = min(g.kb_per_split, g.n_kb - kb0);
    pdl_trigger();

    if (threadIdx.x == 0) {
        for (int s = 0; s < Cfg::STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_init(done, 1);
        *abort = 0;
        fence_mbar_init();
        prefetch_tmap(&map_w);
        prefetch_tmap(&map_xhi);
        prefetch_tmap(&map_xlo);
    }
    if (warp == 2) {
        tmem_alloc(tmem_slot, Cfg::TMEM_COLS);
        tmem_relinquish();
    }
    // rotation epilogue: the rows' positions and k_new rows, resolved from the
    // caller's ids and lengths while the main loop runs (they need no wait)
    int2 *pos_s = (int2 *)(smem + Cfg::OFF_POS);
    const bool rope_on = g.rope.rope_cs != nullptr;
    if (rope_on && threadIdx.x >= 64) {
        for (int j = threadIdx.x - 64; j < BN; j += TILE_THREADS - 64) {
            const int m = m0 + j;
            int2 pm = make_int2(0, 0);
            if (m < g.M) {
                const int b = m / g.rope.k, r = m - b * g.rope.k;
                const SeqRef sq = resolve_seq(g.rope.seq_ids, g.rope.seq_lens, g.rope.lens_by_batch, b,
                                              g.rope.n_seqs, g.rope.max_seq_len,
                                              blockIdx.y == 0 ? g.rope.status : nullptr);
                pm.x = sq.len + g.rope.r0 + (g.rope.k_task ? r % g.rope.k_task : r);
                pm.y = b * (g.rope.kn_stride ? g.rope.kn_stride : g.rope.k) + g.rope.r0 + r;
            }
            pos_s[j] = pm;
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    int issued = 0;
    if (warp == 0 && lane == 0) {
        // producer: weights streamed once (evict-first), activations reused (evict-last).
        // The weights are constant, so the first ring of weight tiles is requested
        // before waiting for the previous kernel; the activations it writes after.
        const uint64_t pol_w = policy_evict_first();
        const uint64_t pol_x = policy_evict_last();
        const int pre = nkb < Cfg::STAGES ? nkb : Cfg::STAGES;
        const bool skip0 = g.inject_stall && blockIdx.x == 0 && blockIdx.y == 0 && blockIdx.z == 0;
        auto load_w = [&](int i, uint8_t *st, uint64_t *bar) {
#pragma unroll
            for (int j = 0; j < NT; ++j)
                tma_load_2d_hint(st + j * A_BYTES, &map_w, bar, g.w_blocked ? 0 : (kb0 + i) * BK,
                                 g.w_blocked ? ((t0 + j) * g.n_kb + kb0 + i) * 128 : n0 + j * 128, pol_w);
        };
        for (int i = 0; i < pre; ++i) {
            if (skip0 && i == 0) continue;
            mbar_arrive_expect_tx(&full[i], Cfg::STAGE);
            load_w(i, smem + i * Cfg::STAGE, &full[i]);
        }
        issued = pre;
        pdl_wait();
        for (int i = 0; i < nkb; ++i) {
            const int s = i % Cfg::STAGES;
            const uint32_t ph = (i / Cfg::STAGES) & 1;
            uint8_t *st = smem + s * Cfg::STAGE;
            const int kc = (kb0 + i) * BK;
            if (skip0 && i == 0) continue;
            if (i >= pre) {
                if (!mbar_wait(&empty[s], ph ^ 1, abort, g.wait_ns)) break;
                mbar_arrive_expect_tx(&full[s], Cfg::STAGE);
                load_w(i, st, &full[s]);
                issued = i + 1;
            }
            tma_load_2d_hint(st + NT * A_BYTES, &map_xhi, &full[s], kc, m0, pol_x);
            if (LO) tma_load_2d_hint(st + NT * A_BYTES + Cfg::B_BYTES, &map_xlo, &full[s], kc, m0, pol_x);
        }
    } else if (warp == 1 && lane == 0) {
        // MMA issuer
        constexpr uint32_t idesc = idesc_bf16_f32(128, Cfg::NB);
        for (int i = 0; i < nkb; ++i) {
            const int s = i % Cfg::STAGES;
            const uint32_t ph = (i / Cfg::STAGES) & 1;
            if (!mbar_wait(&full[s], ph, abort, g.wait_ns)) break;
            tc_fence_after();
            uint8_t *st = smem + s * Cfg::STAGE;
            const uint64_t bh = sw128_kmajor_desc(st + NT * A_BYTES);  // [hi; lo], 2 BN rows
#pragma unroll
            for (int kk = 0; kk < BK / 16; ++kk) {
#pragma unroll
                for (int j = 0; j < NT; ++j) {
                    // +32 bytes along K per 16-element MMA step (encoded >> 4)
                    const uint64_t a = sw128_kmajor_desc(st + j * A_BYTES);
                    mma_bf16(tmem + (uint32_t)(j * Cfg::NB), a + 2 * kk, bh + 2 * kk, idesc,
                             (i > 0 || kk > 0) ? 1u : 0u);
                }
            }
            mma_commit(&empty[s]);
        }
        mma_commit(done);  // completes once every MMA issued above has finished
    }
    __syncwarp();
    pdl_wait();  // before writing partials a previous kernel may still be reading

    // epilogue: TMEM -> registers -> fp32 partial tile
    const bool have = mbar_wait_drain(done, 0) && !*abort;
    tc_fence_after();
    // epilogue over all eight warps: warp w reads TMEM lanes 32 (w & 3).. and
    // the column chunks of half w >> 2
    const int quad = warp & 3, half = warp >> 2;
    if (rope_on && blockIdx.x == 0 && blockIdx.y == 0 && blockIdx.z == 0)
        for (int t = threadIdx.x; t < g.rope.n_zero; t += TILE_THREADS) g.rope.zero_ints[t] = 0;
#pragma unroll 1
    for (int tj = 0; tj < NT; ++tj) {
    const uint32_t trow = tmem + ((uint32_t)(quad * 32) << 16) + (uint32_t)(tj * Cfg::NB);
    if (rope_on) {
        if constexpr (BN >= 32) {
            // rotation epilogue, per 64-column chunk: the rows go through the idle
            // ring as in the SwiGLU epilogue, then thread (fq, cg) rotates pairs
            // (i, i + 64), i = 4 fq..4 fq + 3, of columns 4 cg..4 cg + 3 (TMEM
            // lanes i and 64 + i), or copies them for a value head
            float *xb = (float *)smem;
            const int row = quad * 32 + lane, fq = threadIdx.x & 15, cg = threadIdx.x >> 4;
            const int h = blockIdx.y, i = 4 * fq;  // head = weight tile
            const int Hq = g.rope.Hq, Hkv = g.rope.Hkv;
#pragma unroll 1
            for (int c0 = 0; c0 < BN; c0 += 64) {
                float *buf = xb + ((c0 >> 6) & 1) * (64 * 132);
                if (have && c0 + half * 32 < BN) {
                    float v[32], u[32] = {};
                    tmem_ld32(trow + c0 + half * 32, v);
                    if (LO) tmem_ld32(trow + BN + c0 + half * 32, u);
#pragma unroll
                    for (int j = 0; j < 32; ++j) buf[(half * 32 + j) * 132 + row] = v[j] + u[j];
                }
                __syncthreads();
                if (have) {
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const int cc = 4 * cg + e, m = m0 + c0 + cc;
                        if (c0 + cc >= BN || m >= g.M) break;
                        const float4 x0 = ld_shared_v4f(buf + cc * 132 + i);
                        const float4 x1 = ld_shared_v4f(buf + cc * 132 + 64 + i);
                        const int2 pm = pos_s[c0 + cc];
                        float *dst;
                        if (h < Hq + Hkv) {
                            const float2 *cs = g.rope.rope_cs + (size_t)pm.x * 64;
                            const float4 c01 = *(const float4 *)(cs + i), c23 = *(const float4 *)(cs + i + 2);
                            const float c[4] = {c01.x, c01.z, c23.x, c23.z}, sn[4] = {c01.y, c01.w, c23.y, c23.w};
                            const float a0[4] = {x0.x, x0.y, x0.z, x0.w}, a1[4] = {x1.x, x1.y, x1.z, x1.w};
                            float o0[4], o1[4];
#pragma unroll
                            for (int q4 = 0; q4 < 4; ++q4) {
                                o0[q4] = a0[q4] * c[q4] - a1[q4] * sn[q4];
                                o1[q4] = a1[q4] * c[q4] + a0[q4] * sn[q4];
                            }
                            dst = h < Hq ? g.rope.q + ((size_t)m * Hq + h) * 128
                                         : g.rope.k_new + ((size_t)pm.y * Hkv + (h - Hq)) * 128;
                            *(float4 *)(dst + i) = make_float4(o0[0], o0[1], o0[2], o0[3]);
                            *(float4 *)(dst + i + 64) = make_float4(o1[0], o1[1], o1[2], o1[3]);
                        } else {
                            dst = g.rope.v_new + ((size_t)pm.y * Hkv + (h - Hq - Hkv)) * 128;
                            *(float4 *)(dst + i) = x0;
                            *(float4 *)(dst + i + 64) = x1;
                        }
                    }
                }
            }
        }
    } else if (g.glu_f) {
        if constexpr (BN >= 32) {
            // SwiGLU epilogue, per 64-column chunk: every warp puts 32 columns of
            // its 32 rows (TMEM lanes) into the idle ring as [column][132] fp32
            // (two buffers), then thread (fq, cg) forms features 4 fq..4 fq + 3
            // of columns 4 cg..4 cg + 3 from gate rows 4 fq.. and up rows
            // 64 + 4 fq..: 16-byte shared loads, four features per store
            float *xb = (float *)smem;
            const int row = quad * 32 + lane, fq = threadIdx.x & 15, cg = threadIdx.x >> 4;
            const size_t feat = (size_t)(t0 + tj) * 64 + 4 * fq;
#pragma unroll 1
            for (int c0 = 0; c0 < BN; c0 += 64) {
                float *buf = xb + ((tj * ((BN + 63) / 64) + (c0 >> 6)) & 1) * (64 * 132);  // chunks alternate
                if (have && c0 + half * 32 < BN) {
                    float v[32], u[32] = {};
                    tmem_ld32(trow + c0 + half * 32, v);
                    if (LO) tmem_ld32(trow + BN + c0 + half * 32, u);
#pragma unroll
                    for (int j = 0; j < 32; ++j) buf[(half * 32 + j) * 132 + row] = v[j] + u[j];
                }
                __syncthreads();
                if (have) {
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const int cc = 4 * cg + e, m = m0 + c0 + cc;
                        if (c0 + cc >= BN || m >= g.M) break;
                        const float4 gt = ld_shared_v4f(buf + cc * 132 + 4 * fq);
                        const float4 up = ld_shared_v4f(buf + cc * 132 + 64 + 4 * fq);
                        act_store4(g.glu, (size_t)m * g.glu_f + feat,
                                   make_float4(__fdividef(gt.x, 1.f + __expf(-gt.x)) * up.x,
                                               __fdividef(gt.y, 1.f + __expf(-gt.y)) * up.y,
                                               __fdividef(gt.z, 1.f + __expf(-gt.z)) * up.z,
                                               __fdividef(gt.w, 1.f + __expf(-gt.w)) * up.w));
                    }
                }
            }
        }
    } else if (have) {
        const int n = n0 + tj * 128 + quad * 32 + lane;
        float *y = g.y + (size_t)blockIdx.z * g.split_stride;
        if constexpr (BN == 16) {
            if (half == 0) {
                float v[16], u[16] = {};
                tmem_ld16(trow, v);
                if (LO) tmem_ld16(trow + 16, u);
#pragma unroll
                for (int j = 0; j < 16; ++j) {
                    const int m = m0 + j;
                    if (m < g.M) y[(size_t)m * g.N + n] = v[j] + u[j];
                }
            }
        } else {
#pragma unroll 1
            for (int c0 = half * 32; c0 < BN; c0 += 64) {
                float v[32], u[32] = {};
                tmem_ld32(trow + c0, v);
                if (LO) tmem_ld32(trow + BN + c0, u);
#pragma unroll
                for (int j = 0; j < 32; ++j) {
                    const int m = m0 + c0 + j;
                    if (m < g.M) y[(size_t)m * g.N + n] = v[j] + u[j];
                }
            }
        }
    }
    }  // weight tiles of the CTA
    if (warp == 0 && lane == 0) {
        // no TMA write may still be in flight when the CTA's shared memory goes away
        for (int i = issued > Cfg::STAGES ? issued - Cfg::STAGES : 0; i < issued; ++i)
            mbar_wait_drain(&full[i % Cfg::STAGES], (i / Cfg::STAGES) & 1, g.wait_ns);
    }
    tc_fence_before();
    __syncthreads();
    if (threadIdx.x == 0 && *abort && g.status) atomicOr(g.status, SP_DEV_TIMEOUT);
    if (warp == 2) tmem_dealloc(tmem, Cfg::TMEM_COLS);
}

template <int BN, bool LO, int NT = 1>
cudaError_t launch_tile(const CUtensorMap &mw, const CUtensorMap &mh, const CUtensorMap &ml,
                      const TcArgs &g, dim3 grid, cudaStream_t st) {
    const int smem = TileCfg<BN, LO, NT>::SMEM;
    static bool attr_set = false;  // per device process-wide (one device per process here)
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(gemm_tile_kernel<BN, LO, NT>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    return launch_k(gemm_tile_kernel<BN, LO, NT>, grid, dim3(TILE_THREADS), (size_t)smem, st, mw, mh, ml,
                    g);
}


// ------------------------------------------------------ persistent stream-K
constexpr int GEMM_THREADS = 224;
constexpr int W_WARP = 4, X_WARP = 5, MMA_WARP_G = 6;

template <int BN, bool LO>
struct PkCfg {
    static constexpr int B_BYTES = BN * BK * 2;       // one activation plane of a k-block
    static constexpr int NB = (LO ? 2 : 1) * BN;      // MMA N
    static constexpr int X_STAGE = (LO ? 2 : 1) * B_BYTES;  // hi (+ lo)
    static constexpr int W_STAGES = BN <= 32 ? 8 : (BN == 64 ? 6 : (LO || BN == 256 ? 5 : 6));
    static constexpr int X_STAGES = BN <= 32 ? 4 : (LO || BN == 256 ? 3 : 4);
    static constexpr int ACC_COLS = NB < 32 ? 32 : NB;     // hi and lo halves
    static constexpr int TMEM_COLS = 2 * ACC_COLS;              // double-buffered
    static constexpr int OFF_X = W_STAGES * A_BYTES;
    static constexpr int OFF_BAR = OFF_X + X_STAGES * X_STAGE;
    static constexpr int SMEM = OFF_BAR + 512 /*barriers*/ + 1024 /*align*/;
    static_assert(SMEM <= 227 * 1024, "shared memory");
    static_assert((2 * W_STAGES + 2 * X_STAGES + 5) * 8 + 8 <= 512, "barrier area");
};

struct PkArgs {
    int M, N, n_kb, m_tiles, tiles;
    int w_blocked;    // weights stored as contiguous [tile][k-block][128][64] blocks
    int L;            // units per CTA
    int planes;       // partial planes in y
    float *y;         // [planes][M][N]
    size_t plane_stride;
    int *status;
};

// The CTA's tile segments: tiles t_first..t_last, k-blocks [lo, hi) of each.
struct Seg {
    int t, kb_lo, kb_hi;
};
__device__ __forceinline__ Seg segment(const PkArgs &g, long long u0, long long u1, int t) {
    const long long base = (long long)t * g.n_kb;
    Seg s;
    s.t = t;
    s.kb_lo = (int)(max(u0, base) - base);
    s.kb_hi = (int)(min(u1, base + g.n_kb) - base);
    return s;
}

template <int BN, bool LO>
__global__ void __launch_bounds__(GEMM_THREADS, 1)
    gemm_pk_kernel(const __grid_constant__ CUtensorMap map_w,
                   const __grid_constant__ CUtensorMap map_xhi,
                   const __grid_constant__ CUtensorMap map_xlo, PkArgs g) {
    using Cfg = PkCfg<BN, LO>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint64_t *w_full = (uint64_t *)(smem + Cfg::OFF_BAR);
    uint64_t *w_empty = w_full + Cfg::W_STAGES;
    uint64_t *x_full = w_empty + Cfg::W_STAGES;
    uint64_t *x_empty = x_full + Cfg::X_STAGES;
    uint64_t *acc_full = x_empty + Cfg::X_STAGES;  // [2]
    uint64_t *acc_empty = acc_full + 2;             // [2]
    uint64_t *done = acc_empty + 2;
    uint32_t *tmem_slot = (uint32_t *)(done + 1);
    volatile int *abort = (volatile int *)(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const long long U = (long long)g.tiles * g.n_kb;
    const long long u0 = (long long)blockIdx.x * g.L;
    const long long u1 = min(U, u0 + g.L);
    pdl_trigger();
    if (u0 >= U) {
        pdl_wait();
        return;  // uniform over the CTA
    }
    const int t_first = (int)(u0 / g.n_kb), t_last = (int)((u1 - 1) / g.n_kb);

    if (threadIdx.x == 0) {
        for (int s = 0; s < Cfg::W_STAGES; ++s) {
            mbar_init(&w_full[s], 1);
            mbar_init(&w_empty[s], 1);
        }
        for (int s = 0; s < Cfg::X_STAGES; ++s) {
            mbar_init(&x_full[s], 1);
            mbar_init(&x_empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&acc_full[b], 1);
            mbar_init(&acc_empty[b], 128);
        }
        mbar_init(done, 1);
        *abort = 0;
        fence_mbar_init();
        prefetch_tmap(&map_w);
        prefetch_tmap(&map_xhi);
        prefetch_tmap(&map_xlo);
    }
    if (warp == MMA_WARP_G) {
        tmem_alloc(tmem_slot, Cfg::TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    int issued = 0;  // TMA k-blocks issued by this producer
    if (warp == W_WARP && lane == 0) {
        // weights: streamed once (evict-first) and constant, so loading starts
        // before the previous kernel has finished
        const uint64_t pol_w = policy_evict_first();
        int i = 0;
        bool ok = true;
        for (int t = t_first; ok && t <= t_last; ++t) {
            const Seg sg = segment(g, u0, u1, t);
            const int n0 = (t / g.m_tiles) * 128;
            for (int kb = sg.kb_lo; kb < sg.kb_hi; ++kb, ++i) {
                const int s = i % Cfg::W_STAGES;
                if (i >= Cfg::W_STAGES && !mbar_wait(&w_empty[s], ((i / Cfg::W_STAGES) & 1) ^ 1, abort)) {
                    ok = false;
                    break;
                }
                mbar_arrive_expect_tx(&w_full[s], A_BYTES);
                tma_load_2d_hint(smem + s * A_BYTES, &map_w, &w_full[s], g.w_blocked ? 0 : kb * BK,
                                 g.w_blocked ? ((t / g.m_tiles) * g.n_kb + kb) * 128 : n0, pol_w);
                issued = i + 1;
            }
        }
    } else if (warp == X_WARP && lane == 0) {
        // activations (re-read by every CTA: evict-last), written by the previous kernel
        const uint64_t pol_x = policy_evict_last();
        pdl_wait();
        int i = 0;
        bool ok = true;
        for (int t = t_first; ok && t <= t_last; ++t) {
            const Seg sg = segment(g, u0, u1, t);
            const int m0 = (t % g.m_tiles) * BN;
            for (int kb = sg.kb_lo; kb < sg.kb_hi; ++kb, ++i) {
                const int s = i % Cfg::X_STAGES;
                if (i >= Cfg::X_STAGES && !mbar_wait(&x_empty[s], ((i / Cfg::X_STAGES) & 1) ^ 1, abort)) {
                    ok = false;
                    break;
                }
                uint8_t *st = smem + Cfg::OFF_X + s * Cfg::X_STAGE;
                mbar_arrive_expect_tx(&x_full[s], Cfg::X_STAGE);
                tma_load_2d_hint(st, &map_xhi, &x_full[s], kb * BK, m0, pol_x);
                if (LO) tma_load_2d_hint(st + Cfg::B_BYTES, &map_xlo, &x_full[s], kb * BK, m0, pol_x);
                issued = i + 1;
            }
        }
    } else if (warp == MMA_WARP_G && lane == 0) {
        constexpr uint32_t idesc = idesc_bf16_f32(128, Cfg::NB);
        int i = 0, sgi = 0;
        bool ok = true;
        for (int t = t_first; ok && t <= t_last; ++t, ++sgi) {
            const Seg sg = segment(g, u0, u1, t);
            const int buf = sgi & 1;
            const uint32_t acc = tmem + (uint32_t)(buf * Cfg::ACC_COLS);
            // the epilogue has drained this buffer's previous segment
            if (sgi >= 2 && !mbar_wait(&acc_empty[buf], ((sgi >> 1) - 1) & 1, abort)) break;
            tc_fence_after();
            for (int kb = sg.kb_lo; kb < sg.kb_hi; ++kb, ++i) {
                const int sw = i % Cfg::W_STAGES, sx = i % Cfg::X_STAGES;
                if (!mbar_wait(&w_full[sw], (i / Cfg::W_STAGES) & 1, abort) ||
                    !mbar_wait(&x_full[sx], (i / Cfg::X_STAGES) & 1, abort)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint8_t *xs = smem + Cfg::OFF_X + sx * Cfg::X_STAGE;
                const uint64_t a = sw128_kmajor_desc(smem + sw * A_BYTES);
                const uint64_t bh = sw128_kmajor_desc(xs);  // [hi; lo], 2 BN rows
#pragma unroll
                for (int kk = 0; kk < BK / 16; ++kk) {
                    // +32 bytes along K per 16-element MMA step (encoded >> 4)
                    mma_bf16(acc, a + 2 * kk, bh + 2 * kk, idesc, (kb > sg.kb_lo || kk > 0) ? 1u : 0u);
                }
                mma_commit(&w_empty[sw]);
                mma_commit(&x_empty[sx]);
            }
            if (ok) mma_commit(&acc_full[buf]);
        }
        mma_commit(done);  // completes once every MMA issued above has finished
    } else if (warp < 4) {
        // epilogue: TMEM -> registers -> fp32 partial plane of each tile segment
        pdl_wait();  // before writing partials a previous kernel may still be reading
        const int r = warp * 32 + lane;  // weight row within the tile (TMEM lane)
        const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);
        int sgi = 0;
        for (int t = t_first; t <= t_last; ++t, ++sgi) {
            const int buf = sgi & 1;
            if (!mbar_wait(&acc_full[buf], (sgi >> 1) & 1, abort)) break;
            tc_fence_after();
            const int n = (t / g.m_tiles) * 128 + r;
            const int m0 = (t % g.m_tiles) * BN;
            const int plane = blockIdx.x - (int)(((long long)t * g.n_kb) / g.L);
            const int last = (int)((((long long)t + 1) * g.n_kb - 1) / g.L);
            float *y = g.y + (size_t)plane * g.plane_stride;
            const uint32_t ta = trow + (uint32_t)(buf * Cfg::ACC_COLS);
            if constexpr (BN == 16) {
                float v[16], u[16] = {};
                tmem_ld16(ta, v);
                if (LO) tmem_ld16(ta + 16, u);
#pragma unroll
                for (int j = 0; j < 16; ++j) {
                    const int m = m0 + j;
                    if (m < g.M) y[(size_t)m * g.N + n] = v[j] + u[j];
                }
            } else {
#pragma unroll 1
                for (int c0 = 0; c0 < BN; c0 += 32) {
                    float v[32], u[32] = {};
                    tmem_ld32(ta + c0, v);
                    if (LO) tmem_ld32(ta + BN + c0, u);
#pragma unroll
                    for (int j = 0; j < 32; ++j) {
                        const int m = m0 + c0 + j;
                        if (m < g.M) y[(size_t)m * g.N + n] = v[j] + u[j];
                    }
                }
            }
            tc_fence_before();
            mbar_arrive(&acc_empty[buf]);
            if ((int)blockIdx.x == last) {
                // planes past the tile's last segment hold zeros
                for (int p = plane + 1; p < g.planes; ++p) {
                    float *yz = g.y + (size_t)p * g.plane_stride;
                    for (int j = 0; j < BN; ++j) {
                        const int m = m0 + j;
                        if (m < g.M) yz[(size_t)m * g.N + n] = 0.f;
                    }
                }
            }
        }
    }
    __syncwarp();
    if (lane == 0) mbar_wait_drain(done, 0);
    // no TMA write may still be in flight when the CTA's shared memory goes away
    if (warp == W_WARP && lane == 0)
        for (int i = issued > Cfg::W_STAGES ? issued - Cfg::W_STAGES : 0; i < issued; ++i)
            mbar_wait_drain(&w_full[i % Cfg::W_STAGES], (i / Cfg::W_STAGES) & 1);
    if (warp == X_WARP && lane == 0)
        for (int i = issued > Cfg::X_STAGES ? issued - Cfg::X_STAGES : 0; i < issued; ++i)
            mbar_wait_drain(&x_full[i % Cfg::X_STAGES], (i / Cfg::X_STAGES) & 1);
    tc_fence_before();
    __syncthreads();
    if (threadIdx.x == 0 && *abort && g.status) atomicOr(g.status, SP_DEV_TIMEOUT);
    if (warp == MMA_WARP_G) tmem_dealloc(tmem, Cfg::TMEM_COLS);
}

template <int BN, bool LO>
cudaError_t launch_pk(const CUtensorMap &mw, const CUtensorMap &mh, const CUtensorMap &ml,
                      const PkArgs &g, int grid, cudaStream_t st) {
    const int smem = PkCfg<BN, LO>::SMEM;
    static bool attr_set = false;  // per device process-wide (one device per process here)
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(gemm_pk_kernel<BN, LO>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    return launch_k(gemm_pk_kernel<BN, LO>, dim3(grid), dim3(GEMM_THREADS), (size_t)smem, st, mw, mh, ml,
                    g);
}

}  // namespace

// ---------------------------------------------------------------------------
// host side: tensor maps and the plan
// ---------------------------------------------------------------------------
static PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        cudaDriverEntryPointQueryResult q;
        void *p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = (PFN_cuTensorMapEncodeTiled_v12000)p;
    }
    return fn;
}

bool encode_kmajor_bf16(CUtensorMap *map, const void *base, int rows, int K, int box_rows) {
    PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
    if (!fn || ((uintptr_t)base & 15) || (K * 2) % 16) return false;
    cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)K * 2};
    cuuint32_t box[2] = {(cuuint32_t)BK, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims,
                    strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

bool encode_kv_pages_bf16(CUtensorMap *map, const void *pool, long long n_page_heads, int page_size) {
    // pool [n_page_heads][page_size][128] bf16 viewed as (64 dims, 8 rows,
    // 2 dim halves, row groups of 8): one box = one (page, head) block laid out
    // in shared memory as [row group][dim half][8 rows][128 B], 128-byte swizzle
    PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
    if (!fn || ((uintptr_t)pool & 15) || page_size % 8 || page_size > 64) return false;
    const long long groups = n_page_heads * (page_size / 8);
    if (groups <= 0 || groups > 0x7fffffffLL) return false;
    cuuint64_t dims[4] = {64, 8, 2, (cuuint64_t)groups};
    cuuint64_t strides[3] = {256, 128, 2048};
    cuuint32_t box[4] = {64, 8, 2, (cuuint32_t)(page_size / 8)};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(pool), dims, strides,
                    box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

bool encode_q_group_f32(CUtensorMap *map, const float *q, int rows, int Hq, int G, int k) {
    // q [rows = B*k][Hq][128] fp32; one box = the G heads of one kv group for
    // the k rows of one sequence: [k][G][128], unswizzled
    PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
    if (!fn || ((uintptr_t)q & 15) || G > 256 || k > 256) return false;
    cuuint64_t dims[3] = {128, (cuuint64_t)Hq, (cuuint64_t)rows};
    cuuint64_t strides[2] = {128 * 4, (cuuint64_t)Hq * 128 * 4};
    cuuint32_t box[3] = {128, (cuuint32_t)G, (cuuint32_t)k};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, const_cast<float *>(q), dims, strides,
                    box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

int tc_bn_for(int M, bool lo) {
    if (M <= 16) return 16;
    if (M <= 32) return 32;
    if (M <= 64) return 64;
    return (!lo && M >= 256) ? 256 : 128;
}

bool tc_supported(int N, int K) { return N % 128 == 0 && K % BK == 0 && K >= BK; }

// Partial planes the stream-K split needs: the most CTAs any tile spans.
static int planes_for(long long tiles, int n_kb, long long L) {
    int most = 1;
    for (long long t = 0; t < tiles; ++t) {
        const long long c0 = t * n_kb / L, c1 = ((t + 1) * n_kb - 1) / L;
        if (c1 - c0 + 1 > most) most = (int)(c1 - c0 + 1);
    }
    return most;
}

TcPlan tc_plan(int M, int N, int K, int n_sm, size_t y_capacity_bytes, bool lo, int sched) {
    TcPlan p;
    p.nt = 1;
    p.bn = tc_bn_for(M, lo);
    p.m_tiles = ceil_div(M, p.bn);
    p.n_tiles = N / 128;
    p.n_kb = K / BK;
    const int tiles = p.m_tiles * p.n_tiles;
    // Tile kernel: split K until one wave of CTAs covers the SMs (>= 2 k-blocks
    // per split, partials within the buffer).
    int S = 1;
    if (tiles < n_sm) {
        S = n_sm / tiles;
        const int max_s = p.n_kb / 2 > 0 ? p.n_kb / 2 : 1;
        if (S > max_s) S = max_s;
    }
    while (S > 1 && (size_t)S * M * N * sizeof(float) > y_capacity_bytes) --S;
    p.kb_per_split = ceil_div(p.n_kb, S);
    p.splits = ceil_div(p.n_kb, p.kb_per_split);  // no empty split
    p.persistent = false;
    p.grid = tiles * p.splits;
    p.units_per_cta = p.kb_per_split;
    // Persistent stream-K when the tile kernel's last wave would leave more
    // than a fifth of the SMs idle and the extra partial planes are cheap
    // (estimates in units of one CTA's k-block time, 16 KB of weights).
    const int waves = ceil_div(tiles * p.splits, n_sm);
    const double fill = (double)tiles * p.splits / ((double)waves * n_sm);
    // Two weight tiles per CTA (plain bf16, up to 128 rows: HBM-bound): each stage
    // carries twice the weight bytes for the same activation bytes.  Taken when
    // the paired grid still fills ~all SMs in one wave with no more K splits
    // (extra splits cost the consumer more partial planes than the pairing saves:
    // 27b_long gate/up 65.5 -> 63.4 us, its down projection unchanged at 7
    // splits instead of 3 while the readout slowed by 2 us).
    if (sched == 0 && !lo && p.bn <= 128 && p.n_tiles % 2 == 0) {
        const int pairs = p.m_tiles * (p.n_tiles / 2);
        int S2 = 1;
        if (pairs < n_sm) {
            S2 = n_sm / pairs;
            const int max_s = p.n_kb / 2 > 0 ? p.n_kb / 2 : 1;
            if (S2 > max_s) S2 = max_s;
        }
        while (S2 > 1 && (size_t)S2 * M * N * sizeof(float) > y_capacity_bytes) --S2;
        const int kbs2 = ceil_div(p.n_kb, S2);
        S2 = ceil_div(p.n_kb, kbs2);
        // (S2 <= splits also keeps an unsplit gate/up unsplit for its SwiGLU epilogue)
        if (S2 <= p.splits && pairs * S2 <= n_sm && pairs * S2 * 100 >= n_sm * 85) {
            p.nt = 2;
            p.kb_per_split = kbs2;
            p.splits = S2;
            p.grid = pairs * S2;
            p.units_per_cta = kbs2;
            return p;
        }
    }
    if (sched == 1) return p;
    if (sched == 2 || (waves > 1 && fill < 0.8)) {
        const long long U = (long long)tiles * p.n_kb;
        long long L = (U + n_sm - 1) / n_sm;
        if (L < 2) L = 2;
        const int planes = planes_for(tiles, p.n_kb, L);
        const double plane_units = 2.0 * (double)M * N * 4.0 / ((double)n_sm * 16384.0);
        const double cost_tile = (double)waves * (p.kb_per_split + 4);
        const double cost_pk = (double)L + 4.0 + planes * plane_units;
        if ((sched == 2 || cost_pk < cost_tile) && (size_t)planes * M * N * sizeof(float) <= y_capacity_bytes) {
            p.persistent = true;
            p.units_per_cta = (int)L;
            p.splits = planes;
            p.grid = (int)((U + L - 1) / L);
        }
    }
    return p;
}

cudaError_t launch_gemm_tc(const CUtensorMap &map_w, const CUtensorMap &map_xhi,
                           const CUtensorMap &map_xlo, const TcPlan &p, int M, int N, int K,
                           float *y, int *status, cudaStream_t st, bool w_blocked, bool lo,
                           int inject_stall, const ActOut *glu, const RopeEpi *rope) {
    if (p.persistent) {
        PkArgs g;
        g.M = M;
        g.N = N;
        g.n_kb = p.n_kb;
        g.m_tiles = p.m_tiles;
        g.tiles = p.m_tiles * p.n_tiles;
        g.w_blocked = w_blocked;
        g.L = p.units_per_cta;
        g.planes = p.splits;
        g.y = y;
        g.plane_stride = (size_t)M * N;
        g.status = status;
        switch (p.bn) {
        case 16: return lo ? launch_pk<16, true>(map_w, map_xhi, map_xlo, g, p.grid, st)
                        : launch_pk<16, false>(map_w, map_xhi, map_xlo, g, p.grid, st);
        case 32: return lo ? launch_pk<32, true>(map_w, map_xhi, map_xlo, g, p.grid, st)
                        : launch_pk<32, false>(map_w, map_xhi, map_xlo, g, p.grid, st);
        case 64: return lo ? launch_pk<64, true>(map_w, map_xhi, map_xlo, g, p.grid, st)
                        : launch_pk<64, false>(map_w, map_xhi, map_xlo, g, p.grid, st);
        case 128: return lo ? launch_pk<128, true>(map_w, map_xhi, map_xlo, g, p.grid, st)
                        : launch_pk<128, false>(map_w, map_xhi, map_xlo, g, p.grid, st);
        case 256: return lo ? cudaErrorInvalidValue  // N = 512: beyond one MMA
                        : launch_pk<256, false>(map_w, map_xhi, map_xlo, g, p.grid, st);
        default: return cudaErrorInvalidValue;
        }
    }
    TcArgs g;
    g.M = M;
    g.N = N;
    g.K = K;
    g.kb_per_split = p.kb_per_split;
    g.n_kb = p.n_kb;
    g.w_blocked = w_blocked;
    g.y = y;
    g.split_stride = (size_t)M * N;
    g.status = status;
    g.inject_stall = inject_stall;
    g.wait_ns = inject_stall ? 1000000ull : sm100::kWaitLimitNs;
    g.glu_f = 0;
    memset(&g.glu, 0, sizeof g.glu);
    memset(&g.rope, 0, sizeof g.rope);
    if (rope) {
        if (p.persistent || p.splits != 1 || p.nt != 1 || p.bn < 32 || glu) return cudaErrorInvalidValue;
        g.rope = *rope;
    }
    if (glu) {
        if (p.persistent || p.splits != 1 || p.bn < 32 || N % 128) return cudaErrorInvalidValue;
        g.glu_f = N / 2;
        g.glu = *glu;
    }
    dim3 grid(p.m_tiles, p.n_tiles / p.nt, p.splits);
    if (p.nt == 2) {
        if (lo || p.n_tiles % 2) return cudaErrorInvalidValue;
        switch (p.bn) {
        case 16: return launch_tile<16, false, 2>(map_w, map_xhi, map_xlo, g, grid, st);
        case 32: return launch_tile<32, false, 2>(map_w, map_xhi, map_xlo, g, grid, st);
        case 64: return launch_tile<64, false, 2>(map_w, map_xhi, map_xlo, g, grid, st);
        case 128: return launch_tile<128, false, 2>(map_w, map_xhi, map_xlo, g, grid, st);
        default: return cudaErrorInvalidValue;
        }
    }
    switch (p.bn) {
    case 16: return lo ? launch_tile<16, true>(map_w, map_xhi, map_xlo, g, grid, st)
                    : launch_tile<16, false>(map_w, map_xhi, map_xlo, g, grid, st);
    case 32: return lo ? launch_tile<32, true>(map_w, map_xhi, map_xlo, g, grid, st)
                    : launch_tile<32, false>(map_w, map_xhi, map_xlo, g, grid, st);
    case 64: return lo ? launch_tile<64, true>(map_w, map_xhi, map_xlo, g, grid, st)
                    : launch_tile<64, false>(map_w, map_xhi, map_xlo, g, grid, st);
    case 128: return lo ? launch_tile<128, true>(map_w, map_xhi, map_xlo, g, grid, st)
                    : launch_tile<128, false>(map_w, map_xhi, map_xlo, g, grid, st);
    case 256: return lo ? cudaErrorInvalidValue  // N = 512: beyond one MMA
                    : launch_tile<256, false>(map_w, map_xhi, map_xlo, g, grid, st);
    default: return cudaErrorInvalidValue;
    }
}

}  // namespace sp
