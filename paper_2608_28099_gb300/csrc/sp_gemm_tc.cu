// Tensor-core projection for the decoder layer (Sec. 3.1: Q/K/V, output,
// gate/up and down projections): Y[M][N] = X[M][K] W[N][K]^T with bf16 weights.
//
// One CTA computes a 128 (weight rows) x BN (activation rows) tile over its
// share of K with tcgen05.mma, accumulating in TMEM.  Weights are the MMA's A
// operand (M = 128), activations its B operand (N = BN): the handful of rows a
// classify call has fill the N side of the instruction instead of wasting
// 7/8 of a 128-row M tile.  Both operands arrive by TMA in 128-byte swizzled
// K-major tiles through a STAGES-deep mbarrier ring.
//
// Activations come as two bf16 planes hi = rn(x), lo = rn(x - hi); every
// k-block issues W*hi and W*lo into the same accumulator, so the product
// carries ~16 bits of the activation's mantissa for the price of a second MMA
// (free while the projection is bound by weight bandwidth).
//
// Split-K: blockIdx.z takes a contiguous range of k-blocks and stores an fp32
// partial tile; the consumer kernels add the partials.
//
// Roles: warp 0 lane 0 issues TMA, warp 1 lane 0 issues MMA, warp 2 owns
// TMEM, all four warps run the epilogue (warp w reads TMEM lanes 32w..32w+31).
#include <cudaTypedefs.h>

#include "sp_common.cuh"
#include "sp_gemm.cuh"
#include "sp_sm100.cuh"

namespace sp {

namespace {

using namespace sm100;

constexpr int BK = 64;               // bf16 elements per 128-byte swizzle row
constexpr int A_BYTES = 128 * BK * 2;

template <int BN>
struct TcCfg {
    static constexpr int B_BYTES = BN * BK * 2;
    static constexpr int STAGE = A_BYTES + 2 * B_BYTES;
    static constexpr int STAGES = (BN <= 32) ? 8 : (BN == 64 ? 6 : 4);
    static constexpr int TMEM_COLS = BN < 32 ? 32 : BN;
    static constexpr int SMEM = STAGES * STAGE + 1024 /*align*/ + 256 /*barriers*/;
};

struct TcArgs {
    int M, N, K;
    int kb_per_split, n_kb;
    float *y;         // [split][M][N]
    size_t split_stride;
    int *status;
};

template <int BN>
__global__ void __launch_bounds__(128, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap map_w,
                   const __grid_constant__ CUtensorMap map_xhi,
                   const __grid_constant__ CUtensorMap map_xlo, TcArgs g) {
    using Cfg = TcCfg<BN>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint64_t *full = (uint64_t *)(smem + Cfg::STAGES * Cfg::STAGE);
    uint64_t *empty = full + Cfg::STAGES;
    uint64_t *done = empty + Cfg::STAGES;
    uint32_t *tmem_slot = (uint32_t *)(done + 1);
    volatile int *abort = (volatile int *)(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int m0 = blockIdx.x * BN, n0 = blockIdx.y * 128;
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
        for (int i = 0; i < pre; ++i) {
            mbar_arrive_expect_tx(&full[i], Cfg::STAGE);
            tma_load_2d_hint(smem + i * Cfg::STAGE, &map_w, &full[i], (kb0 + i) * BK, n0, pol_w);
        }
        issued = pre;
        pdl_wait();
        for (int i = 0; i < nkb; ++i) {
            const int s = i % Cfg::STAGES;
            const uint32_t ph = (i / Cfg::STAGES) & 1;
            uint8_t *st = smem + s * Cfg::STAGE;
            const int kc = (kb0 + i) * BK;
            if (i >= pre) {
                if (!mbar_wait(&empty[s], ph ^ 1, abort)) break;
                mbar_arrive_expect_tx(&full[s], Cfg::STAGE);
                tma_load_2d_hint(st, &map_w, &full[s], kc, n0, pol_w);
                issued = i + 1;
            }
            tma_load_2d_hint(st + A_BYTES, &map_xhi, &full[s], kc, m0, pol_x);
            tma_load_2d_hint(st + A_BYTES + Cfg::B_BYTES, &map_xlo, &full[s], kc, m0, pol_x);
        }
    } else if (warp == 1 && lane == 0) {
        // MMA issuer
        constexpr uint32_t idesc = idesc_bf16_f32(128, BN);
        for (int i = 0; i < nkb; ++i) {
            const int s = i % Cfg::STAGES;
            const uint32_t ph = (i / Cfg::STAGES) & 1;
            if (!mbar_wait(&full[s], ph, abort)) break;
            tc_fence_after();
            uint8_t *st = smem + s * Cfg::STAGE;
            const uint64_t a = sw128_kmajor_desc(st);
            const uint64_t bh = sw128_kmajor_desc(st + A_BYTES);
            const uint64_t bl = sw128_kmajor_desc(st + A_BYTES + Cfg::B_BYTES);
#pragma unroll
            for (int kk = 0; kk < BK / 16; ++kk) {
                // +32 bytes along K per 16-element MMA step (encoded >> 4)
                mma_bf16(tmem, a + 2 * kk, bh + 2 * kk, idesc, (i > 0 || kk > 0) ? 1u : 0u);
                mma_bf16(tmem, a + 2 * kk, bl + 2 * kk, idesc, 1u);
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
    if (have) {
        const int n = n0 + warp * 32 + lane;
        float *y = g.y + (size_t)blockIdx.z * g.split_stride;
        const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);
        if constexpr (BN == 16) {
            float v[16];
            tmem_ld16(trow, v);
#pragma unroll
            for (int j = 0; j < 16; ++j) {
                const int m = m0 + j;
                if (m < g.M) y[(size_t)m * g.N + n] = v[j];
            }
        } else {
#pragma unroll 1
            for (int c0 = 0; c0 < BN; c0 += 32) {
                float v[32];
                tmem_ld32(trow + c0, v);
#pragma unroll
                for (int j = 0; j < 32; ++j) {
                    const int m = m0 + c0 + j;
                    if (m < g.M) y[(size_t)m * g.N + n] = v[j];
                }
            }
        }
    }
    if (warp == 0 && lane == 0) {
        // no TMA write may still be in flight when the CTA's shared memory goes away
        for (int i = issued > Cfg::STAGES ? issued - Cfg::STAGES : 0; i < issued; ++i)
            mbar_wait_drain(&full[i % Cfg::STAGES], (i / Cfg::STAGES) & 1);
    }
    tc_fence_before();
    __syncthreads();
    if (threadIdx.x == 0 && *abort && g.status) atomicOr(g.status, SP_DEV_TIMEOUT);
    if (warp == 2) tmem_dealloc(tmem, Cfg::TMEM_COLS);
}

template <int BN>
cudaError_t launch_bn(const CUtensorMap &mw, const CUtensorMap &mh, const CUtensorMap &ml,
                      const TcArgs &g, dim3 grid, cudaStream_t st) {
    const int smem = TcCfg<BN>::SMEM;
    static bool attr_set = false;  // per device process-wide (one device per process here)
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(gemm_tc_kernel<BN>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    return launch_k(gemm_tc_kernel<BN>, grid, dim3(128), (size_t)smem, st, mw, mh, ml, g);
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

int tc_bn_for(int M) {
    if (M <= 16) return 16;
    if (M <= 32) return 32;
    if (M <= 64) return 64;
    return 128;
}

bool tc_supported(int N, int K) { return N % 128 == 0 && K % BK == 0 && K >= BK; }

TcPlan tc_plan(int M, int N, int K, int n_sm, size_t y_capacity_bytes) {
    TcPlan p;
    p.bn = tc_bn_for(M);
    p.m_tiles = ceil_div(M, p.bn);
    p.n_tiles = N / 128;
    p.n_kb = K / BK;
    const int tiles = p.m_tiles * p.n_tiles;
    int S = 1;
    if (tiles < n_sm) {
        S = n_sm / tiles;
        const int max_s = p.n_kb / 2 > 0 ? p.n_kb / 2 : 1;  // >= 2 k-blocks per split
        if (S > max_s) S = max_s;
    }
    while (S > 1 && (size_t)S * M * N * sizeof(float) > y_capacity_bytes) --S;
    p.kb_per_split = ceil_div(p.n_kb, S);
    p.splits = ceil_div(p.n_kb, p.kb_per_split);  // no empty split
    return p;
}

cudaError_t launch_gemm_tc(const CUtensorMap &map_w, const CUtensorMap &map_xhi,
                           const CUtensorMap &map_xlo, const TcPlan &p, int M, int N, int K,
                           float *y, int *status, cudaStream_t st) {
    TcArgs g;
    g.M = M;
    g.N = N;
    g.K = K;
    g.kb_per_split = p.kb_per_split;
    g.n_kb = p.n_kb;
    g.y = y;
    g.split_stride = (size_t)M * N;
    g.status = status;
    dim3 grid(p.m_tiles, p.n_tiles, p.splits);
    switch (p.bn) {
    case 16: return launch_bn<16>(map_w, map_xhi, map_xlo, g, grid, st);
    case 32: return launch_bn<32>(map_w, map_xhi, map_xlo, g, grid, st);
    case 64: return launch_bn<64>(map_w, map_xhi, map_xlo, g, grid, st);
    case 128: return launch_bn<128>(map_w, map_xhi, map_xlo, g, grid, st);
    default: return cudaErrorInvalidValue;
    }
}

}  // namespace sp
