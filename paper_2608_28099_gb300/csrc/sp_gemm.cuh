// Projection dispatch for Y[M][N] = X[M][K] W[N][K]^T.
//  - tensor cores (tcgen05, sp_gemm_tc.cu): bf16 weights with N % 128 == 0 and
//    K % 64 == 0; activations as bf16 hi/lo planes; fp32 split-K partials.
//  - CUDA cores (sp_rowops.cu): anything else; fp32 activations; one partial.
#pragma once

#include <cuda.h>
#include <string.h>

#include "sp_common.cuh"

namespace sp {

// Rotation epilogue of the Q/K/V projection (rows [(Hq + 2 Hkv) 128][K], one
// 128-row weight tile per head): the CTA of tile t writes head t of its rows
// rotated at L_b + r0 + (k_task ? r % k_task : r) into q (query heads) or k_new,
// or copied into v_new, instead of a partial plane (Sec. 3.3; the same
// arithmetic as the separate rotation kernel).
struct RopeEpi {
    const float2 *rope_cs;   // [max_seq_len + k][64] (cos, sin)
    int Hq, Hkv, k, kn_stride, r0, k_task;
    const int *seq_ids, *seq_lens;
    int lens_by_batch, n_seqs, max_seq_len;
    float *q, *k_new, *v_new;
    int *status;
    int *zero_ints;          // cleared for the next kernel (the attention's merge counters)
    int n_zero;
};

struct TcPlan {
    int bn, m_tiles, n_tiles, n_kb;
    bool persistent;    // persistent stream-K kernel, else one CTA per (tile, K split)
    int kb_per_split;   // tile kernel: k-blocks per split
    int units_per_cta;  // persistent: (tile, k-block) units per CTA
    int grid;           // CTAs
    int splits;         // partial planes of Y
    int nt;             // tile kernel: weight tiles per CTA (1, or 2 sharing each activation block)
};

bool encode_kmajor_bf16(CUtensorMap *map, const void *base, int rows, int K, int box_rows);
// TMA map of a paged K or V pool [n_page_heads][page_size][128] bf16 whose box
// is one (page, head) block in the attention kernel's shared-memory tile layout.
bool encode_kv_pages_bf16(CUtensorMap *map, const void *pool, long long n_page_heads, int page_size);
// TMA map of rotated queries [rows][Hq][128] fp32 by (k rows x G heads) boxes.
bool encode_q_group_f32(CUtensorMap *map, const float *q, int rows, int Hq, int G, int k);
bool tc_supported(int N, int K);
// Rows per tile for M activation rows: 16..128, or 256 (plain bf16 only: the
// MMA's N side is then 256) for M >= 256.
int tc_bn_for(int M, bool lo = true);
// sched: 0 = automatic, 1 = tile kernel, 2 = persistent stream-K (when its
// partial planes fit).
TcPlan tc_plan(int M, int N, int K, int n_sm, size_t y_capacity_bytes, bool lo = true,
               int sched = 0);
// w_blocked: the weights are stored blocked (block_weights_layout) and map_w
// views them as [N K / 64][64] rows.
cudaError_t launch_gemm_tc(const CUtensorMap &map_w, const CUtensorMap &map_xhi,
                           const CUtensorMap &map_xlo, const TcPlan &p, int M, int N, int K,
                           float *y, int *status, cudaStream_t st, bool w_blocked = false,
                           bool lo = true, int inject_stall = 0, const ActOut *glu = nullptr,
                           const RopeEpi *rope = nullptr);

// Weights [N][K] (es bytes per element) re-laid out as contiguous 16 KB blocks
// [N / 128][K / 64][128][64]: one weight tile's k-block is one sequential read
// instead of 128 row pieces K * es bytes apart (+13-17 % weight bandwidth in the
// GEMV regime).  Needs N % 128 == 0 and K % 64 == 0.
inline void block_weights_layout(const char *src, char *dst, int N, int K, size_t es) {
    const int nkb = K / 64;
    for (int n = 0; n < N; ++n)
        for (int kb = 0; kb < nkb; ++kb) {
            const size_t blk = ((size_t)(n / 128) * nkb + kb) * 128 * 64;
            memcpy(dst + (blk + (size_t)(n % 128) * 64) * es, src + ((size_t)n * K + kb * 64) * es,
                   64 * es);
        }
}

constexpr int kNumBn = 5;  // tile widths 16, 32, 64, 128, 256
inline int bn_index(int bn) { return bn == 16 ? 0 : bn == 32 ? 1 : bn == 64 ? 2 : bn == 128 ? 3 : 4; }
inline int bn_value(int i) { return 16 << i; }

// A frozen weight matrix on the device, with its TMA map when tensor cores apply.
struct WeightMat {
    const void *ptr = nullptr;
    int N = 0, K = 0;
    bool tc = false;
    bool blocked = false;  // stored by block_weights_layout
    CUtensorMap map;
};

// An activation buffer holding up to rows_max rows of K values, either as fp32
// [rows][K] or as two bf16 planes hi [rows_max][K] then lo [rows_max][K].
struct ActBuf {
    void *ptr = nullptr;
    int K = 0, rows_max = 0;
    bool maps = false;
    CUtensorMap hi[kNumBn], lo[kNumBn];
    // tc: the consumer is a tensor-core projection (bf16 planes), else fp32;
    // lo: with the lo plane (hi + lo ~ 16 mantissa bits), else plain bf16
    ActOut out(bool tc, bool lo = true) const {
        ActOut o;
        if (tc) {
            o.f32 = nullptr;
            o.hi = (bf16 *)ptr;
            o.lo = lo ? (bf16 *)ptr + (size_t)rows_max * K : nullptr;
        } else {
            o.f32 = (float *)ptr;
            o.hi = o.lo = nullptr;
        }
        return o;
    }
};

inline bool init_weight(WeightMat &w, const void *ptr, int N, int K, int w_bf16,
                        bool blocked = false) {
    w.ptr = ptr;
    w.N = N;
    w.K = K;
    w.blocked = blocked;
    w.tc = w_bf16 && tc_supported(N, K) &&
           (blocked ? encode_kmajor_bf16(&w.map, ptr, (int)((long long)N * K / 64), 64, 128)
                    : encode_kmajor_bf16(&w.map, ptr, N, K, 128));
    return true;
}

inline void init_act(ActBuf &a, void *ptr, int rows_max, int K, bool want_maps) {
    a.ptr = ptr;
    a.K = K;
    a.rows_max = rows_max;
    a.maps = false;
    if (!want_maps || K % 64) return;
    bool ok = true;
    const bf16 *hi = (const bf16 *)ptr, *lo = hi + (size_t)rows_max * K;
    for (int i = 0; i < kNumBn; ++i) {
        if (bn_value(i) > 128 && rows_max < bn_value(i)) break;  // never planned (M <= rows_max)
        ok = ok && encode_kmajor_bf16(&a.hi[i], hi, rows_max, K, bn_value(i));
        ok = ok && encode_kmajor_bf16(&a.lo[i], lo, rows_max, K, bn_value(i));
    }
    a.maps = ok;
}

struct GemmPlanner {
    int n_sm = 148;
    size_t y_capacity = 0;  // bytes available for [splits][M][N] partials
    int sched = 0;          // SP_OPT_GEMM_SCHEDULE
    void init(int sms, size_t cap) {
        n_sm = sms;
        y_capacity = cap;
    }
    // Does this projection run on tensor cores under path option `path`
    // (0 automatic, 1 CUDA cores, 2 tensor cores where supported)?
    bool use_tc(const WeightMat &w, const ActBuf &x, int path) const {
        return path != 1 && w.tc && x.maps;
    }
    // Would the gate/up projection ([gate block; up block] per 128-row tile)
    // run with the SwiGLU epilogue (one CTA per tile, no K split)?
    bool glu_fusable(const WeightMat &w, const ActBuf &x, int path, int M, bool lo) const {
        if (!use_tc(w, x, path)) return false;
        const TcPlan p = tc_plan(M, w.N, w.K, n_sm, y_capacity, lo, sched);
        return !p.persistent && p.splits == 1 && p.bn >= 32;
    }
    // Would the Q/K/V projection run with the rotation epilogue (one CTA per
    // weight tile = head, no K split)?
    bool rope_fusable(const WeightMat &w, const ActBuf &x, int path, int M, bool lo) const {
        if (!use_tc(w, x, path)) return false;
        const TcPlan p = tc_plan(M, w.N, w.K, n_sm, y_capacity, lo, sched);
        return !p.persistent && p.splits == 1 && p.nt == 1 && p.bn >= 32;
    }
    // Enqueue the projection; *nsplit receives the number of partials in y.
    // glu: write silu(gate) * up there instead of partials (glu_fusable);
    // rope: the rotation epilogue (rope_fusable).
    sp_status run(int w_bf16, int path, const ActBuf &x, const WeightMat &w, float *y, int M,
                  int *status, cudaStream_t st, int *launches, int *nsplit, bool lo = true,
                  int inject_stall = 0, const ActOut *glu = nullptr,
                  const RopeEpi *rope = nullptr) const {
        cudaError_t e;
        if (use_tc(w, x, path)) {
            const TcPlan p = tc_plan(M, w.N, w.K, n_sm, y_capacity, lo, sched);
            const int bi = bn_index(p.bn);
            e = launch_gemm_tc(w.map, x.hi[bi], x.lo[bi], p, M, w.N, w.K, y, status, st, w.blocked, lo,
                               inject_stall, glu, rope);
            *nsplit = p.splits;
        } else {
            e = launch_gemm_simt(w_bf16, x.ptr, w.ptr, y, M, w.N, w.K, st, w.blocked);
            *nsplit = 1;
        }
        if (e != cudaSuccess) return SP_ERR_CUDA;
        ++*launches;
        return SP_OK;
    }
};

}  // namespace sp
