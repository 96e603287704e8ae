// Internal declarations shared by the CUDA translation units of libsp.so.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/sp.h"

namespace sp {

typedef __nv_bfloat16 bf16;

__host__ __device__ inline int ceil_div(int a, int b) { return (a + b - 1) / b; }
__host__ __device__ inline long long ceil_div_ll(long long a, long long b) { return (a + b - 1) / b; }

__device__ __forceinline__ float to_f(float x) { return x; }
__device__ __forceinline__ float to_f(bf16 x) { return __bfloat162float(x); }
template <typename T> __device__ __forceinline__ T from_f(float x);
template <> __device__ __forceinline__ float from_f<float>(float x) { return x; }
template <> __device__ __forceinline__ bf16 from_f<bf16>(float x) { return __float2bfloat16_rn(x); }

// Programmatic dependent launch.  Every kernel of the path is launched with
// programmatic stream serialisation (launch_k), so its CTAs may start -- and do
// their independent set-up -- while the previous kernel on the stream drains.
// pdl_wait() returns once the previous kernel has completed and its writes are
// visible; every kernel calls it before touching data an earlier kernel
// writes, and before writing scratch an earlier kernel may still read.
// pdl_trigger() allows the next kernel to launch (it still waits in pdl_wait).
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename Kern, typename... Args>
inline cudaError_t launch_k(Kern kernel, dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                            Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = st ? 1 : 0;  // the legacy default stream keeps plain serialisation
    return cudaLaunchKernelEx(&cfg, kernel, args...);
}

// Where a producer writes an activation: fp32 (f32 != null), plain bf16
// (hi != null, lo == null) or the two-plane form hi = rn(v), lo = rn(v - hi)
// that the tensor-core projections consume.
struct ActOut {
    float *f32;
    bf16 *hi;
    bf16 *lo;
};
__device__ __forceinline__ void act_store(const ActOut &o, size_t idx, float v) {
    if (o.f32) {
        o.f32[idx] = v;
        return;
    }
    const bf16 h = __float2bfloat16_rn(v);
    o.hi[idx] = h;
    if (o.lo) o.lo[idx] = __float2bfloat16_rn(v - __bfloat162float(h));
}

// A projection result held as `n` fp32 partial sums `stride` elements apart
// (split-K); readers add them.
struct PartIn {
    const float *y;
    int n;
    size_t stride;
};
// Loads of up to eight partials are issued together before they are added
// (the adds would otherwise serialise one memory latency per partial).
__device__ __forceinline__ float part_get(const PartIn &p, size_t idx) {
    float s = 0.f;
    for (int i0 = 0; i0 < p.n; i0 += 8) {
        float v[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) v[j] = (i0 + j < p.n) ? p.y[(size_t)(i0 + j) * p.stride + idx] : 0.f;
#pragma unroll
        for (int j = 0; j < 8; ++j) s += v[j];
    }
    return s;
}
// Four consecutive values (idx and stride multiples of 4).
__device__ __forceinline__ float4 part_get4(const PartIn &p, size_t idx) {
    float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int i0 = 0; i0 < p.n; i0 += 4) {
        float4 v[4];
#pragma unroll
        for (int j = 0; j < 4; ++j)
            v[j] = (i0 + j < p.n) ? *(const float4 *)(p.y + (size_t)(i0 + j) * p.stride + idx)
                                  : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            s.x += v[j].x;
            s.y += v[j].y;
            s.z += v[j].z;
            s.w += v[j].w;
        }
    }
    return s;
}

// Vector helpers for 8 consecutive elements (16-byte aligned bf16, 32-byte fp32).
__device__ __forceinline__ void load8(const float *p, float (&v)[8]) {
    const float4 a = *(const float4 *)p, b = *(const float4 *)(p + 4);
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
    v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}
__device__ __forceinline__ void load8(const bf16 *p, float (&v)[8]) {
    const uint4 u = *(const uint4 *)p;
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        v[2 * i] = __uint_as_float(w[i] << 16);
        v[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
    }
}
__device__ __forceinline__ uint32_t pack2_bf16(float a, float b) {
    __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<uint32_t *>(&h);
}
// act_store of 4 consecutive values (idx multiple of 4)
__device__ __forceinline__ void act_store4(const ActOut &o, size_t idx, float4 v) {
    if (o.f32) {
        *(float4 *)(o.f32 + idx) = v;
        return;
    }
    const float x[4] = {v.x, v.y, v.z, v.w};
    float h[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) h[i] = __bfloat162float(__float2bfloat16_rn(x[i]));
    *(uint2 *)(o.hi + idx) = make_uint2(pack2_bf16(h[0], h[1]), pack2_bf16(h[2], h[3]));
    if (o.lo)
        *(uint2 *)(o.lo + idx) = make_uint2(pack2_bf16(x[0] - h[0], x[1] - h[1]),
                                            pack2_bf16(x[2] - h[2], x[3] - h[3]));
}

// Cache description as the kernels see it (same fields as sp_kv_cache).
struct KVDev {
    int layout;
    const void *const *k_seq;
    const void *const *v_seq;
    const void *k_pool;
    const void *v_pool;
    const int *page_table;
    int page_size;
    int n_pages;
    int max_pages;
    int n_seqs;
};

// Per-sequence bookkeeping shared by every kernel that reads ids/lengths:
// out-of-range ids or lengths set a status bit and are clamped so that no
// access leaves the caller's buffers.
struct SeqRef {
    int sid;   // cache sequence id (clamped to a valid id, or -1)
    int len;   // cached length L_b, clamped to [0, max_seq_len]
};

// Lengths are indexed by sequence id (lens_by_batch = 0) or by batch entry.
__device__ __forceinline__ SeqRef resolve_seq(const int *seq_ids, const int *seq_lens,
                                              int lens_by_batch, int b, int n_seqs,
                                              int max_seq_len, int *status) {
    SeqRef r;
    int sid = seq_ids ? seq_ids[b] : b;
    if (sid < 0 || sid >= n_seqs) {
        if (status) atomicOr(status, SP_DEV_BAD_SEQ_ID);
        r.sid = -1;
        r.len = 0;
        return r;
    }
    int L = seq_lens[lens_by_batch ? b : sid];
    if (L < 0 || L > max_seq_len) {
        if (status) atomicOr(status, SP_DEV_BAD_LENGTH);
        L = L < 0 ? 0 : max(max_seq_len, 0);  // a negative bound never yields a negative length
    }
    r.sid = sid;
    r.len = L;
    return r;
}

// ---------------------------------------------------------------------------
// attention step
// ---------------------------------------------------------------------------
struct AttnArgs {
    int B, Hq, Hkv, dh, k, G, R;  // R = G * k query rows per (sequence, kv head)
    int r0;                       // the pass's query row r is new row r0 + r (position
                                  // L + r0 + r) and sees new keys 0..r0 + r
    int kn_stride;                // rows per sequence of k_new / v_new (0 = k)
    int k_task;                   // rows per task (0 = k): query row r belongs to task
                                  // r / k_task and sees only that task's new rows
    int kv_bf16;                  // cache element type: 1 bf16, 0 fp32
    int split_tokens;             // tokens per work unit
    int n_splits;                 // work units per (sequence, kv head) in the grid
    int max_seq_len;
    const int *seq_ids;
    const int *seq_lens;
    int lens_by_batch;
    KVDev kv;
    const float *q;               // [B][k][Hq][dh], rotated
    const float *k_new;           // [B][kn_stride][Hkv][dh], rotated
    const float *v_new;           // [B][kn_stride][Hkv][dh]
    int subs;                     // partials per work unit (1)
    int tc_ctas;                  // tensor-core kernel: persistent CTAs (one per SM)
    int tc_min_tiles;             // tensor-core kernel: fewest 64-token tiles per CTA
    int tc_seg_cost;              // tensor-core kernel: cost of a segment boundary, in tiles,
                                  // that the cuts between shares balance
    int tc_q_plain;               // tensor-core kernel: 1 = queries as plain bf16 (one score
                                  // MMA per step), 0 = bf16 hi + lo (two)
    int tc_merge_kernel;          // tensor-core kernel: 1 = merge in a second kernel (small
                                  // batches), 0 = inside the attention kernel
    float *part_o;                // CUDA cores: [B][Hkv][n_splits][subs][R][dh]; tensor
                                  // cores: [tc_ctas + B Hkv][R][dh] (slot c + pair); unnormalised
    float *part_ml;               // same slots, [R][2] each (max in log2 units, sum)
    int *counters;                // [B][Hkv] finished segments, zero before the launch (tensor
                                  // cores: the last segment of a pair merges it)
    int *status;
    int *gathered;                // [B][max_pages] or NULL
    float scale_log2;             // log2(e) / sqrt(dh)
    ActOut out;                   // merge output [B][k][Hq][dh]
    const void *l2_next;          // tensor-core kernel: prefetched into L2 by the CTAs as
    size_t l2_next_bytes;         // they finish (the next projection's weights), or NULL
};

// Plan: tokens per split-KV work unit and number of units per sequence.
void plan_attention(int B, int Hkv, int k, int max_seq_len, int forced_split, int n_sm,
                    int *split_tokens, int *n_splits);
// Attention scratch: merge counters [B][Hkv] int, then partials (part_o,
// part_ml) sized for either kernel: B Hkv n_splits units (CUDA cores) or
// attn_tc_ctas(n_sm, Hkv) + B Hkv slots (tensor cores).
size_t attention_workspace_bytes(int B, int Hkv, int R, int dh, int n_splits, int n_sm);
// Default fewest tiles per CTA of the tensor-core kernel (64 tokens each).
constexpr int kAttnMinTiles = 8;
// Default cost of a segment boundary in the tensor-core kernel, in 64-token
// tiles (a pipeline drain, the epilogue and the next queries' load).
constexpr int kAttnSegCost = 12;
// The same for contiguous caches (cp.async tiles), measured on the 4B shape
// (B = 16, ~16 tiles per share): 28 gave the attention 40.5 us against 42.6 us
// at 12; on paged caches 20 was slower than 12 (27B long +1.3 us, 8B paged +6 us).
constexpr int kAttnSegCostContiguous = 28;
// Persistent CTAs of the tensor-core kernel: whole groups of Hkv (one CTA per
// kv head), as many groups as the SMs hold, at least one.
inline int attn_tc_ctas(int n_sm, int Hkv) { return (n_sm / Hkv > 1 ? n_sm / Hkv : 1) * Hkv; }
cudaError_t launch_attention_simt(const AttnArgs &a, cudaStream_t st);
// tcgen05 kernel: head_dim 128, bf16 cache, R <= 128, B <= 2048; paged caches
// need TMA maps of the K and V pools from encode_kv_pages_bf16.  The merge
// runs inside it (counters must be zero at launch) or, with tc_merge_kernel,
// in a second kernel launched behind it (two launches).
bool attention_tc_supported(const AttnArgs &a);
cudaError_t launch_attention_tc(const AttnArgs &a, const CUtensorMap *map_k,
                                const CUtensorMap *map_v, cudaStream_t st);
cudaError_t launch_attention_merge(const AttnArgs &a, cudaStream_t st);

// ---------------------------------------------------------------------------
// row-wise steps
// ---------------------------------------------------------------------------
// out[m] = RMSNorm(x[src(m)]) * gain, src(m) = m or m % row_mod (shared rows);
// x is bf16 (x_bf16) or fp32.
cudaError_t launch_rmsnorm_rows(int x_bf16, const void *x, int row_mod, const float *gain, float eps,
                                int M, int d, ActOut out, cudaStream_t st);

struct QkvRopeArgs {
    PartIn y;                // projections [rows][(Hq + 2 Hkv) dh]
    int shared;              // 1: row of m is m % k (shared soft prompt), 0: row m
    int B, k, Hq, Hkv, dh;
    int r0;                  // row m = b k + r is new row r0 + r, at position L_b + r0 + r
    int kn_stride;           // rows per sequence of k_new / v_new (0 = k)
    int k_task;              // rows per task (0 = k): the position is L_b + r0 + r % k_task
    const int *seq_ids, *seq_lens;
    int lens_by_batch;
    int n_seqs, max_seq_len;
    const float2 *rope_cs;   // [max_seq_len + k][dh/2] (cos, sin)
    float *q, *k_new, *v_new;
    int *status;
    int *zero_ints;          // optional: n_zero ints cleared for the next kernel
    int n_zero;
};
cudaError_t launch_qkv_rope(const QkvRopeArgs &a, cudaStream_t st);

// h1 = x + y ; n = RMSNorm(h1) * gain   (x: input rows, bf16 or fp32; row m
// reads x row m % row_mod (row_mod > 0) or m, and y row m / y_div)
cudaError_t launch_residual_norm(int x_bf16, PartIn y, const void *x, int row_mod,
                                 const float *gain, float eps, int M, int d, float *h1, ActOut n,
                                 cudaStream_t st, int y_div = 1);

// a[m][j] = silu(g) * u for gate/up columns laid out in blocks of `blk`
// (gate block i at columns 2*i*blk.., up block right after it)
cudaError_t launch_swiglu(PartIn y, int M, int f, int blk, ActOut a, cudaStream_t st);

// logits[b] = W_head pool_r(h1 + y) + bias, via per-chunk partial dot
// products in `scratch` (readout_scratch_bytes); one launch: the block that
// finishes a sequence's last chunk (counters[b], zero before the launch and
// cleared again by that block) adds the chunks up.
size_t readout_scratch_bytes(int B, int d, int C);
// Row r of sequence b of (h1 + y) sits at b sb + r sr (0 = the dense [B][k][d]
// strides k d and d).  With n_tasks > 1, "sequence" b is (sequence b / n_tasks,
// task b % n_tasks) and reads head [b % n_tasks] of head_w [n_tasks][C][d].
cudaError_t launch_readout(PartIn y, const float *h1, const float *head_w, const float *head_b,
                           int pool, int B, int k, int d, int C, float *scratch, float *logits,
                           int *counters, cudaStream_t st, size_t sb = 0, size_t sr = 0, int n_tasks = 1,
                           const float *g_final = nullptr, float eps = 0.f);

// ---------------------------------------------------------------------------
// projections
// ---------------------------------------------------------------------------
// out = x split into ActOut form (n elements); out = sum of the partials.
cudaError_t launch_to_act(const float *x, size_t n, ActOut out, cudaStream_t st);
cudaError_t launch_sum_partials(PartIn y, size_t n, float *out, cudaStream_t st);

// Y[M][N] (fp32) = X[M][K] (fp32) * W[N][K]^T (bf16 or fp32) on CUDA cores.
// w_blocked: W stored as [N / 128][K / 64][128][64] blocks (N % 128 == 0, K % 64 == 0).
cudaError_t launch_gemm_simt(int w_bf16, const void *X, const void *W, float *Y, int M, int N,
                             int K, cudaStream_t st, bool w_blocked = false);

// Replace the text sp_last_error() returns on this thread.
void set_error_text(const char *msg);

}  // namespace sp
