// Split-KV attention of the k appended rows over [cached ; new] keys
// (Sec. 3.3, Eq. 1-3), CUDA-core version for any head_dim in {32, 64, 128} and
// either cache dtype, plus the split merge shared by every attention kernel.
//
// Work unit: (split s, kv head g, sequence b).  The keys of sequence b are the
// concatenation [cache tokens 0..L_b-1 ; new keys 0..k-1]; unit s covers
// positions [s*split_tokens, (s+1)*split_tokens) of it.  Query row
// rr = hl*k + r (query head g*G + hl, soft row r) sees position t iff
// t <= L_b + r.  Each unit writes an unnormalised partial (O, running max m in
// log2 units, running sum l); the merge rescales partials by 2^(m_s - max m).
#include "sp_common.cuh"

namespace sp {

namespace {

constexpr int kTile = 32;       // tokens per smem tile
constexpr int kThreads = 128;

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Address of (token t < L, kv head g) in either cache layout; nullptr when the
// page-table entry is outside the pool (status bit set by the caller).
template <typename T>
__device__ __forceinline__ const T *cache_row(const KVDev &kv, const void *pool_or_null, int sid,
                                              int t, int g, int Hkv, int dh, bool is_v, int *bad) {
    if (kv.layout == SP_KV_CONTIGUOUS) {
        const T *base = (const T *)(is_v ? kv.v_seq[sid] : kv.k_seq[sid]);
        return base + ((size_t)t * Hkv + g) * dh;
    }
    const int P = kv.page_size;
    const int lp = t / P;
    if (lp >= kv.max_pages) {  // a length beyond the page-table row
        *bad = 1;
        return nullptr;
    }
    const int page = kv.page_table[(size_t)sid * kv.max_pages + lp];
    if (page < 0 || page >= kv.n_pages) {
        *bad = 1;
        return nullptr;
    }
    const T *pool = (const T *)pool_or_null;
    return pool + (((size_t)page * Hkv + g) * P + (t % P)) * dh;
}

template <typename TKV, int DH>
__global__ void __launch_bounds__(kThreads) attn_split_simt(AttnArgs a) {
    pdl_trigger();
    pdl_wait();
    extern __shared__ float smem[];
    const int s = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
    const int R = a.R, k = a.k;
    float *Qs = smem;                      // [R][DH]
    float *Ks = Qs + R * DH;               // [kTile][DH + 1]
    float *Vs = Ks + kTile * (DH + 1);     // [kTile][DH]
    float *S = Vs + kTile * DH;            // [R][kTile]
    float *Os = S + R * kTile;             // [R][DH]
    float *mrow = Os + R * DH;             // [R]
    float *lrow = mrow + R;                // [R]
    float *arow = lrow + R;                // [R]

    const SeqRef sq = resolve_seq(a.seq_ids, a.seq_lens, a.lens_by_batch, b, a.kv.n_seqs, a.max_seq_len,
                                  (threadIdx.x == 0 && s == 0 && g == 0) ? a.status : nullptr);
    const int L = sq.len;
    const int total = L + a.r0 + k;
    const int kns = a.kn_stride ? a.kn_stride : k;
    const int t_begin = s * a.split_tokens;
    if (t_begin >= total) return;  // the merge reads only units below ceil(total / split)
    const int t_end = min(total, t_begin + a.split_tokens);

    for (int idx = threadIdx.x; idx < R * DH; idx += kThreads) {
        const int rr = idx / DH, c = idx - rr * DH;
        const int hl = rr / k, r = rr - hl * k;
        const int h = g * a.G + hl;
        Qs[idx] = a.q[(((size_t)b * k + r) * a.Hq + h) * DH + c] * a.scale_log2;
        Os[idx] = 0.f;
    }
    for (int rr = threadIdx.x; rr < R; rr += kThreads) {
        mrow[rr] = -INFINITY;
        lrow[rr] = 0.f;
    }
    int bad = 0;
    __syncthreads();

    for (int t0 = t_begin; t0 < t_end; t0 += kTile) {
        for (int idx = threadIdx.x; idx < kTile * DH; idx += kThreads) {
            const int tt = idx / DH, c = idx - tt * DH;
            const int t = t0 + tt;
            float kv_k = 0.f, kv_v = 0.f;
            if (t < t_end) {
                if (t < L) {
                    const TKV *kr = cache_row<TKV>(a.kv, a.kv.k_pool, sq.sid, t, g, a.Hkv, DH,
                                                   false, &bad);
                    const TKV *vr = cache_row<TKV>(a.kv, a.kv.v_pool, sq.sid, t, g, a.Hkv, DH,
                                                   true, &bad);
                    if (kr) kv_k = to_f(kr[c]);
                    if (vr) kv_v = to_f(vr[c]);
                    if (c == 0 && a.gathered && a.kv.layout == SP_KV_PAGED &&
                        (t % a.kv.page_size == 0 || tt == 0) && t / a.kv.page_size < a.kv.max_pages)
                        a.gathered[(size_t)b * a.kv.max_pages + t / a.kv.page_size] =
                            a.kv.page_table[(size_t)sq.sid * a.kv.max_pages + t / a.kv.page_size];
                } else {
                    const int j = t - L;
                    const size_t o = (((size_t)b * kns + j) * a.Hkv + g) * DH + c;
                    kv_k = a.k_new[o];
                    kv_v = a.v_new[o];
                }
            }
            Ks[tt * (DH + 1) + c] = kv_k;
            Vs[tt * DH + c] = kv_v;
        }
        __syncthreads();
        for (int idx = threadIdx.x; idx < R * kTile; idx += kThreads) {
            const int rr = idx / kTile, tt = idx - rr * kTile;
            const int t = t0 + tt;
            const int r = rr % k;
            float sc = -INFINITY;
            const int lo = a.k_task ? (r / a.k_task) * a.k_task : 0;  // the task's first new row
            if (t < t_end && t <= L + a.r0 + r && (t < L || t >= L + lo)) {
                const float *qr = Qs + rr * DH;
                const float *kr = Ks + tt * (DH + 1);
                float acc = 0.f;
#pragma unroll 8
                for (int c = 0; c < DH; ++c) acc = fmaf(qr[c], kr[c], acc);
                sc = acc;
            }
            S[idx] = sc;
        }
        __syncthreads();
        const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
        for (int rr = w; rr < R; rr += kThreads / 32) {
            const float sc = S[rr * kTile + lane];
            const float m_old = mrow[rr];
            const float m_new = fmaxf(m_old, warp_max(sc));
            float p = 0.f, alpha = 1.f;
            if (m_new != -INFINITY) {
                p = (sc == -INFINITY) ? 0.f : exp2f(sc - m_new);
                alpha = (m_old == -INFINITY) ? 0.f : exp2f(m_old - m_new);
            }
            const float psum = warp_sum(p);
            S[rr * kTile + lane] = p;
            if (lane == 0) {
                lrow[rr] = lrow[rr] * alpha + psum;
                mrow[rr] = m_new;
                arow[rr] = alpha;
            }
        }
        __syncthreads();
        for (int idx = threadIdx.x; idx < R * DH; idx += kThreads) {
            const int rr = idx / DH, c = idx - rr * DH;
            const float *pr = S + rr * kTile;
            float acc = Os[idx] * arow[rr];
#pragma unroll 8
            for (int tt = 0; tt < kTile; ++tt) acc = fmaf(pr[tt], Vs[tt * DH + c], acc);
            Os[idx] = acc;
        }
        __syncthreads();
    }
    if (bad && a.status) atomicOr(a.status, SP_DEV_BAD_PAGE);

    const size_t unit = ((size_t)b * a.Hkv + g) * a.n_splits + s;
    float *po = a.part_o + unit * R * DH;
    for (int idx = threadIdx.x; idx < R * DH; idx += kThreads) po[idx] = Os[idx];
    float *pml = a.part_ml + unit * R * 2;
    for (int rr = threadIdx.x; rr < R; rr += kThreads) {
        pml[2 * rr] = mrow[rr];
        pml[2 * rr + 1] = lrow[rr];
    }
}

// Merge the partials of one query row: block (kv head g, sequence b, row rr),
// thread c = output column c (head_dim threads).  Each pass issues the loads
// of up to eight partials before combining them.
__global__ void attn_merge_kernel(AttnArgs a) {
    pdl_trigger();
    pdl_wait();
    const int g = blockIdx.x, b = blockIdx.y, rr = blockIdx.z;
    const int R = a.R, dh = a.dh, k = a.k;
    const SeqRef sq = resolve_seq(a.seq_ids, a.seq_lens, a.lens_by_batch, b, a.kv.n_seqs,
                                  a.max_seq_len, nullptr);
    const int n_valid = min(a.n_splits, ceil_div(sq.len + a.r0 + k, a.split_tokens)) * a.subs;
    const size_t unit0 = ((size_t)b * a.Hkv + g) * a.n_splits * a.subs;
    const int c = threadIdx.x;
    float mmax = -INFINITY;
    for (int s0 = 0; s0 < n_valid; s0 += 8) {
        float mv[8];
#pragma unroll
        for (int j = 0; j < 8; ++j)
            mv[j] = s0 + j < n_valid ? a.part_ml[((unit0 + s0 + j) * R + rr) * 2] : -INFINITY;
#pragma unroll
        for (int j = 0; j < 8; ++j) mmax = fmaxf(mmax, mv[j]);
    }
    float l = 0.f, o = 0.f;
    for (int s0 = 0; s0 < n_valid; s0 += 8) {
        float ms[8], ls[8], os[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const bool in = s0 + j < n_valid;
            const size_t u = unit0 + s0 + j;
            ms[j] = in ? a.part_ml[(u * R + rr) * 2] : -INFINITY;
            ls[j] = in ? a.part_ml[(u * R + rr) * 2 + 1] : 0.f;
            os[j] = in ? a.part_o[(u * R + rr) * dh + c] : 0.f;
        }
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            if (ms[j] == -INFINITY) continue;
            const float wgt = exp2f(ms[j] - mmax);
            l += ls[j] * wgt;
            o += os[j] * wgt;
        }
    }
    const int hl = rr / k, r = rr - hl * k;
    const int h = g * a.G + hl;
    act_store(a.out, (((size_t)b * k + r) * a.Hq + h) * dh + c, l > 0.f ? o / l : 0.f);
}

template <typename TKV, int DH>
cudaError_t launch_simt_t(const AttnArgs &a, cudaStream_t st) {
    const int R = a.R;
    const size_t smem =
        sizeof(float) * ((size_t)R * DH + kTile * (DH + 1) + kTile * DH + (size_t)R * kTile +
                         (size_t)R * DH + 3 * (size_t)R);
    if (smem > 227 * 1024) return cudaErrorInvalidConfiguration;
    cudaError_t e = cudaFuncSetAttribute(attn_split_simt<TKV, DH>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    dim3 grid(a.n_splits, a.Hkv, a.B);
    return launch_k(attn_split_simt<TKV, DH>, grid, dim3(kThreads), smem, st, a);
}

}  // namespace

void plan_attention(int B, int Hkv, int k, int max_seq_len, int forced_split, int n_sm,
                    int *split_tokens, int *n_splits) {
    const int total = max_seq_len + k;
    const int tiles = (total + 63) / 64;
    int chunk;
    if (forced_split > 0) {
        chunk = forced_split;
    } else {
        // Choose the number of splits s of the longest sequence that minimises
        // waves(s) * (tiles per unit + start-up), for one work unit per SM at a
        // time: waves = ceil(B * Hkv * s / n_sm), start-up ~ 6 tiles of work.
        // Splits stay <= 16384 tokens (one split's page ids fit in shared memory).
        const long long units = (long long)B * Hkv;
        const int s_min = (tiles + 255) / 256;
        long long best_cost = -1;
        int best_s = s_min;
        for (int s = s_min; s <= tiles && s <= 64; ++s) {
            const long long waves = (units * s + n_sm - 1) / n_sm;
            const long long cost = waves * ((tiles + s - 1) / s + 6);
            if (best_cost < 0 || cost < best_cost) {
                best_cost = cost;
                best_s = s;
            }
        }
        chunk = ((tiles + best_s - 1) / best_s) * 64;
    }
    *split_tokens = chunk;
    *n_splits = ceil_div(total, chunk);
}

size_t attention_workspace_bytes(int B, int Hkv, int R, int dh, int n_splits, int n_sm) {
    const size_t pairs = (size_t)B * Hkv;
    size_t parts = pairs * n_splits;
    const size_t tc_slots = (size_t)attn_tc_ctas(n_sm, Hkv) + pairs;
    if (tc_slots > parts) parts = tc_slots;
    const auto al = [](size_t x) { return (x + 255) & ~(size_t)255; };
    return al(pairs * sizeof(int)) + al(parts * R * dh * sizeof(float)) +
           al(parts * R * 2 * sizeof(float));
}

cudaError_t launch_attention_simt(const AttnArgs &a, cudaStream_t st) {
    if (a.kv_bf16) {
        if (a.dh == 32) return launch_simt_t<bf16, 32>(a, st);
        if (a.dh == 64) return launch_simt_t<bf16, 64>(a, st);
        if (a.dh == 128) return launch_simt_t<bf16, 128>(a, st);
    } else {
        if (a.dh == 32) return launch_simt_t<float, 32>(a, st);
        if (a.dh == 64) return launch_simt_t<float, 64>(a, st);
        if (a.dh == 128) return launch_simt_t<float, 128>(a, st);
    }
    return cudaErrorInvalidValue;
}

cudaError_t launch_attention_merge(const AttnArgs &a, cudaStream_t st) {
    dim3 grid(a.Hkv, a.B, a.R);
    return launch_k(attn_merge_kernel, grid, dim3(a.dh), 0, st, a);
}

}  // namespace sp
