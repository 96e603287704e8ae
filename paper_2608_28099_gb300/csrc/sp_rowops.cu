// Row-wise steps of the decoder layer (Sec. 3.1) and the CUDA-core projection:
// RMSNorm, rotary embedding of the new queries/keys (positions L_b..L_b+k-1,
// Sec. 3.3), residual + post-norm, SwiGLU, pooling + linear readout (Sec. 3.2).
#include "sp_common.cuh"

namespace sp {

namespace {

constexpr int kRowThreads = 256;
constexpr int kWideThreads = 1024;

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Block-wide sum (any multiple of 32 threads up to 1024).
__device__ __forceinline__ float block_sum(float v, float *red) {
    v = warp_sum(v);
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
    __syncthreads();
    if (l == 0) red[w] = v;
    __syncthreads();
    float t = (l < (int)(blockDim.x >> 5)) ? red[l] : 0.f;
    return warp_sum(t);
}

// RMSNorm for rows wider than the register-resident kernel below takes (d >
// 8192): one block per row, d % 8 == 0, 8-element vector loads, four chunks in
// flight per thread, two passes over the row.
template <typename T>
__global__ void __launch_bounds__(256) rmsnorm_rows_loop_kernel(const T *__restrict__ x, int row_mod,
                                                           const float *__restrict__ gain, float eps,
                                                           int d, ActOut out) {
    pdl_trigger();
    pdl_wait();
    __shared__ float red[32];
    const int m = blockIdx.x;
    const T *xr = x + (size_t)(row_mod ? m % row_mod : m) * d;
    const int nch = d >> 3;
    float ss = 0.f;
#pragma unroll 4
    for (int c = threadIdx.x; c < nch; c += blockDim.x) {
        float v[8];
        load8(xr + c * 8, v);
#pragma unroll
        for (int e = 0; e < 8; ++e) ss += v[e] * v[e];
    }
    ss = block_sum(ss, red);
    const float inv = rsqrtf(ss / (float)d + eps);
#pragma unroll 4
    for (int c = threadIdx.x; c < nch; c += blockDim.x) {
        float v[8], gv[8];
        load8(xr + c * 8, v);
        load8(gain + c * 8, gv);
        const size_t o = (size_t)m * d + c * 8;
        act_store4(out, o, make_float4(v[0] * inv * gv[0], v[1] * inv * gv[1], v[2] * inv * gv[2],
                                       v[3] * inv * gv[3]));
        act_store4(out, o + 4, make_float4(v[4] * inv * gv[4], v[5] * inv * gv[5],
                                           v[6] * inv * gv[6], v[7] * inv * gv[7]));
    }
}

// One block per row m = b k + r: the row's position L_b + r0 + r is resolved
// once (from the caller's ids and lengths, before the dependency wait), then
// each thread rotates four pairs (i, i + dh/2) of a query or key head at a time
// (16-byte loads of the partial sums and of the (cos, sin) table) or copies
// four values.  With few rows the block has 1024 threads, so that a row's items
// take one pass.
template <int TPB>
__global__ void __launch_bounds__(TPB) qkv_rope_kernel(QkvRopeArgs a) {
    pdl_trigger();
    __shared__ int s_pos;
    const int m = blockIdx.x;
    const int b = m / a.k, r = m % a.k;
    if (threadIdx.x == 0) {
        const SeqRef s = resolve_seq(a.seq_ids, a.seq_lens, a.lens_by_batch, b, a.n_seqs,
                                     a.max_seq_len, a.status);
        s_pos = s.len + a.r0 + (a.k_task ? r % a.k_task : r);
    }
    pdl_wait();
    if (a.zero_ints && m == 0)
        for (int t = threadIdx.x; t < a.n_zero; t += blockDim.x) a.zero_ints[t] = 0;
    __syncthreads();
    const int dh = a.dh, half = dh >> 1, q4 = half >> 2;
    const int nqkv = (a.Hq + 2 * a.Hkv) * dh;
    const size_t row = (size_t)(a.shared ? r : m) * nqkv;
    const int kns = a.kn_stride ? a.kn_stride : a.k;
    const size_t mn = (size_t)b * kns + a.r0 + r;  // row of k_new / v_new
    const float2 *cs = a.rope_cs + (size_t)s_pos * half;
    const int nrot = (a.Hq + a.Hkv) * q4, nval = a.Hkv * dh / 4, total = nrot + nval;
    constexpr int U = 1;  // items per pass (two per pass measured slower with many rows)
    for (int base = threadIdx.x; base < total; base += U * TPB) {
        float4 x0[U], x1[U], c01[U], c23[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int it = base + u * TPB;
            if (it < nrot) {
                const int h = it / q4, i = (it - h * q4) * 4;
                x0[u] = part_get4(a.y, row + (size_t)h * dh + i);
                x1[u] = part_get4(a.y, row + (size_t)h * dh + i + half);
                c01[u] = *(const float4 *)(cs + i);
                c23[u] = *(const float4 *)(cs + i + 2);
            } else if (it < total) {
                x0[u] = part_get4(a.y, row + (size_t)(a.Hq + a.Hkv) * dh + (it - nrot) * 4);
            }
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int it = base + u * TPB;
            if (it < nrot) {
                const int h = it / q4, i = (it - h * q4) * 4;
                const float c[4] = {c01[u].x, c01[u].z, c23[u].x, c23[u].z};
                const float sn[4] = {c01[u].y, c01[u].w, c23[u].y, c23[u].w};
                const float a0[4] = {x0[u].x, x0[u].y, x0[u].z, x0[u].w};
                const float a1[4] = {x1[u].x, x1[u].y, x1[u].z, x1[u].w};
                float o0[4], o1[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    o0[e] = a0[e] * c[e] - a1[e] * sn[e];
                    o1[e] = a1[e] * c[e] + a0[e] * sn[e];
                }
                float *dst = h < a.Hq ? a.q + ((size_t)m * a.Hq + h) * dh
                                      : a.k_new + (mn * a.Hkv + (h - a.Hq)) * dh;
                *(float4 *)(dst + i) = make_float4(o0[0], o0[1], o0[2], o0[3]);
                *(float4 *)(dst + i + half) = make_float4(o1[0], o1[1], o1[2], o1[3]);
            } else if (it < total) {
                *(float4 *)(a.v_new + mn * a.Hkv * dh + (it - nrot) * 4) = x0[u];
            }
        }
    }
}

// The same with 256 threads and one item per loop step (many rows).
__global__ void __launch_bounds__(256) qkv_rope_rows_kernel(QkvRopeArgs a) {
    pdl_trigger();
    __shared__ int s_pos;
    const int m = blockIdx.x;
    const int b = m / a.k, r = m % a.k;
    if (threadIdx.x == 0) {
        const SeqRef s = resolve_seq(a.seq_ids, a.seq_lens, a.lens_by_batch, b, a.n_seqs,
                                     a.max_seq_len, a.status);
        s_pos = s.len + a.r0 + (a.k_task ? r % a.k_task : r);
    }
    pdl_wait();
    if (a.zero_ints && m == 0)
        for (int t = threadIdx.x; t < a.n_zero; t += blockDim.x) a.zero_ints[t] = 0;
    __syncthreads();
    const int dh = a.dh, half = dh >> 1, q4 = half >> 2;
    const int nqkv = (a.Hq + 2 * a.Hkv) * dh;
    const size_t row = (size_t)(a.shared ? r : m) * nqkv;
    const int kns = a.kn_stride ? a.kn_stride : a.k;
    const size_t mn = (size_t)b * kns + a.r0 + r;  // row of k_new / v_new
    const float2 *cs = a.rope_cs + (size_t)s_pos * half;
    const int nrot = (a.Hq + a.Hkv) * q4, nval = a.Hkv * dh / 4;
    for (int it = threadIdx.x; it < nrot + nval; it += blockDim.x) {
        if (it < nrot) {
            const int h = it / q4, i = (it - h * q4) * 4;
            const float4 x0 = part_get4(a.y, row + (size_t)h * dh + i);
            const float4 x1 = part_get4(a.y, row + (size_t)h * dh + i + half);
            const float4 c01 = *(const float4 *)(cs + i), c23 = *(const float4 *)(cs + i + 2);
            const float c[4] = {c01.x, c01.z, c23.x, c23.z}, sn[4] = {c01.y, c01.w, c23.y, c23.w};
            const float a0[4] = {x0.x, x0.y, x0.z, x0.w}, a1[4] = {x1.x, x1.y, x1.z, x1.w};
            float o0[4], o1[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                o0[e] = a0[e] * c[e] - a1[e] * sn[e];
                o1[e] = a1[e] * c[e] + a0[e] * sn[e];
            }
            float *dst = h < a.Hq ? a.q + ((size_t)m * a.Hq + h) * dh
                                  : a.k_new + (mn * a.Hkv + (h - a.Hq)) * dh;
            *(float4 *)(dst + i) = make_float4(o0[0], o0[1], o0[2], o0[3]);
            *(float4 *)(dst + i + half) = make_float4(o1[0], o1[1], o1[2], o1[3]);
        } else {
            const int j = (it - nrot) * 4;
            *(float4 *)(a.v_new + mn * a.Hkv * dh + j) =
                part_get4(a.y, row + (size_t)(a.Hq + a.Hkv) * dh + j);
        }
    }
}

// h1 = x + y, n = RMSNorm(h1) for d > 8192: one block per row, 4-element
// vectors, h1 re-read for the second pass.  Row m reads x row (row_mod ? m %
// row_mod : m) and y row m / y_div (as the register-resident kernel below).
template <typename TX>
__global__ void __launch_bounds__(1024) residual_norm_loop_kernel(PartIn y, int y_div,
                                                             const TX *__restrict__ x,
                                                             int row_mod,
                                                             const float *__restrict__ gain,
                                                             float eps, int d,
                                                             float *__restrict__ h1, ActOut n) {
    pdl_trigger();
    pdl_wait();
    __shared__ float red[32];
    const int m = blockIdx.x;
    const TX *xr = x + (size_t)(row_mod ? m % row_mod : m) * d;
    float *hr = h1 + (size_t)m * d;
    const int nch = d >> 2;
    float ss = 0.f;
#pragma unroll 2
    for (int c = threadIdx.x; c < nch; c += blockDim.x) {
        const float4 yv = part_get4(y, (size_t)(m / y_div) * d + c * 4);
        float4 v = make_float4(to_f(xr[c * 4]) + yv.x, to_f(xr[c * 4 + 1]) + yv.y,
                               to_f(xr[c * 4 + 2]) + yv.z, to_f(xr[c * 4 + 3]) + yv.w);
        *(float4 *)(hr + c * 4) = v;
        ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
    }
    ss = block_sum(ss, red);
    const float inv = rsqrtf(ss / (float)d + eps);
    __syncthreads();  // h1 row written by this block is re-read below
#pragma unroll 2
    for (int c = threadIdx.x; c < nch; c += blockDim.x) {
        const float4 v = *(const float4 *)(hr + c * 4);
        const float4 gv = *(const float4 *)(gain + c * 4);
        act_store4(n, (size_t)m * d + c * 4,
                   make_float4(v.x * inv * gv.x, v.y * inv * gv.y, v.z * inv * gv.z, v.w * inv * gv.w));
    }
}

// Register-resident norms for d <= 8192: one block of kNormThreads per row; each
// thread keeps its chunks in registers between the sum of squares and the
// output (no second pass over the row), with every load of the row issued
// before the first add.
constexpr int kNormThreads = 256;
constexpr int kNormMaxD = 8192;

int sm_count_cached() {
    static int n = 0;
    if (!n) {
        int dev = 0;
        cudaGetDevice(&dev);
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 148;
    }
    return n;
}

__device__ __forceinline__ float4 load4(const float *p) { return *(const float4 *)p; }
__device__ __forceinline__ float4 load4(const bf16 *p) {
    const uint2 u = *(const uint2 *)p;
    return make_float4(__uint_as_float(u.x << 16), __uint_as_float(u.x & 0xffff0000u),
                       __uint_as_float(u.y << 16), __uint_as_float(u.y & 0xffff0000u));
}

template <int TPB>
__device__ __forceinline__ float norm_block_sum(float v, float *red) {
    v = warp_sum(v);
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
    if (l == 0) red[w] = v;
    __syncthreads();
    float t = l < TPB / 32 ? red[l] : 0.f;
    return warp_sum(t);
}

template <typename T, int V, int TPB>  // V: 4-element chunks per thread, d <= 4 V TPB
__global__ void __launch_bounds__(TPB) rmsnorm_rows_kernel(const T *__restrict__ x, int row_mod,
                                                                    const float *__restrict__ gain,
                                                                    float eps, int d, ActOut out) {
    pdl_trigger();
    __shared__ float red[TPB / 32];
    const int m = blockIdx.x, nch = d >> 2;
    float4 gv[V];
#pragma unroll
    for (int i = 0; i < V; ++i) {  // constant: before the dependency wait
        const int c = threadIdx.x + i * TPB;
        gv[i] = c < nch ? *(const float4 *)(gain + c * 4) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
    pdl_wait();
    const T *xr = x + (size_t)(row_mod ? m % row_mod : m) * d;
    float4 v[V];
    float ss = 0.f;
#pragma unroll
    for (int i = 0; i < V; ++i) {
        const int c = threadIdx.x + i * TPB;
        v[i] = c < nch ? load4(xr + c * 4) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int i = 0; i < V; ++i) ss += v[i].x * v[i].x + v[i].y * v[i].y + v[i].z * v[i].z + v[i].w * v[i].w;
    ss = norm_block_sum<TPB>(ss, red);
    const float inv = rsqrtf(ss / (float)d + eps);
#pragma unroll
    for (int i = 0; i < V; ++i) {
        const int c = threadIdx.x + i * TPB;
        if (c < nch)
            act_store4(out, (size_t)m * d + c * 4,
                       make_float4(v[i].x * inv * gv[i].x, v[i].y * inv * gv[i].y, v[i].z * inv * gv[i].z,
                                   v[i].w * inv * gv[i].w));
    }
}

// h1 = x + y, n = RMSNorm(h1): as above, h1 kept in registers.
template <typename TX, int V, int TPB>
__global__ void __launch_bounds__(TPB) residual_norm_kernel(PartIn y, int y_div,
                                                                     const TX *__restrict__ x, int row_mod,
                                                                     const float *__restrict__ gain,
                                                                     float eps, int d,
                                                                     float *__restrict__ h1, ActOut n) {
    pdl_trigger();
    __shared__ float red[TPB / 32];
    const int m = blockIdx.x, nch = d >> 2;
    float4 gv[V];
#pragma unroll
    for (int i = 0; i < V; ++i) {
        const int c = threadIdx.x + i * TPB;
        gv[i] = c < nch ? *(const float4 *)(gain + c * 4) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
    pdl_wait();
    const TX *xr = x + (size_t)(row_mod ? m % row_mod : m) * d;
    const size_t yrow = (size_t)(m / y_div) * d;
    float4 v[V];
#pragma unroll
    for (int i = 0; i < V; ++i) {
        const int c = threadIdx.x + i * TPB;
        if (c < nch) {
            const float4 yv = part_get4(y, yrow + c * 4);
            const float4 xv = load4(xr + c * 4);
            v[i] = make_float4(xv.x + yv.x, xv.y + yv.y, xv.z + yv.z, xv.w + yv.w);
        } else {
            v[i] = make_float4(0.f, 0.f, 0.f, 0.f);
        }
    }
    float ss = 0.f;
    float *hr = h1 + (size_t)m * d;
#pragma unroll
    for (int i = 0; i < V; ++i) {
        const int c = threadIdx.x + i * TPB;
        if (c < nch) *(float4 *)(hr + c * 4) = v[i];
        ss += v[i].x * v[i].x + v[i].y * v[i].y + v[i].z * v[i].z + v[i].w * v[i].w;
    }
    ss = norm_block_sum<TPB>(ss, red);
    const float inv = rsqrtf(ss / (float)d + eps);
#pragma unroll
    for (int i = 0; i < V; ++i) {
        const int c = threadIdx.x + i * TPB;
        if (c < nch)
            act_store4(n, (size_t)m * d + c * 4,
                       make_float4(v[i].x * inv * gv[i].x, v[i].y * inv * gv[i].y, v[i].z * inv * gv[i].z,
                                   v[i].w * inv * gv[i].w));
    }
}

// a = silu(g) * u over 4-element vectors (f and blk multiples of 4).
__global__ void swiglu_kernel(PartIn y, int M, int f, int blk, ActOut a) {
    pdl_trigger();
    pdl_wait();
    const long long total4 = (long long)M * f / 4;
    for (long long i4 = blockIdx.x * (long long)blockDim.x + threadIdx.x; i4 < total4;
         i4 += (long long)gridDim.x * blockDim.x) {
        const long long idx = i4 * 4;
        const int m = (int)(idx / f), j = (int)(idx - (long long)m * f);
        const int blkid = j / blk, jj = j - blkid * blk;
        const size_t row = (size_t)m * 2 * f;
        const float4 g = part_get4(y, row + 2 * blkid * blk + jj);
        const float4 u = part_get4(y, row + 2 * blkid * blk + blk + jj);
        const float gx[4] = {g.x, g.y, g.z, g.w}, ux[4] = {u.x, u.y, u.z, u.w};
        float r[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) r[e] = __fdividef(gx[e], 1.f + __expf(-gx[e])) * ux[e];
        act_store4(a, (size_t)idx, make_float4(r[0], r[1], r[2], r[3]));
    }
}

// Pooling and the linear head, column-parallel: block (chunk, b) pools 256
// hidden columns of sequence b (h2 = h1 + y summed over the k rows by four row
// groups, four columns per thread with 16-byte loads, then mean or last) and
// writes its partial dot products with every head row to part[b][chunk][C];
// four classes are reduced at a time (one per row group).
constexpr int kReadoutCols = 256;
constexpr int kReadoutGroups = 4;  // row groups of a block (threads = 64 x 4)

__device__ __forceinline__ float4 f4_add(float4 a, float4 b) {
    return make_float4(a.x + b.x, a.y + b.y, a.z + b.z, a.w + b.w);
}

__global__ void __launch_bounds__(64 * kReadoutGroups, 2)
readout_partial_kernel(PartIn y, const float *__restrict__ h1, const float *__restrict__ head_w,
                       int pool, int k, int d, int C, float *__restrict__ part, size_t sb, size_t sr,
                       int n_tasks, const float *__restrict__ g_final, float *__restrict__ part_ss,
                       int *__restrict__ counters, const float *__restrict__ head_b,
                       float *__restrict__ logits, float eps) {
    pdl_trigger();
    __shared__ float4 acc_s[kReadoutGroups][64];
    __shared__ int is_last;
    __shared__ float pooled[kReadoutCols];
    __shared__ float red[4][8];
    const int chunk = blockIdx.x, b = blockIdx.y;
    const int c = threadIdx.x & 63, rg = threadIdx.x >> 6;
    const int col = chunk * kReadoutCols + 4 * c;  // d % 4 == 0: a group is all in or all out
    const bool in_d = col < d;
    const size_t base = (size_t)b * sb;
    head_w += (size_t)(b % n_tasks) * C * d;  // this task's head
    // the head is a constant of the handle, not an output of the previous
    // kernel: the first classes' weights are fetched before the wait
    const float4 hw0 = (rg < C && in_d) ? *(const float4 *)(head_w + (size_t)rg * d + col)
                                        : make_float4(0.f, 0.f, 0.f, 0.f);
    pdl_wait();
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    if (in_d) {
        // rows rg, rg + G, ... (G row groups) four at a time (all rows when
        // pooling the last one is a single row), the loads of their h1 values
        // and of up to four partials each issued together
        const int r_first = pool == SP_POOL_LAST ? k - 1 : rg;
        const int r_step = pool == SP_POOL_LAST ? k : kReadoutGroups;
        if (pool != SP_POOL_LAST || rg == 0) {
            for (int r0 = r_first; r0 < k; r0 += 4 * r_step) {
                size_t o[4];
                bool in[4];
                float4 v[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int r = r0 + u * r_step;
                    in[u] = r < k;
                    o[u] = base + (size_t)(in[u] ? r : r0) * sr + col;
                    v[u] = in[u] ? *(const float4 *)(h1 + o[u]) : make_float4(0.f, 0.f, 0.f, 0.f);
                }
                for (int i0 = 0; i0 < y.n; i0 += 4) {  // up to four planes per round
                    float4 pv[4][4];
#pragma unroll
                    for (int u = 0; u < 4; ++u)
#pragma unroll
                        for (int jj = 0; jj < 4; ++jj)
                            pv[u][jj] = (in[u] && i0 + jj < y.n)
                                            ? *(const float4 *)(y.y + (size_t)(i0 + jj) * y.stride + o[u])
                                            : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                    for (int u = 0; u < 4; ++u)
#pragma unroll
                        for (int jj = 0; jj < 4; ++jj) v[u] = f4_add(v[u], pv[u][jj]);
                }
                acc = f4_add(acc, f4_add(f4_add(v[0], v[1]), f4_add(v[2], v[3])));
            }
        }
    }
    acc_s[rg][c] = acc;
    __syncthreads();
    if (threadIdx.x < 64) {
        float4 sum = acc_s[0][c];
#pragma unroll
        for (int q = 1; q < kReadoutGroups; ++q) sum = f4_add(sum, acc_s[q][c]);
        const float dv = pool == SP_POOL_LAST ? 1.f : (float)k;
        const float p[4] = {sum.x / dv, sum.y / dv, sum.z / dv, sum.w / dv};
        if (g_final) {
            // LM-head readout: the chunk's share of the pooled row's square sum,
            // and the pooled values times the final-norm gain (the 1/rms factor
            // is applied to the finished dot products)
            float sq = in_d ? (p[0] * p[0] + p[1] * p[1]) + (p[2] * p[2] + p[3] * p[3]) : 0.f;
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
            if ((threadIdx.x & 31) == 0) red[3][4 + (threadIdx.x >> 5)] = sq;
#pragma unroll
            for (int e = 0; e < 4; ++e) pooled[4 * c + e] = in_d ? p[e] * g_final[col + e] : 0.f;
        } else {
#pragma unroll
            for (int e = 0; e < 4; ++e) pooled[4 * c + e] = p[e];
        }
    }
    __syncthreads();
    if (g_final && threadIdx.x == 0)
        part_ss[(size_t)b * gridDim.x + chunk] = red[3][4] + red[3][5];
    // row group rg takes class c0 + rg; its two warps hold the chunk's 256 columns
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int c0 = 0; c0 < C; c0 += kReadoutGroups) {
        const int cls = c0 + rg;
        const bool use = cls < C && in_d;
        const float4 hw = c0 == 0 ? hw0
                                  : (use ? *(const float4 *)(head_w + (size_t)cls * d + col)
                                         : make_float4(0.f, 0.f, 0.f, 0.f));
        float v = use ? (hw.x * pooled[4 * c] + hw.y * pooled[4 * c + 1]) +
                            (hw.z * pooled[4 * c + 2] + hw.w * pooled[4 * c + 3])
                      : 0.f;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
        if (lane == 0) red[w >> 1][w & 1] = v;
        __syncthreads();
        if (threadIdx.x < kReadoutGroups && c0 + (int)threadIdx.x < C)
            part[((size_t)b * gridDim.x + chunk) * C + c0 + threadIdx.x] =
                red[threadIdx.x][0] + red[threadIdx.x][1];
        __syncthreads();
    }
    // the block that finishes sequence b's last chunk adds the chunks' dot
    // products in chunk order (the bits do not depend on which block is last),
    // applies the LM-head 1/rms and the bias, and clears the counter
    __threadfence();  // this block's partials are visible before it is counted
    __syncthreads();
    if (threadIdx.x == 0) {
        const int before = atomicAdd(counters + b, 1);
        is_last = before == (int)gridDim.x - 1;
        if (is_last) counters[b] = 0;
    }
    __syncthreads();
    if (!is_last) return;
    __threadfence();  // the other blocks' partials are read after their count
    const int n_chunks = gridDim.x;
    float inv = 1.f;  // 1 / rms of the pooled row (LM-head readout)
    if (g_final) {
        float ss = 0.f;
        for (int j = 0; j < n_chunks; ++j) ss += __ldcg(part_ss + (size_t)b * n_chunks + j);
        inv = rsqrtf(ss / (float)d + eps);
    }
    const float *hb = head_b ? head_b + (size_t)(b % n_tasks) * C : nullptr;
    for (int cl = threadIdx.x; cl < C; cl += blockDim.x) {
        float acc = 0.f;
        for (int j = 0; j < n_chunks; ++j) acc += __ldcg(part + ((size_t)b * n_chunks + j) * C + cl);
        logits[(size_t)b * C + cl] = acc * inv + (hb ? hb[cl] : 0.f);
    }
}

__global__ void to_act_kernel(const float *__restrict__ x, size_t n, ActOut out) {
    pdl_trigger();
    pdl_wait();
    for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n;
         i += (size_t)gridDim.x * blockDim.x)
        act_store(out, i, x[i]);
}

__global__ void sum_partials_kernel(PartIn y, size_t n, float *__restrict__ out) {
    pdl_trigger();
    pdl_wait();
    for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n;
         i += (size_t)gridDim.x * blockDim.x)
        out[i] = part_get(y, i);
}

// CUDA-core tiled GEMM: Y[M][N] = X[M][K] W[N][K]^T, fp32 accumulation.
// 64x64 output tile, 32-deep k slices, 256 threads, 4x4 outputs per thread.
template <typename T>
__global__ void __launch_bounds__(256) gemm_simt_kernel(const float *__restrict__ X,
                                                        const T *__restrict__ W,
                                                        float *__restrict__ Y, int M, int N,
                                                        int K, int w_blocked) {
    pdl_trigger();
    pdl_wait();
    constexpr int BM = 64, BN = 64, BK = 32;
    __shared__ float Xs[BK][BM + 4];
    __shared__ float Ws[BK][BN + 4];
    const int tid = threadIdx.x;
    const int m0 = blockIdx.y * BM, n0 = blockIdx.x * BN;
    const int ty = tid >> 4, tx = tid & 15;
    float acc[4][4] = {};
    for (int k0 = 0; k0 < K; k0 += BK) {
        for (int idx = tid; idx < BM * BK; idx += 256) {
            const int row = idx / BK, kk = idx - row * BK;
            const int gm = m0 + row, gk = k0 + kk;
            Xs[kk][row] = (gm < M && gk < K) ? X[(size_t)gm * K + gk] : 0.f;
            const int gn = n0 + row;
            const size_t wi = w_blocked ? (((size_t)(gn >> 7) * (K >> 6) + (gk >> 6)) * 128 + (gn & 127)) * 64 +
                                              (gk & 63)
                                        : (size_t)gn * K + gk;
            Ws[kk][row] = (gn < N && gk < K) ? to_f(W[wi]) : 0.f;
        }
        __syncthreads();
#pragma unroll 8
        for (int kk = 0; kk < BK; ++kk) {
            float xa[4], wb[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) xa[i] = Xs[kk][ty * 4 + i];
#pragma unroll
            for (int j = 0; j < 4; ++j) wb[j] = Ws[kk][tx * 4 + j];
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(xa[i], wb[j], acc[i][j]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int gm = m0 + ty * 4 + i;
        if (gm >= M) continue;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int gn = n0 + tx * 4 + j;
            if (gn < N) Y[(size_t)gm * N + gn] = acc[i][j];
        }
    }
}

}  // namespace

cudaError_t launch_rmsnorm_rows(int x_bf16, const void *x, int row_mod, const float *gain,
                                float eps, int M, int d, ActOut out, cudaStream_t st) {
    if (d > kNormMaxD) {
        if (x_bf16)
            return launch_k(rmsnorm_rows_loop_kernel<bf16>, dim3(M), dim3(kRowThreads), 0, st,
                            (const bf16 *)x, row_mod, gain, eps, d, out);
        return launch_k(rmsnorm_rows_loop_kernel<float>, dim3(M), dim3(kRowThreads), 0, st,
                        (const float *)x, row_mod, gain, eps, d, out);
    }
    // few rows: 1024 threads per row, else 256 (more rows in flight per SM)
    const bool wide = M < 2 * sm_count_cached();
    const int V = ceil_div(d / 4, wide ? 1024 : kNormThreads);
#define SP_NORM_CASE(VV, TT)                                                                   \
    case VV:                                                                                   \
        return x_bf16 ? launch_k(rmsnorm_rows_kernel<bf16, VV, TT>, dim3(M), dim3(TT), 0, st,  \
                                 (const bf16 *)x, row_mod, gain, eps, d, out)                  \
                      : launch_k(rmsnorm_rows_kernel<float, VV, TT>, dim3(M), dim3(TT), 0, st, \
                                 (const float *)x, row_mod, gain, eps, d, out);
    if (wide) {
        switch (V) { SP_NORM_CASE(1, 1024) SP_NORM_CASE(2, 1024) }
    } else {
        switch (V) {
            SP_NORM_CASE(1, 256) SP_NORM_CASE(2, 256) SP_NORM_CASE(3, 256) SP_NORM_CASE(4, 256)
            SP_NORM_CASE(5, 256) SP_NORM_CASE(6, 256) SP_NORM_CASE(7, 256) SP_NORM_CASE(8, 256)
        }
    }
#undef SP_NORM_CASE
    return cudaErrorInvalidValue;
}

cudaError_t launch_qkv_rope(const QkvRopeArgs &a, cudaStream_t st) {
    // few rows: 1024 threads per row (one pass of items), else 256
    if (a.B * a.k < 2 * sm_count_cached())
        return launch_k(qkv_rope_kernel<1024>, dim3(a.B * a.k), dim3(1024), 0, st, a);
    return launch_k(qkv_rope_rows_kernel, dim3(a.B * a.k), dim3(256), 0, st, a);
}

cudaError_t launch_residual_norm(int x_bf16, PartIn y, const void *x, int row_mod,
                                 const float *gain, float eps, int M, int d, float *h1, ActOut n,
                                 cudaStream_t st, int y_div) {
    if (d > kNormMaxD) {
        if (x_bf16)
            return launch_k(residual_norm_loop_kernel<bf16>, dim3(M), dim3(kWideThreads), 0, st, y, y_div,
                            (const bf16 *)x, row_mod, gain, eps, d, h1, n);
        return launch_k(residual_norm_loop_kernel<float>, dim3(M), dim3(kWideThreads), 0, st, y, y_div,
                        (const float *)x, row_mod, gain, eps, d, h1, n);
    }
    const bool wide = M < 2 * sm_count_cached();
    const int V = ceil_div(d / 4, wide ? 1024 : kNormThreads);
#define SP_NORM_CASE(VV, TT)                                                                     \
    case VV:                                                                                     \
        return x_bf16 ? launch_k(residual_norm_kernel<bf16, VV, TT>, dim3(M), dim3(TT), 0, st, y,  \
                                 y_div, (const bf16 *)x, row_mod, gain, eps, d, h1, n)           \
                      : launch_k(residual_norm_kernel<float, VV, TT>, dim3(M), dim3(TT), 0, st, y, \
                                 y_div, (const float *)x, row_mod, gain, eps, d, h1, n);
    if (wide) {
        switch (V) { SP_NORM_CASE(1, 1024) SP_NORM_CASE(2, 1024) }
    } else {
        switch (V) {
            SP_NORM_CASE(1, 256) SP_NORM_CASE(2, 256) SP_NORM_CASE(3, 256) SP_NORM_CASE(4, 256)
            SP_NORM_CASE(5, 256) SP_NORM_CASE(6, 256) SP_NORM_CASE(7, 256) SP_NORM_CASE(8, 256)
        }
    }
#undef SP_NORM_CASE
    return cudaErrorInvalidValue;
}

cudaError_t launch_swiglu(PartIn y, int M, int f, int blk, ActOut a, cudaStream_t st) {
    const long long total = (long long)M * f / 4;
    int grid = (int)((total + 255) / 256);
    if (grid > 152 * 16) grid = 152 * 16;
    return launch_k(swiglu_kernel, dim3(grid), dim3(256), 0, st, y, M, f, blk, a);
}

size_t readout_scratch_bytes(int B, int d, int C) {
    // partial dot products [B][chunks][C], then square sums [B][chunks]
    return (size_t)B * ceil_div(d, kReadoutCols) * (C + 1) * sizeof(float);
}

cudaError_t launch_readout(PartIn y, const float *h1, const float *head_w, const float *head_b,
                           int pool, int B, int k, int d, int C, float *scratch, float *logits,
                           int *counters, cudaStream_t st, size_t sb, size_t sr, int n_tasks,
                           const float *g_final, float eps) {
    const int chunks = ceil_div(d, kReadoutCols);
    if (!sb) sb = (size_t)k * d;
    if (!sr) sr = d;
    if (n_tasks < 1) n_tasks = 1;
    float *ss = g_final ? scratch + (size_t)B * chunks * C : nullptr;
    return launch_k(readout_partial_kernel, dim3(chunks, B), dim3(64 * kReadoutGroups), 0, st, y, h1,
                    head_w, pool, k, d, C, scratch, sb, sr, n_tasks, g_final, ss, counters, head_b,
                    logits, eps);
}

cudaError_t launch_to_act(const float *x, size_t n, ActOut out, cudaStream_t st) {
    size_t grid = (n + 255) / 256;
    if (grid > 152 * 16) grid = 152 * 16;
    if (grid == 0) grid = 1;
    return launch_k(to_act_kernel, dim3((unsigned)grid), dim3(256), 0, st, x, n, out);
}

cudaError_t launch_sum_partials(PartIn y, size_t n, float *out, cudaStream_t st) {
    size_t grid = (n + 255) / 256;
    if (grid > 152 * 16) grid = 152 * 16;
    if (grid == 0) grid = 1;
    return launch_k(sum_partials_kernel, dim3((unsigned)grid), dim3(256), 0, st, y, n, out);
}

cudaError_t launch_gemm_simt(int w_bf16, const void *X, const void *W, float *Y, int M, int N,
                             int K, cudaStream_t st, bool w_blocked) {
    dim3 grid(ceil_div(N, 64), ceil_div(M, 64));
    if (w_bf16)
        return launch_k(gemm_simt_kernel<bf16>, grid, dim3(256), 0, st, (const float *)X, (const bf16 *)W,
                        Y, M, N, K, (int)w_blocked);
    else
        return launch_k(gemm_simt_kernel<float>, grid, dim3(256), 0, st, (const float *)X,
                        (const float *)W, Y, M, N, K, (int)w_blocked);
}

}  // namespace sp
