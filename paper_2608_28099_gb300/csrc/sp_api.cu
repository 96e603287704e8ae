// C ABI of libsp.so: handle lifetime, argument checks, the classify launch
// sequence (Sec. 3.2-3.3) and the stand-alone attention step (Eq. 1-3).
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <string>
#include <vector>

#include "sp_common.cuh"
#include "sp_gemm.cuh"

using namespace sp;

namespace {

thread_local std::string g_err;

sp_status fail(sp_status st, const char *fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    g_err = buf;
    return st;
}

#define SP_CUDA(call)                                                                       \
    do {                                                                                    \
        cudaError_t e_ = (call);                                                            \
        if (e_ != cudaSuccess)                                                              \
            return fail(SP_ERR_CUDA, "%s failed: %s (%s:%d)", #call, cudaGetErrorString(e_), \
                        __FILE__, __LINE__);                                                \
    } while (0)

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

// One device allocation carved into 256-byte aligned pieces.
struct Arena {
    char *base = nullptr;
    size_t used = 0, cap = 0;
    void *take(size_t bytes) {
        void *p = base + used;
        used += align256(bytes);
        return p;
    }
};

}  // namespace

void sp::set_error_text(const char *msg) { g_err = msg; }

struct sp_handle {
    sp_config cfg;
    int device = 0, n_sm = 148;
    int es = 2;        // bytes per stored weight element
    int nqkv = 0;      // (Hq + 2 Hkv) dh
    int gu_blk = 0;    // gate/up interleave block (columns)
    // weights
    WeightMat w_qkv, w_o, w_gu, w_down;
    float *g_in = nullptr, *g_post = nullptr, *head_w = nullptr, *head_b = nullptr;
    float *g_final = nullptr;     // LM-head readout: final RMSNorm gain (NULL: linear head)
    void *soft_prompt = nullptr;
    float *qkv_shared = nullptr;  // [k][nqkv] projections of the shared soft prompt
    float2 *rope_cs = nullptr;    // [max_seq_len + k][dh/2]
    // scratch
    Arena arena;
    ActBuf xn, o, n, a;           // inputs of the four projections
    float *y = nullptr;           // projection partials [splits][M][N]
    size_t y_bytes = 0;
    float *q = nullptr, *k_new = nullptr, *v_new = nullptr;
    void *attn_ws = nullptr;
    size_t attn_ws_bytes = 0;
    float *h1 = nullptr;          // [M][d]
    int *status = nullptr;
    int *stage_ids = nullptr, *stage_lens = nullptr;
    void *stage_rows = nullptr;
    float *stage_logits = nullptr;
    float *readout_part = nullptr;  // [B][chunks][C] partial head dot products
    int *readout_cnt = nullptr;     // [max_batch T] finished chunks per sequence (zero between calls)
    // input fusion (optional): x_{b,r} = W_fc_h RMSNorm(h_b; g_h) + fc_prompt[r]
    bool fused = false;
    WeightMat w_fc_h;             // [d][d]: the columns of W_fc acting on the hidden state
    float *g_h = nullptr;
    float *fc_prompt = nullptr;   // [k][d] W_fc (embedding columns) RMSNorm(soft_prompt; g_e)
    ActBuf xh;                    // normalised hidden states [max_batch][d]
    float *xrows = nullptr;       // fused input rows [max_batch k][d] fp32
    void *stage_hidden = nullptr; // host-entry staging [max_batch][d] w_dtype
    GemmPlanner gemm;
    // options
    int opt_split = 0, opt_gemm = 0, opt_attn = 0, opt_profile = 0, opt_recursive = 0;
    int opt_seg_cost = -1;  // attention segment-boundary cost in tiles (-1 = default)
    int opt_prec = 0;       // activation precision of the MLP inputs (SP_OPT_ACT_PRECISION)
    int opt_stall = 0;      // one-shot failure-path test (SP_OPT_DEBUG_STALL)
    int opt_merge = 0;      // where the attention partials are merged (SP_OPT_ATTN_MERGE)
    int opt_qprec = 0;      // attention query precision (SP_OPT_QUERY_PRECISION)
    int *dbg_pages = nullptr;     // sp_debug_gathered_pages: recording buffer (device)
    size_t dbg_pages_cap = 0;     // its capacity in ints
    int T = 1;        // tasks sharing the pass; cfg.k_rows holds T * k_task rows per sequence
    int k_task = 0;   // soft-prompt rows per task
    float *h2_all = nullptr;      // recursive probing: step outputs [k][max_batch][d] fp32
    int last_launches = 0;
    cudaEvent_t ev[SP_N_STAGES][2] = {};
    bool ev_used[SP_N_STAGES] = {};
    std::vector<void *> allocs;
};

namespace {

sp_status dev_alloc(sp_handle *h, void **p, size_t bytes) {
    *p = nullptr;
    if (bytes == 0) bytes = 256;
    cudaError_t e = cudaMalloc(p, bytes);
    if (e != cudaSuccess) {
        *p = nullptr;
        return fail(SP_ERR_OOM, "cudaMalloc(%zu) failed: %s", bytes, cudaGetErrorString(e));
    }
    h->allocs.push_back(*p);
    return SP_OK;
}

sp_status upload(sp_handle *h, void **dst, const void *src, size_t bytes) {
    sp_status st = dev_alloc(h, dst, bytes);
    if (st != SP_OK) return st;
    SP_CUDA(cudaMemcpy(*dst, src, bytes, cudaMemcpyHostToDevice));
    return SP_OK;
}

sp_status check_config(const sp_config *c) {
    if (!c) return fail(SP_ERR_INVALID_ARG, "config is NULL");
    if (c->d_model <= 0 || c->d_model % 8) return fail(SP_ERR_INVALID_ARG, "d_model must be a positive multiple of 8");
    if (c->n_kv_heads <= 0 || c->n_q_heads <= 0 || c->n_q_heads % c->n_kv_heads)
        return fail(SP_ERR_INVALID_ARG, "n_q_heads must be a positive multiple of n_kv_heads");
    if (c->head_dim != 32 && c->head_dim != 64 && c->head_dim != 128)
        return fail(SP_ERR_UNSUPPORTED, "head_dim %d unsupported (32, 64, 128)", c->head_dim);
    if (c->d_ff <= 0 || c->d_ff % 8) return fail(SP_ERR_INVALID_ARG, "d_ff must be a positive multiple of 8");
    if (c->k_rows < 1 || c->k_rows > 32) return fail(SP_ERR_INVALID_ARG, "k_rows must be in 1..32");
    if (c->n_tasks < 0 || c->n_tasks > 64) return fail(SP_ERR_INVALID_ARG, "n_tasks must be in 0..64");
    if (c->n_classes < 1) return fail(SP_ERR_INVALID_ARG, "n_classes must be >= 1");
    if (c->pool != SP_POOL_MEAN && c->pool != SP_POOL_LAST) return fail(SP_ERR_INVALID_ARG, "bad pool");
    if (c->w_dtype != SP_F32 && c->w_dtype != SP_BF16) return fail(SP_ERR_INVALID_ARG, "bad w_dtype");
    if (c->kv_dtype != SP_F32 && c->kv_dtype != SP_BF16) return fail(SP_ERR_INVALID_ARG, "bad kv_dtype");
    if (c->max_batch < 1) return fail(SP_ERR_INVALID_ARG, "max_batch must be >= 1");
    if (c->max_seq_len < 0) return fail(SP_ERR_INVALID_ARG, "max_seq_len must be >= 0");
    if (!(c->rope_theta > 0.f) || !(c->rms_eps >= 0.f)) return fail(SP_ERR_INVALID_ARG, "bad theta/eps");
    const int R = (c->n_q_heads / c->n_kv_heads) * c->k_rows * (c->n_tasks > 1 ? c->n_tasks : 1);
    if (R * c->head_dim > 128 * 128)
        return fail(SP_ERR_UNSUPPORTED, "query group x k_rows x head_dim too large (%d rows)", R);
    return SP_OK;
}

sp_status check_kv(const sp_kv_cache *kv, int kv_dtype) {
    (void)kv_dtype;
    if (!kv) return fail(SP_ERR_INVALID_ARG, "kv cache descriptor is NULL");
    if (kv->n_seqs < 1) return fail(SP_ERR_INVALID_ARG, "kv->n_seqs must be >= 1");
    if (kv->layout == SP_KV_CONTIGUOUS) {
        if (!kv->k_seq || !kv->v_seq) return fail(SP_ERR_INVALID_ARG, "contiguous cache needs k_seq and v_seq");
    } else if (kv->layout == SP_KV_PAGED) {
        if (!kv->k_pool || !kv->v_pool || !kv->page_table)
            return fail(SP_ERR_INVALID_ARG, "paged cache needs k_pool, v_pool and page_table");
        if ((((uintptr_t)kv->k_pool) | ((uintptr_t)kv->v_pool)) & 15)
            return fail(SP_ERR_INVALID_ARG, "k_pool and v_pool must be 16-byte aligned");
        if (kv->page_size != 16 && kv->page_size != 32 && kv->page_size != 64)
            return fail(SP_ERR_UNSUPPORTED, "page_size %d unsupported (16, 32, 64)", kv->page_size);
        if (kv->n_pages < 1 || kv->max_pages_per_seq < 1)
            return fail(SP_ERR_INVALID_ARG, "n_pages and max_pages_per_seq must be >= 1");
    } else {
        return fail(SP_ERR_INVALID_ARG, "bad kv layout %d", kv->layout);
    }
    return SP_OK;
}

KVDev to_dev(const sp_kv_cache *kv) {
    KVDev d;
    d.layout = kv->layout;
    d.k_seq = kv->k_seq;
    d.v_seq = kv->v_seq;
    d.k_pool = kv->k_pool;
    d.v_pool = kv->v_pool;
    d.page_table = kv->page_table;
    d.page_size = kv->page_size;
    d.n_pages = kv->n_pages;
    d.max_pages = kv->max_pages_per_seq;
    d.n_seqs = kv->n_seqs;
    return d;
}

int sm_count() {
    int dev = 0, n = 148;
    if (cudaGetDevice(&dev) == cudaSuccess)
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    return n;
}

// Largest attention workspace over every batch size up to max_batch.
size_t max_attention_ws(const sp_config &c, int n_sm, int forced_split) {
    const int G = c.n_q_heads / c.n_kv_heads;
    size_t best = 0;
    for (int B = 1; B <= c.max_batch; ++B) {
        int split, ns;
        plan_attention(B, c.n_kv_heads, c.k_rows, c.max_seq_len, forced_split, n_sm, &split, &ns);
        size_t b = attention_workspace_bytes(B, c.n_kv_heads, G * c.k_rows, c.head_dim, ns, n_sm);
        if (b > best) best = b;
    }
    return best;
}

// The merge counters of the attention workspace: [B][Hkv] ints at its start.
int *attention_counters(void *ws) { return (int *)ws; }

// Enqueue the attention step for AttnArgs with the counters and partial
// buffers taken from `ws`: the tensor-core kernel (balanced over the SMs, merge
// inside) or the CUDA-core split kernel followed by its merge kernel.
// counters_zeroed: the preceding kernel of this stream cleared the merge
// counters (else they are cleared here).
sp_status enqueue_attention(AttnArgs &a, void *ws, size_t ws_bytes, int attn_path, int n_sm,
                            int forced_split, int *launches, cudaStream_t st, bool counters_zeroed,
                            cudaEvent_t *ev_attn = nullptr, cudaEvent_t *ev_merge = nullptr,
                            int seg_cost = -1, int merge_mode = 0) {
    a.tc_ctas = attn_tc_ctas(n_sm, a.Hkv);
    a.tc_min_tiles = forced_split > 0 ? forced_split / 64 : kAttnMinTiles;
    a.tc_seg_cost = seg_cost >= 0 ? seg_cost
                                  : (a.kv.layout == SP_KV_CONTIGUOUS ? kAttnSegCostContiguous : kAttnSegCost);
    // few sequences over many groups: each pair has many partials, merged by a
    // kernel spread over (head, sequence, row) instead of one CTA per pair
    a.tc_merge_kernel = merge_mode == 2 || (merge_mode == 0 && 4 * a.B < a.tc_ctas / a.Hkv);
    const size_t need = attention_workspace_bytes(a.B, a.Hkv, a.R, a.dh, a.n_splits, n_sm);
    if (ws_bytes < need) return fail(SP_ERR_INVALID_ARG, "attention workspace too small (%zu < %zu)", ws_bytes, need);
    const size_t pairs = (size_t)a.B * a.Hkv;
    size_t parts = pairs * a.n_splits;
    if ((size_t)a.tc_ctas + pairs > parts) parts = (size_t)a.tc_ctas + pairs;
    a.counters = attention_counters(ws);
    a.part_o = (float *)((char *)ws + align256(pairs * sizeof(int)));
    a.part_ml = (float *)((char *)a.part_o + align256(parts * a.R * a.dh * sizeof(float)));
    bool tc = attn_path != 1 && attention_tc_supported(a);
    CUtensorMap mk, mv;
    const CUtensorMap *pk = nullptr, *pv = nullptr;
    if (tc && a.kv.layout == SP_KV_PAGED) {
        const long long blocks = (long long)a.kv.n_pages * a.Hkv;
        tc = encode_kv_pages_bf16(&mk, a.kv.k_pool, blocks, a.kv.page_size) &&
             encode_kv_pages_bf16(&mv, a.kv.v_pool, blocks, a.kv.page_size);
        pk = &mk;
        pv = &mv;
    }
    if (attn_path == 2 && !tc)
        return fail(SP_ERR_UNSUPPORTED, "tensor-core attention needs head_dim 128, a bf16 cache, "
                                        "at most 128 query rows per kv head and at most 2048 sequences");
    a.subs = 1;  // one partial per unit on the CUDA-core path
    if (tc && !counters_zeroed) SP_CUDA(cudaMemsetAsync(a.counters, 0, pairs * sizeof(int), st));
    if (ev_attn) cudaEventRecordWithFlags(ev_attn[0], st, cudaEventRecordExternal);
    if (tc)
        SP_CUDA(launch_attention_tc(a, pk, pv, st));
    else
        SP_CUDA(launch_attention_simt(a, st));
    if (ev_attn) cudaEventRecordWithFlags(ev_attn[1], st, cudaEventRecordExternal);
    if (ev_merge) cudaEventRecordWithFlags(ev_merge[0], st, cudaEventRecordExternal);
    if (!tc) SP_CUDA(launch_attention_merge(a, st));
    if (ev_merge) cudaEventRecordWithFlags(ev_merge[1], st, cudaEventRecordExternal);
    *launches += tc && !a.tc_merge_kernel ? 1 : 2;
    return SP_OK;
}

}  // namespace

extern "C" {

const char *sp_last_error(void) { return g_err.c_str(); }

sp_status sp_create(const sp_config *cfg, const sp_weights *w, sp_handle **out) {
    if (!out) return fail(SP_ERR_INVALID_ARG, "out is NULL");
    *out = nullptr;
    sp_status st = check_config(cfg);
    if (st != SP_OK) return st;
    if (!w || !w->w_q || !w->w_k || !w->w_v || !w->w_o || !w->w_gate || !w->w_up || !w->w_down ||
        !w->g_in || !w->g_post || !w->soft_prompt || !w->head_w)
        return fail(SP_ERR_INVALID_ARG, "a required weight pointer is NULL");

    sp_handle *h = new sp_handle();
    h->cfg = *cfg;
    // several tasks: their rows are stacked per sequence ([T][k] rows), so the
    // layer runs on T k rows; k_task keeps the per-task row count
    h->T = cfg->n_tasks > 1 ? cfg->n_tasks : 1;
    h->k_task = cfg->k_rows;
    h->cfg.k_rows = cfg->k_rows * h->T;
    const sp_config &c = h->cfg;
    cudaGetDevice(&h->device);
    h->n_sm = sm_count();
    h->es = c.w_dtype == SP_BF16 ? 2 : 4;
    const int d = c.d_model, hq = c.n_q_heads, hkv = c.n_kv_heads, dh = c.head_dim, f = c.d_ff;
    const int k = c.k_rows, C = c.n_classes;
    h->nqkv = (hq + 2 * hkv) * dh;
    // [W_gate; W_up] for the tensor cores: 64-row blocks interleaved (gate rows
    // 64i.., then the matching up rows), so that one 128-row weight tile holds
    // both halves of 64 SwiGLU features and the gate/up projection can apply
    // SwiGLU in its epilogue; otherwise the gate block then the up block
    const bool gu_tc = c.w_dtype == SP_BF16 && tc_supported(2 * f, d) && f % 64 == 0;
    h->gu_blk = gu_tc ? 64 : f;
    const size_t es = h->es;
    auto cleanup = [&](sp_status s) {
        sp_destroy(h);
        return s;
    };

    // weights: [W_q; W_k; W_v] and [W_gate; W_up] concatenated along the output
    // dim; bf16 matrices the tensor cores take are stored in 16 KB (tile,
    // k-block) blocks (block_weights_layout), the rest row-major
    const int wb = c.w_dtype == SP_BF16;
    auto upload_weight = [&](WeightMat &wm, const char *src, int N, int K) -> sp_status {
        const size_t bytes = (size_t)N * K * es;
        const bool blocked = wb && tc_supported(N, K);
        std::vector<char> blk;
        if (blocked) {
            blk.resize(bytes);
            block_weights_layout(src, blk.data(), N, K, es);
            src = blk.data();
        }
        void *p = nullptr;
        sp_status s2 = upload(h, &p, src, bytes);
        if (s2 != SP_OK) return s2;
        init_weight(wm, p, N, K, wb, blocked);
        return SP_OK;
    };
    {
        std::vector<char> buf((size_t)h->nqkv * d * es);
        memcpy(buf.data(), w->w_q, (size_t)hq * dh * d * es);
        memcpy(buf.data() + (size_t)hq * dh * d * es, w->w_k, (size_t)hkv * dh * d * es);
        memcpy(buf.data() + (size_t)(hq + hkv) * dh * d * es, w->w_v, (size_t)hkv * dh * d * es);
        if ((st = upload_weight(h->w_qkv, buf.data(), h->nqkv, d)) != SP_OK) return cleanup(st);
    }
    {
        std::vector<char> buf((size_t)2 * f * d * es);
        const int blk = h->gu_blk;
        const size_t rowb = (size_t)d * es;
        for (int i = 0; i < f / blk; ++i) {
            memcpy(buf.data() + (size_t)2 * i * blk * rowb, (const char *)w->w_gate + (size_t)i * blk * rowb,
                   (size_t)blk * rowb);
            memcpy(buf.data() + (size_t)(2 * i + 1) * blk * rowb, (const char *)w->w_up + (size_t)i * blk * rowb,
                   (size_t)blk * rowb);
        }
        if ((st = upload_weight(h->w_gu, buf.data(), 2 * f, d)) != SP_OK) return cleanup(st);
    }
    if ((st = upload_weight(h->w_o, (const char *)w->w_o, d, hq * dh)) != SP_OK) return cleanup(st);
    if ((st = upload_weight(h->w_down, (const char *)w->w_down, d, f)) != SP_OK) return cleanup(st);
    if ((st = upload(h, (void **)&h->g_in, w->g_in, d * sizeof(float))) != SP_OK) return cleanup(st);
    if ((st = upload(h, (void **)&h->g_post, w->g_post, d * sizeof(float))) != SP_OK) return cleanup(st);
    if ((st = upload(h, &h->soft_prompt, w->soft_prompt, (size_t)k * d * es)) != SP_OK) return cleanup(st);
    if ((st = upload(h, (void **)&h->head_w, w->head_w, (size_t)h->T * C * d * sizeof(float))) != SP_OK)
        return cleanup(st);
    if (w->head_b &&
        (st = upload(h, (void **)&h->head_b, w->head_b, (size_t)h->T * C * sizeof(float))) != SP_OK)
        return cleanup(st);
    if (w->g_final &&
        (st = upload(h, (void **)&h->g_final, w->g_final, d * sizeof(float))) != SP_OK)
        return cleanup(st);
    // input fusion: W_fc [d][2d] split into its hidden-state half (a projection
    // of every call) and its embedding half (applied once to the soft prompt below)
    std::vector<char> w_fc_e;
    if (w->w_fc || w->g_h || w->g_e) {
        if (!w->w_fc || !w->g_h || !w->g_e)
            return cleanup(fail(SP_ERR_INVALID_ARG, "input fusion needs w_fc, g_h and g_e together"));
        std::vector<char> wh((size_t)d * d * es);
        w_fc_e.resize((size_t)d * d * es);
        for (int i = 0; i < d; ++i) {
            const char *row = (const char *)w->w_fc + (size_t)i * 2 * d * es;
            memcpy(wh.data() + (size_t)i * d * es, row, (size_t)d * es);
            memcpy(w_fc_e.data() + (size_t)i * d * es, row + (size_t)d * es, (size_t)d * es);
        }
        if ((st = upload_weight(h->w_fc_h, wh.data(), d, d)) != SP_OK) return cleanup(st);
        if ((st = upload(h, (void **)&h->g_h, w->g_h, d * sizeof(float))) != SP_OK) return cleanup(st);
        h->fused = true;
    }

    // rotary table: angle (position p, pair i) = p * theta^(-2i/dh), evaluated in double
    {
        const int npos = c.max_seq_len + k, half = dh / 2;
        std::vector<float2> cs((size_t)npos * half);
        std::vector<double> freq(half);
        for (int i = 0; i < half; ++i) freq[i] = pow((double)c.rope_theta, -2.0 * i / dh);
        for (int p = 0; p < npos; ++p)
            for (int i = 0; i < half; ++i) {
                const double ang = (double)p * freq[i];
                cs[(size_t)p * half + i] = make_float2((float)cos(ang), (float)sin(ang));
            }
        if ((st = upload(h, (void **)&h->rope_cs, cs.data(), cs.size() * sizeof(float2))) != SP_OK)
            return cleanup(st);
    }

    // scratch for max_batch sequences
    const size_t M = (size_t)c.max_batch * k;
    size_t maxN = (size_t)h->nqkv;
    if ((size_t)d > maxN) maxN = d;
    if ((size_t)2 * f > maxN) maxN = 2 * (size_t)f;
    h->attn_ws_bytes = max_attention_ws(c, h->n_sm, 0);
    // projection partials: room for up to 4 splits of the widest output, and
    // for as many splits as one wave of CTAs can use on the narrow outputs
    h->y_bytes = M * maxN * 4 * 4;
    const size_t narrow = (size_t)h->n_sm * (M < 128 ? 128 : M) * 128 * 4;
    if (narrow > h->y_bytes) h->y_bytes = narrow;
    h->gemm.init(h->n_sm, h->y_bytes);
    size_t total = 0;
    const size_t sizes[] = {M * d * 4,                  // xn (fp32, or bf16 hi+lo)
                            h->y_bytes,                 // y partials
                            M * hq * dh * 4,            // q
                            M * hkv * dh * 4,           // k_new
                            M * hkv * dh * 4,           // v_new
                            h->attn_ws_bytes,           // attention partials
                            M * hq * dh * 4,            // o
                            M * d * 4,                  // h1
                            M * d * 4,                  // n
                            M * f * 4,                  // a
                            256,                        // status
                            (size_t)c.max_batch * 4,    // stage ids
                            (size_t)c.max_batch * 4,    // stage lens
                            M * d * es,                 // stage rows
                            (size_t)c.max_batch * h->T * C * 4,  // stage logits
                            (size_t)k * h->nqkv * 4,    // qkv_shared
                            readout_scratch_bytes(c.max_batch * h->T, d, C),  // readout partials
                            h->fused ? (size_t)c.max_batch * d * 4 : 0,  // xh
                            h->fused ? M * d * 4 : 0,                    // xrows
                            h->fused ? (size_t)k * d * 4 : 0,            // fc_prompt
                            h->fused ? (size_t)c.max_batch * d * es : 0,  // stage hidden
                            h->fused ? M * d * 4 : 0,                    // h2_all
                            (size_t)c.max_batch * h->T * 4};             // readout counters
    for (size_t sz : sizes) total += align256(sz);
    void *arena = nullptr;
    if ((st = dev_alloc(h, &arena, total)) != SP_OK) return cleanup(st);
    h->arena.base = (char *)arena;
    h->arena.cap = total;
    void *p_xn = h->arena.take(sizes[0]);
    h->y = (float *)h->arena.take(sizes[1]);
    h->q = (float *)h->arena.take(sizes[2]);
    h->k_new = (float *)h->arena.take(sizes[3]);
    h->v_new = (float *)h->arena.take(sizes[4]);
    h->attn_ws = h->arena.take(sizes[5]);
    void *p_o_act = h->arena.take(sizes[6]);
    h->h1 = (float *)h->arena.take(sizes[7]);
    void *p_n = h->arena.take(sizes[8]);
    void *p_a = h->arena.take(sizes[9]);
    h->status = (int *)h->arena.take(sizes[10]);
    h->stage_ids = (int *)h->arena.take(sizes[11]);
    h->stage_lens = (int *)h->arena.take(sizes[12]);
    h->stage_rows = h->arena.take(sizes[13]);
    h->stage_logits = (float *)h->arena.take(sizes[14]);
    h->qkv_shared = (float *)h->arena.take(sizes[15]);
    h->readout_part = (float *)h->arena.take(sizes[16]);
    void *p_xh = h->arena.take(sizes[17]);
    h->xrows = (float *)h->arena.take(sizes[18]);
    h->fc_prompt = (float *)h->arena.take(sizes[19]);
    h->stage_hidden = h->arena.take(sizes[20]);
    h->h2_all = (float *)h->arena.take(sizes[21]);
    h->readout_cnt = (int *)h->arena.take(sizes[22]);
    if (h->fused) init_act(h->xh, p_xh, c.max_batch, d, h->w_fc_h.tc);
    init_act(h->xn, p_xn, (int)M, d, h->w_qkv.tc);
    init_act(h->o, p_o_act, (int)M, hq * dh, h->w_o.tc);
    init_act(h->n, p_n, (int)M, d, h->w_gu.tc);
    init_act(h->a, p_a, (int)M, f, h->w_down.tc);
    if (cudaMemset(h->status, 0, 256) != cudaSuccess ||
        cudaMemset(h->readout_cnt, 0, sizes[22]) != cudaSuccess)
        return cleanup(fail(SP_ERR_CUDA, "memset failed"));

    // projections of the shared soft prompt rows (they do not depend on the
    // sequence), on CUDA cores with fp32 activations
    {
        cudaError_t e = launch_rmsnorm_rows(wb, h->soft_prompt, 0, h->g_in, c.rms_eps, k, d,
                                            h->xn.out(false), 0);
        if (e == cudaSuccess)
            e = launch_gemm_simt(wb, h->xn.ptr, h->w_qkv.ptr, h->qkv_shared, k, h->nqkv, d, 0,
                                 h->w_qkv.blocked);
        if (e == cudaSuccess) e = cudaDeviceSynchronize();
        if (e != cudaSuccess)
            return cleanup(fail(SP_ERR_CUDA, "shared prompt projection failed: %s", cudaGetErrorString(e)));
    }
    // the soft prompt's share of the fused input: fc_prompt = W_fc_e RMSNorm(e; g_e),
    // fp32, on CUDA cores (temporaries freed before returning)
    if (h->fused) {
        void *p_we = nullptr, *p_ge = nullptr, *p_en = nullptr;
        cudaError_t e = cudaMalloc(&p_we, w_fc_e.size());
        if (e == cudaSuccess) e = cudaMalloc(&p_ge, d * sizeof(float));
        if (e == cudaSuccess) e = cudaMalloc(&p_en, (size_t)k * d * sizeof(float));
        if (e == cudaSuccess) e = cudaMemcpy(p_we, w_fc_e.data(), w_fc_e.size(), cudaMemcpyHostToDevice);
        if (e == cudaSuccess) e = cudaMemcpy(p_ge, w->g_e, d * sizeof(float), cudaMemcpyHostToDevice);
        ActOut en = {(float *)p_en, nullptr, nullptr};
        if (e == cudaSuccess)
            e = launch_rmsnorm_rows(wb, h->soft_prompt, 0, (const float *)p_ge, c.rms_eps, k, d, en, 0);
        if (e == cudaSuccess) e = launch_gemm_simt(wb, p_en, p_we, h->fc_prompt, k, d, d, 0);
        if (e == cudaSuccess) e = cudaDeviceSynchronize();
        cudaFree(p_we);
        cudaFree(p_ge);
        cudaFree(p_en);
        if (e != cudaSuccess)
            return cleanup(fail(SP_ERR_CUDA, "fused prompt projection failed: %s", cudaGetErrorString(e)));
    }
    *out = h;
    return SP_OK;
}

sp_status sp_destroy(sp_handle *h) {
    if (!h) return SP_OK;
    cudaDeviceSynchronize();
    for (auto &pair : h->ev)
        for (cudaEvent_t &e : pair)
            if (e) cudaEventDestroy(e);
    for (void *p : h->allocs) cudaFree(p);
    delete h;
    return SP_OK;
}

sp_status sp_set_option(sp_handle *h, int key, int value) {
    if (!h) return fail(SP_ERR_INVALID_ARG, "handle is NULL");
    switch (key) {
    case SP_OPT_SPLIT_TOKENS: {
        if (value < 0 || value % 64) return fail(SP_ERR_INVALID_ARG, "split tokens must be a multiple of 64");
        const size_t need = max_attention_ws(h->cfg, h->n_sm, value);
        if (need > h->attn_ws_bytes) {
            // a finer forced plan: grow the attention scratch now, never in classify
            void *p = nullptr;
            sp_status st = dev_alloc(h, &p, need);
            if (st != SP_OK) return st;
            h->attn_ws = p;
            h->attn_ws_bytes = need;
        }
        h->opt_split = value;
        return SP_OK;
    }
    case SP_OPT_GEMM_PATH:
        if (value < 0 || value > 2) return fail(SP_ERR_INVALID_ARG, "bad gemm path");
        h->opt_gemm = value;
        return SP_OK;
    case SP_OPT_ATTN_PATH:
        if (value < 0 || value > 2) return fail(SP_ERR_INVALID_ARG, "bad attention path");
        h->opt_attn = value;
        return SP_OK;
    case SP_OPT_RECURSIVE:
        if (value != 0 && value != 1) return fail(SP_ERR_INVALID_ARG, "bad recursion flag");
        h->opt_recursive = value;
        return SP_OK;
    case SP_OPT_DEBUG_STALL:
        if (value != 0 && value != 1) return fail(SP_ERR_INVALID_ARG, "bad stall flag");
        h->opt_stall = value;
        return SP_OK;
    case SP_OPT_ACT_PRECISION:
        if (value < 0 || value > 4) return fail(SP_ERR_INVALID_ARG, "bad activation precision");
        h->opt_prec = value;
        return SP_OK;
    case SP_OPT_QUERY_PRECISION:
        if (value < 0 || value > 2) return fail(SP_ERR_INVALID_ARG, "bad query precision");
        h->opt_qprec = value;
        return SP_OK;
    case SP_OPT_ATTN_MERGE:
        if (value < 0 || value > 2) return fail(SP_ERR_INVALID_ARG, "bad attention merge mode");
        h->opt_merge = value;
        return SP_OK;
    case SP_OPT_GEMM_SCHEDULE:
        if (value < 0 || value > 2) return fail(SP_ERR_INVALID_ARG, "bad gemm schedule");
        h->gemm.sched = value;
        return SP_OK;
    case SP_OPT_ATTN_SEG_COST:
        if (value < -1 || value > 1024) return fail(SP_ERR_INVALID_ARG, "bad segment cost");
        h->opt_seg_cost = value;
        return SP_OK;
    case SP_OPT_PROFILE:
        if (value != 0 && value != 1) return fail(SP_ERR_INVALID_ARG, "bad profile flag");
        if (value && !h->ev[0][0]) {
            for (auto &pair : h->ev)
                for (cudaEvent_t &e : pair) SP_CUDA(cudaEventCreate(&e));
        }
        h->opt_profile = value;
        return SP_OK;
    default:
        return fail(SP_ERR_INVALID_ARG, "unknown option %d", key);
    }
}

int sp_last_launch_count(const sp_handle *h) { return h ? h->last_launches : -1; }

sp_status sp_debug_gathered_pages(sp_handle *h, int *d_out, size_t capacity) {
    if (!h) return fail(SP_ERR_INVALID_ARG, "handle is NULL");
    if (d_out && capacity == 0) return fail(SP_ERR_INVALID_ARG, "capacity must be > 0");
    h->dbg_pages = d_out;
    h->dbg_pages_cap = d_out ? capacity : 0;
    return SP_OK;
}

sp_status sp_stage_times(sp_handle *h, float *ms, int n) {
    if (!h || !ms || n < 0) return fail(SP_ERR_INVALID_ARG, "bad arguments");
    if (!h->opt_profile) return fail(SP_ERR_INVALID_ARG, "profiling is off (SP_OPT_PROFILE)");
    for (int i = 0; i < n; ++i) {
        ms[i] = -1.f;
        if (i >= SP_N_STAGES || !h->ev_used[i]) continue;
        SP_CUDA(cudaEventSynchronize(h->ev[i][1]));
        SP_CUDA(cudaEventElapsedTime(&ms[i], h->ev[i][0], h->ev[i][1]));
    }
    return SP_OK;
}

// Recursive probing SP-k (Sec. 3.2): k steps, each one layer pass of one row per
// sequence.  Step i fuses the previous step's output (the base hidden state at
// i = 0) with soft-prompt row i, sits at position L_b + i, appends its new key
// and value to the k_new / v_new rows of the sequence and attends to the cache
// and new rows 0..i.  Step outputs go to h2_all (step-major); the head reads
// their pool.  The normalisation of a step's output for the next fusion is
// fused into the kernel that forms it (residual + down projection).
static sp_status recursive_impl(sp_handle *h, cudaStream_t st, int batch, const int *d_seq_ids,
                                const int *d_seq_lens, int lens_by_batch, const sp_kv_cache *kv,
                                const void *d_hidden, float *d_logits) {
    if (h->T > 1) return fail(SP_ERR_UNSUPPORTED, "recursive probing runs one task per handle");
    const sp_config &c = h->cfg;
    const int d = c.d_model, hq = c.n_q_heads, hkv = c.n_kv_heads, dh = c.head_dim, f = c.d_ff;
    const int k = c.k_rows, C = c.n_classes, G = hq / hkv;
    const int B = batch;
    const int wb = c.w_dtype == SP_BF16;
    const size_t Bd = (size_t)B * d;
    int launches = 0;
    sp_status s;
    const bool tc_fc = h->gemm.use_tc(h->w_fc_h, h->xh, h->opt_gemm);
    const bool tc_qkv = h->gemm.use_tc(h->w_qkv, h->xn, h->opt_gemm);
    const bool tc_o = h->gemm.use_tc(h->w_o, h->o, h->opt_gemm);
    const bool tc_gu = h->gemm.use_tc(h->w_gu, h->n, h->opt_gemm);
    const bool tc_down = h->gemm.use_tc(h->w_down, h->a, h->opt_gemm);
    for (bool &u : h->ev_used) u = false;
    int ns = 1;
    SP_CUDA(launch_rmsnorm_rows(wb, d_hidden, 0, h->g_h, c.rms_eps, B, d, h->xh.out(tc_fc), st));
    ++launches;
    // one split plan for every step: keys extend to L_b + k at the last step
    int split_tokens = 0, n_splits = 0;
    plan_attention(B, hkv, k, c.max_seq_len, h->opt_split, h->n_sm, &split_tokens, &n_splits);
    for (int i = 0; i < k; ++i) {
        // fusion: x_i = W_fc_h RMSNorm(prev; g_h) + fc_prompt[i]; x_hat = RMSNorm(x_i; g_in)
        s = h->gemm.run(wb, h->opt_gemm, h->xh, h->w_fc_h, h->y, B, h->status, st, &launches, &ns);
        if (s != SP_OK) return fail(s, "fusion projection launch failed");
        SP_CUDA(launch_residual_norm(0, PartIn{h->y, ns, Bd}, h->fc_prompt + (size_t)i * d, 1, h->g_in,
                                     c.rms_eps, B, d, h->xrows, h->xn.out(tc_qkv), st));
        ++launches;
        s = h->gemm.run(wb, h->opt_gemm, h->xn, h->w_qkv, h->y, B, h->status, st, &launches, &ns);
        if (s != SP_OK) return fail(s, "Q/K/V projection launch failed");
        QkvRopeArgs r;
        memset(&r, 0, sizeof r);
        r.y = PartIn{h->y, ns, (size_t)B * h->nqkv};
        r.shared = 0;
        r.B = B; r.k = 1; r.Hq = hq; r.Hkv = hkv; r.dh = dh;
        r.r0 = i; r.kn_stride = k;
        r.seq_ids = d_seq_ids; r.seq_lens = d_seq_lens; r.lens_by_batch = lens_by_batch;
        r.n_seqs = kv->n_seqs; r.max_seq_len = c.max_seq_len;
        r.rope_cs = h->rope_cs;
        r.q = h->q; r.k_new = h->k_new; r.v_new = h->v_new;
        r.status = h->status;
        r.zero_ints = attention_counters(h->attn_ws);
        r.n_zero = B * hkv;
        SP_CUDA(launch_qkv_rope(r, st));
        ++launches;
        AttnArgs a;
        memset(&a, 0, sizeof a);
        a.B = B; a.Hq = hq; a.Hkv = hkv; a.dh = dh; a.k = 1; a.G = G; a.R = G;
        a.r0 = i; a.kn_stride = k;
        a.kv_bf16 = c.kv_dtype == SP_BF16;
        a.split_tokens = split_tokens;
        a.n_splits = n_splits;
        a.max_seq_len = c.max_seq_len;
        a.seq_ids = d_seq_ids; a.seq_lens = d_seq_lens; a.lens_by_batch = lens_by_batch;
        a.kv = to_dev(kv);
        a.q = h->q; a.k_new = h->k_new; a.v_new = h->v_new;
        a.status = h->status;
        a.scale_log2 = (float)(1.4426950408889634 / sqrt((double)dh));
        a.out = h->o.out(tc_o);
        s = enqueue_attention(a, h->attn_ws, h->attn_ws_bytes, h->opt_attn, h->n_sm, h->opt_split,
                              &launches, st, true);
        if (s != SP_OK) return s;
        s = h->gemm.run(wb, h->opt_gemm, h->o, h->w_o, h->y, B, h->status, st, &launches, &ns);
        if (s != SP_OK) return fail(s, "output projection launch failed");
        SP_CUDA(launch_residual_norm(0, PartIn{h->y, ns, Bd}, h->xrows, 0, h->g_post, c.rms_eps, B, d,
                                     h->h1, h->n.out(tc_gu), st));
        ++launches;
        s = h->gemm.run(wb, h->opt_gemm, h->n, h->w_gu, h->y, B, h->status, st, &launches, &ns);
        if (s != SP_OK) return fail(s, "gate/up projection launch failed");
        SP_CUDA(launch_swiglu(PartIn{h->y, ns, (size_t)B * 2 * f}, B, f, h->gu_blk, h->a.out(tc_down), st));
        ++launches;
        s = h->gemm.run(wb, h->opt_gemm, h->a, h->w_down, h->y, B, h->status, st, &launches, &ns);
        if (s != SP_OK) return fail(s, "down projection launch failed");
        // a_i = h1 + W_down a -> h2_all[i]; RMSNorm(a_i; g_h) is the next step's fusion input
        SP_CUDA(launch_residual_norm(0, PartIn{h->y, ns, Bd}, h->h1, 0, h->g_h, c.rms_eps, B, d,
                                     h->h2_all + (size_t)i * Bd, h->xh.out(tc_fc), st));
        ++launches;
    }
    SP_CUDA(launch_readout(PartIn{nullptr, 0, 0}, h->h2_all, h->head_w, h->head_b, c.pool, B, k, d, C,
                           h->readout_part, d_logits, h->readout_cnt, st, (size_t)d, Bd, 1, h->g_final, c.rms_eps));
    ++launches;
    h->last_launches = launches;
    return SP_OK;
}

static sp_status classify_impl(sp_handle *h, cudaStream_t st, int batch, const int *d_seq_ids,
                               const int *d_seq_lens, int lens_by_batch, const sp_kv_cache *kv,
                               const void *d_rows, float *d_logits, const void *d_hidden = nullptr) {
    if (!h) return fail(SP_ERR_INVALID_ARG, "handle is NULL");
    const sp_config &c = h->cfg;
    if (batch < 1 || batch > c.max_batch)
        return fail(SP_ERR_INVALID_ARG, "batch %d outside 1..max_batch (%d)", batch, c.max_batch);
    if (!d_seq_lens || !d_logits) return fail(SP_ERR_INVALID_ARG, "seq_lens and logits are required");
    sp_status s = check_kv(kv, c.kv_dtype);
    if (s != SP_OK) return s;
    if (!d_seq_ids && batch > kv->n_seqs)
        return fail(SP_ERR_INVALID_ARG, "batch %d exceeds n_seqs %d with implicit ids", batch, kv->n_seqs);
    if (d_rows && ((uintptr_t)d_rows & 15))
        return fail(SP_ERR_INVALID_ARG, "d_rows must be 16-byte aligned");
    if (d_hidden && !h->fused)
        return fail(SP_ERR_INVALID_ARG, "the handle was created without input fusion (w_fc)");
    if (d_hidden && ((uintptr_t)d_hidden & 15))
        return fail(SP_ERR_INVALID_ARG, "d_hidden must be 16-byte aligned");
    if (d_hidden && h->opt_recursive)
        return recursive_impl(h, st, batch, d_seq_ids, d_seq_lens, lens_by_batch, kv, d_hidden,
                              d_logits);

    const int d = c.d_model, hq = c.n_q_heads, hkv = c.n_kv_heads, dh = c.head_dim, f = c.d_ff;
    const int k = c.k_rows, C = c.n_classes, G = hq / hkv;
    const int M = batch * k;
    const int wb = c.w_dtype == SP_BF16;
    int launches = 0;
    for (bool &u : h->ev_used) u = false;
    auto mark = [&](int stage, int end) {
        if (!h->opt_profile) return;
        cudaEventRecordWithFlags(h->ev[stage][end], st, cudaEventRecordExternal);
        h->ev_used[stage] = true;
    };

    const size_t stride_qkv = (size_t)M * h->nqkv;
    const bool tc_qkv = h->gemm.use_tc(h->w_qkv, h->xn, h->opt_gemm);
    const bool tc_o = h->gemm.use_tc(h->w_o, h->o, h->opt_gemm);
    const bool tc_gu = h->gemm.use_tc(h->w_gu, h->n, h->opt_gemm);
    const bool tc_down = h->gemm.use_tc(h->w_down, h->a, h->opt_gemm);
    int ns = 1;
    // The MLP inputs (the post-norm n and the SwiGLU output a) go to the tensor
    // cores as plain bf16 when the head averages at least 8 rows per pooled
    // state (the rows' independent rounding errors average out in the mean;
    // the measured budget is in the design notes), else as hi + lo planes; the
    // Q/K/V and output projection inputs (x_hat, o) as hi + lo unless an option
    // asks otherwise, and the attention's queries as plain bf16 from 16 pooled
    // rows on.
    const bool mean = c.pool == SP_POOL_MEAN;
    const bool mlp_lo = h->opt_prec == 1 || (h->opt_prec == 0 && !(mean && h->k_task >= 8));
    const bool proj_lo = h->opt_prec != 3 && h->opt_prec != 4;
    const bool qkv_lo = h->opt_prec != 3;
    const bool q_plain = h->opt_qprec == 2 || (h->opt_qprec == 0 && mean && h->k_task >= 16);

    // a1-a2: pre-norm, Q/K/V projection, rotation at positions L_b + r (in the
    // projection's epilogue when it runs one CTA per head, else a kernel of its own)
    PartIn yqkv = {h->qkv_shared, 1, 0};
    const bool rope_fused = (d_rows || d_hidden) && dh == 128 &&
                            h->gemm.rope_fusable(h->w_qkv, h->xn, h->opt_gemm, M, qkv_lo);
    RopeEpi re;
    memset(&re, 0, sizeof re);
    re.rope_cs = h->rope_cs;
    re.Hq = hq; re.Hkv = hkv; re.k = k; re.kn_stride = 0; re.r0 = 0; re.k_task = h->k_task;
    re.seq_ids = d_seq_ids; re.seq_lens = d_seq_lens; re.lens_by_batch = lens_by_batch;
    re.n_seqs = kv->n_seqs; re.max_seq_len = c.max_seq_len;
    re.q = h->q; re.k_new = h->k_new; re.v_new = h->v_new;
    re.status = h->status;
    re.zero_ints = attention_counters(h->attn_ws);
    re.n_zero = batch * hkv;
    const RopeEpi *rp = rope_fused ? &re : nullptr;
    if (d_hidden) {
        // input fusion: u_b = W_fc_h RMSNorm(h_b; g_h); x_{b,r} = u_b + fc_prompt[r],
        // stored for the residual, and x_hat = RMSNorm(x; g_in) for Q/K/V
        const bool tc_fc = h->gemm.use_tc(h->w_fc_h, h->xh, h->opt_gemm);
        int ns_fc = 1;
        mark(SP_STAGE_FUSION, 0);
        SP_CUDA(launch_rmsnorm_rows(wb, d_hidden, 0, h->g_h, c.rms_eps, batch, d, h->xh.out(tc_fc), st));
        ++launches;
        s = h->gemm.run(wb, h->opt_gemm, h->xh, h->w_fc_h, h->y, batch, h->status, st, &launches, &ns_fc);
        mark(SP_STAGE_FUSION, 1);
        if (s != SP_OK) return fail(s, "fusion projection launch failed");
        mark(SP_STAGE_INPUT_NORM, 0);
        SP_CUDA(launch_residual_norm(0, PartIn{h->y, ns_fc, (size_t)batch * d}, h->fc_prompt, k,
                                     h->g_in, c.rms_eps, M, d, h->xrows, h->xn.out(tc_qkv, qkv_lo), st, k));
        mark(SP_STAGE_INPUT_NORM, 1);
        ++launches;
        mark(SP_STAGE_QKV, 0);
        s = h->gemm.run(wb, h->opt_gemm, h->xn, h->w_qkv, h->y, M, h->status, st, &launches, &ns, qkv_lo, 0,
                        nullptr, rp);
        mark(SP_STAGE_QKV, 1);
        if (s != SP_OK) return fail(s, "Q/K/V projection launch failed");
        yqkv = PartIn{h->y, ns, stride_qkv};
    } else if (d_rows) {
        mark(SP_STAGE_INPUT_NORM, 0);
        SP_CUDA(launch_rmsnorm_rows(wb, d_rows, 0, h->g_in, c.rms_eps, M, d, h->xn.out(tc_qkv, qkv_lo), st));
        mark(SP_STAGE_INPUT_NORM, 1);
        ++launches;
        mark(SP_STAGE_QKV, 0);
        s = h->gemm.run(wb, h->opt_gemm, h->xn, h->w_qkv, h->y, M, h->status, st, &launches, &ns, qkv_lo, 0,
                        nullptr, rp);
        mark(SP_STAGE_QKV, 1);
        if (s != SP_OK) return fail(s, "Q/K/V projection launch failed");
        yqkv = PartIn{h->y, ns, stride_qkv};
    }
    QkvRopeArgs r;
    memset(&r, 0, sizeof r);  // r0 = 0, kn_stride = 0 (= k): the parallel form
    r.k_task = h->k_task;     // positions L_b .. L_b + k_task - 1 in every task
    r.y = yqkv;
    r.shared = (d_rows || d_hidden) ? 0 : 1;
    r.B = batch; r.k = k; r.Hq = hq; r.Hkv = hkv; r.dh = dh;
    r.seq_ids = d_seq_ids; r.seq_lens = d_seq_lens; r.lens_by_batch = lens_by_batch;
    r.n_seqs = kv->n_seqs; r.max_seq_len = c.max_seq_len;
    r.rope_cs = h->rope_cs;
    r.q = h->q; r.k_new = h->k_new; r.v_new = h->v_new;
    r.status = h->status;
    // the attention's merge counters for this call's plan
    int split_tokens = 0, n_splits = 0;
    plan_attention(batch, hkv, k, c.max_seq_len, h->opt_split, h->n_sm, &split_tokens, &n_splits);
    r.zero_ints = attention_counters(h->attn_ws);
    r.n_zero = batch * hkv;
    if (!rope_fused) {
        mark(SP_STAGE_ROPE, 0);
        SP_CUDA(launch_qkv_rope(r, st));
        mark(SP_STAGE_ROPE, 1);
        ++launches;
    }

    // a3: attention over [cache ; new keys]
    AttnArgs a;
    memset(&a, 0, sizeof a);
    a.B = batch; a.Hq = hq; a.Hkv = hkv; a.dh = dh; a.k = k; a.G = G; a.R = G * k;
    a.k_task = h->k_task;  // each task's rows see only that task's new rows
    a.kv_bf16 = c.kv_dtype == SP_BF16;
    a.split_tokens = split_tokens;
    a.n_splits = n_splits;
    a.max_seq_len = c.max_seq_len;
    a.seq_ids = d_seq_ids; a.seq_lens = d_seq_lens; a.lens_by_batch = lens_by_batch;
    a.kv = to_dev(kv);
    a.q = h->q; a.k_new = h->k_new; a.v_new = h->v_new;
    a.status = h->status;
    a.gathered = nullptr;
    if (h->dbg_pages && kv->layout == SP_KV_PAGED) {
        if ((size_t)batch * kv->max_pages_per_seq > h->dbg_pages_cap)
            return fail(SP_ERR_INVALID_ARG, "gathered-pages buffer holds %zu ids, the call needs %zu",
                        h->dbg_pages_cap, (size_t)batch * kv->max_pages_per_seq);
        a.gathered = h->dbg_pages;
    }
    a.scale_log2 = (float)(1.4426950408889634 / sqrt((double)dh));
    a.tc_q_plain = q_plain;
    a.out = h->o.out(tc_o, proj_lo);
    if (tc_o) {  // the output projection's weights, prefetched by the attention's early finishers
        a.l2_next = h->w_o.ptr;
        a.l2_next_bytes = (size_t)d * hq * dh * h->es;
    }
    s = enqueue_attention(a, h->attn_ws, h->attn_ws_bytes, h->opt_attn, h->n_sm, h->opt_split,
                          &launches, st, true,
                          h->opt_profile ? h->ev[SP_STAGE_ATTN] : nullptr,
                          h->opt_profile ? h->ev[SP_STAGE_MERGE] : nullptr, h->opt_seg_cost,
                          h->opt_merge);
    if (s != SP_OK) return s;
    if (h->opt_profile) h->ev_used[SP_STAGE_ATTN] = h->ev_used[SP_STAGE_MERGE] = true;

    // a4: output projection + residual, post-norm
    const void *x = d_hidden ? (const void *)h->xrows : d_rows ? d_rows : h->soft_prompt;
    const int row_mod = (d_rows || d_hidden) ? 0 : k;
    const int x_bf16 = d_hidden ? 0 : wb;
    const int stall = h->opt_stall;  // one-shot: this call's output projection only
    h->opt_stall = 0;
    mark(SP_STAGE_O_PROJ, 0);
    s = h->gemm.run(wb, h->opt_gemm, h->o, h->w_o, h->y, M, h->status, st, &launches, &ns, proj_lo, stall);
    mark(SP_STAGE_O_PROJ, 1);
    if (s != SP_OK) return fail(s, "output projection launch failed");
    mark(SP_STAGE_POST_NORM, 0);
    SP_CUDA(launch_residual_norm(x_bf16, PartIn{h->y, ns, (size_t)M * d}, x, row_mod, h->g_post,
                                 c.rms_eps, M, d, h->h1, h->n.out(tc_gu, mlp_lo), st));
    mark(SP_STAGE_POST_NORM, 1);
    ++launches;
    // a5: gate/up + SwiGLU: in the projection's epilogue when it runs one CTA
    // per weight tile (no K split), else a separate kernel over the partials
    const ActOut a_out = h->a.out(tc_down, mlp_lo);
    const bool glu = h->gu_blk == 64 && h->gemm.glu_fusable(h->w_gu, h->n, h->opt_gemm, M, mlp_lo);
    mark(SP_STAGE_GATE_UP, 0);
    s = h->gemm.run(wb, h->opt_gemm, h->n, h->w_gu, h->y, M, h->status, st, &launches, &ns, mlp_lo, 0,
                    glu ? &a_out : nullptr);
    mark(SP_STAGE_GATE_UP, 1);
    if (s != SP_OK) return fail(s, "gate/up projection launch failed");
    if (!glu) {
        mark(SP_STAGE_SWIGLU, 0);
        SP_CUDA(launch_swiglu(PartIn{h->y, ns, (size_t)M * 2 * f}, M, f, h->gu_blk, a_out, st));
        mark(SP_STAGE_SWIGLU, 1);
        ++launches;
    }
    // a6-a7: down projection + residual, pooling, linear head
    mark(SP_STAGE_DOWN, 0);
    s = h->gemm.run(wb, h->opt_gemm, h->a, h->w_down, h->y, M, h->status, st, &launches, &ns, mlp_lo);
    mark(SP_STAGE_DOWN, 1);
    if (s != SP_OK) return fail(s, "down projection launch failed");
    mark(SP_STAGE_READOUT, 0);
    // one pooled readout per (sequence, task): rows [B][T][k_task][d]
    SP_CUDA(launch_readout(PartIn{h->y, ns, (size_t)M * d}, h->h1, h->head_w, h->head_b, c.pool,
                           batch * h->T, h->k_task, d, C, h->readout_part, d_logits, h->readout_cnt, st,
                           (size_t)h->k_task * d, (size_t)d, h->T, h->g_final, c.rms_eps));
    mark(SP_STAGE_READOUT, 1);
    ++launches;
    h->last_launches = launches;
    return SP_OK;
}

sp_status sp_classify(sp_handle *h, sp_stream stream, int batch, const int *d_seq_ids,
                      const int *d_seq_lens, const sp_kv_cache *kv, const void *d_rows,
                      float *d_logits) {
    return classify_impl(h, (cudaStream_t)stream, batch, d_seq_ids, d_seq_lens, 0, kv, d_rows,
                         d_logits);
}

sp_status sp_classify_host(sp_handle *h, sp_stream stream, int batch, const int *h_seq_ids,
                           const int *h_seq_lens, const sp_kv_cache *kv, const void *h_rows,
                           float *h_logits) {
    if (!h) return fail(SP_ERR_INVALID_ARG, "handle is NULL");
    const sp_config &c = h->cfg;
    if (batch < 1 || batch > c.max_batch)
        return fail(SP_ERR_INVALID_ARG, "batch %d outside 1..max_batch (%d)", batch, c.max_batch);
    if (!h_seq_lens || !h_logits) return fail(SP_ERR_INVALID_ARG, "seq_lens and logits are required");
    cudaStream_t st = (cudaStream_t)stream;
    if (h_seq_ids)
        SP_CUDA(cudaMemcpyAsync(h->stage_ids, h_seq_ids, batch * sizeof(int), cudaMemcpyHostToDevice, st));
    SP_CUDA(cudaMemcpyAsync(h->stage_lens, h_seq_lens, batch * sizeof(int), cudaMemcpyHostToDevice, st));
    if (h_rows)
        SP_CUDA(cudaMemcpyAsync(h->stage_rows, h_rows, (size_t)batch * c.k_rows * c.d_model * h->es,
                                cudaMemcpyHostToDevice, st));
    sp_status s = classify_impl(h, st, batch, h_seq_ids ? h->stage_ids : nullptr, h->stage_lens, 1,
                                kv, h_rows ? h->stage_rows : nullptr, h->stage_logits);
    if (s != SP_OK) return s;
    SP_CUDA(cudaMemcpyAsync(h_logits, h->stage_logits, (size_t)batch * h->T * c.n_classes * sizeof(float),
                            cudaMemcpyDeviceToHost, st));
    int bits = 0;
    return sp_check_status(h, stream, &bits);
}

sp_status sp_classify_hidden(sp_handle *h, sp_stream stream, int batch, const int *d_seq_ids,
                             const int *d_seq_lens, const sp_kv_cache *kv, const void *d_hidden,
                             float *d_logits) {
    if (!d_hidden) return fail(SP_ERR_INVALID_ARG, "d_hidden is NULL");
    return classify_impl(h, (cudaStream_t)stream, batch, d_seq_ids, d_seq_lens, 0, kv, nullptr,
                         d_logits, d_hidden);
}

sp_status sp_classify_hidden_host(sp_handle *h, sp_stream stream, int batch, const int *h_seq_ids,
                                  const int *h_seq_lens, const sp_kv_cache *kv,
                                  const void *h_hidden, float *h_logits) {
    if (!h) return fail(SP_ERR_INVALID_ARG, "handle is NULL");
    const sp_config &c = h->cfg;
    if (batch < 1 || batch > c.max_batch)
        return fail(SP_ERR_INVALID_ARG, "batch %d outside 1..max_batch (%d)", batch, c.max_batch);
    if (!h_seq_lens || !h_logits || !h_hidden)
        return fail(SP_ERR_INVALID_ARG, "seq_lens, hidden and logits are required");
    if (!h->fused) return fail(SP_ERR_INVALID_ARG, "the handle was created without input fusion (w_fc)");
    cudaStream_t st = (cudaStream_t)stream;
    if (h_seq_ids)
        SP_CUDA(cudaMemcpyAsync(h->stage_ids, h_seq_ids, batch * sizeof(int), cudaMemcpyHostToDevice, st));
    SP_CUDA(cudaMemcpyAsync(h->stage_lens, h_seq_lens, batch * sizeof(int), cudaMemcpyHostToDevice, st));
    SP_CUDA(cudaMemcpyAsync(h->stage_hidden, h_hidden, (size_t)batch * c.d_model * h->es,
                            cudaMemcpyHostToDevice, st));
    sp_status s = classify_impl(h, st, batch, h_seq_ids ? h->stage_ids : nullptr, h->stage_lens, 1,
                                kv, nullptr, h->stage_logits, h->stage_hidden);
    if (s != SP_OK) return s;
    SP_CUDA(cudaMemcpyAsync(h_logits, h->stage_logits, (size_t)batch * h->T * c.n_classes * sizeof(float),
                            cudaMemcpyDeviceToHost, st));
    int bits = 0;
    return sp_check_status(h, stream, &bits);
}

sp_status sp_check_status(sp_handle *h, sp_stream stream, int *bits) {
    if (!h) return fail(SP_ERR_INVALID_ARG, "handle is NULL");
    int v = 0;
    SP_CUDA(cudaStreamSynchronize((cudaStream_t)stream));
    SP_CUDA(cudaMemcpy(&v, h->status, sizeof(int), cudaMemcpyDeviceToHost));
    if (bits) *bits = v;
    if (v) {
        SP_CUDA(cudaMemset(h->status, 0, sizeof(int)));
        return fail(SP_ERR_DEVICE_STATUS, "device reported status bits 0x%x%s%s%s", v,
                    (v & SP_DEV_BAD_SEQ_ID) ? " (sequence id out of range)" : "",
                    (v & SP_DEV_BAD_LENGTH) ? " (cached length out of range)" : "",
                    (v & SP_DEV_BAD_PAGE) ? " (page id outside the pool)" : "");
    }
    return SP_OK;
}

size_t sp_attend_workspace_bytes(const sp_attn_dims *dm, int batch) {
    if (!dm || batch < 1 || dm->n_kv_heads < 1 || dm->n_q_heads % dm->n_kv_heads || dm->k_rows < 1 ||
        dm->k_rows > 32 || dm->max_seq_len < 0 || (dm->split_tokens % 64) || dm->split_tokens < 0)
        return 0;
    int split, ns;
    plan_attention(batch, dm->n_kv_heads, dm->k_rows, dm->max_seq_len, dm->split_tokens, sm_count(),
                   &split, &ns);
    return attention_workspace_bytes(batch, dm->n_kv_heads,
                                     (dm->n_q_heads / dm->n_kv_heads) * dm->k_rows, dm->head_dim, ns,
                                     sm_count());
}

sp_status sp_attend(sp_stream stream, const sp_attn_dims *dm, int batch, const int *d_seq_ids,
                    const int *d_seq_lens, const sp_kv_cache *kv, const float *d_q,
                    const float *d_k_new, const float *d_v_new, void *d_out, int out_dtype,
                    void *d_workspace, size_t workspace_bytes, int *d_status,
                    int *d_gathered_pages) {
    if (!dm) return fail(SP_ERR_INVALID_ARG, "dims is NULL");
    if (dm->n_kv_heads < 1 || dm->n_q_heads < 1 || dm->n_q_heads % dm->n_kv_heads)
        return fail(SP_ERR_INVALID_ARG, "n_q_heads must be a positive multiple of n_kv_heads");
    if (dm->head_dim != 32 && dm->head_dim != 64 && dm->head_dim != 128)
        return fail(SP_ERR_UNSUPPORTED, "head_dim %d unsupported", dm->head_dim);
    if (dm->k_rows < 1 || dm->k_rows > 32) return fail(SP_ERR_INVALID_ARG, "k_rows must be in 1..32");
    if (dm->kv_dtype != SP_F32 && dm->kv_dtype != SP_BF16) return fail(SP_ERR_INVALID_ARG, "bad kv_dtype");
    if (out_dtype != SP_F32 && out_dtype != SP_BF16) return fail(SP_ERR_INVALID_ARG, "bad out_dtype");
    if (dm->split_tokens < 0 || dm->split_tokens % 64)
        return fail(SP_ERR_INVALID_ARG, "split_tokens must be a multiple of 64");
    if (dm->max_seq_len < 0) return fail(SP_ERR_INVALID_ARG, "max_seq_len must be >= 0");
    if (batch < 1) return fail(SP_ERR_INVALID_ARG, "batch must be >= 1");
    if (!d_seq_lens || !d_q || !d_k_new || !d_v_new || !d_out || !d_workspace)
        return fail(SP_ERR_INVALID_ARG, "a required pointer is NULL");
    if (((uintptr_t)d_workspace) & 255) return fail(SP_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
    if ((((uintptr_t)d_q) | ((uintptr_t)d_k_new) | ((uintptr_t)d_v_new) | ((uintptr_t)d_out)) & 15)
        return fail(SP_ERR_INVALID_ARG, "queries, new keys/values and the output must be 16-byte aligned");
    sp_status s = check_kv(kv, dm->kv_dtype);
    if (s != SP_OK) return s;
    if (!d_seq_ids && batch > kv->n_seqs)
        return fail(SP_ERR_INVALID_ARG, "batch %d exceeds n_seqs %d with implicit ids", batch, kv->n_seqs);
    const int G = dm->n_q_heads / dm->n_kv_heads;
    if (G * dm->k_rows * dm->head_dim > 128 * 128)
        return fail(SP_ERR_UNSUPPORTED, "query group x k_rows x head_dim too large");
    AttnArgs a;
    memset(&a, 0, sizeof a);
    a.B = batch; a.Hq = dm->n_q_heads; a.Hkv = dm->n_kv_heads; a.dh = dm->head_dim;
    a.k = dm->k_rows; a.G = G; a.R = G * dm->k_rows;
    a.kv_bf16 = dm->kv_dtype == SP_BF16;
    plan_attention(batch, a.Hkv, a.k, dm->max_seq_len, dm->split_tokens, sm_count(), &a.split_tokens,
                   &a.n_splits);
    a.max_seq_len = dm->max_seq_len;
    a.seq_ids = d_seq_ids; a.seq_lens = d_seq_lens; a.lens_by_batch = 0;
    a.kv = to_dev(kv);
    a.q = d_q; a.k_new = d_k_new; a.v_new = d_v_new;
    a.status = d_status;
    a.gathered = d_gathered_pages;
    a.scale_log2 = (float)(1.4426950408889634 / sqrt((double)a.dh));
    a.out.f32 = out_dtype == SP_F32 ? (float *)d_out : nullptr;
    a.out.hi = out_dtype == SP_BF16 ? (bf16 *)d_out : nullptr;
    a.out.lo = nullptr;
    if (dm->path < 0 || dm->path > 2) return fail(SP_ERR_INVALID_ARG, "bad attention path");
    int launches = 0;
    return enqueue_attention(a, d_workspace, workspace_bytes, dm->path, sm_count(), dm->split_tokens,
                             &launches, (cudaStream_t)stream, false);
}

size_t sp_project_workspace_bytes(int M, int N, int K) {
    if (M < 1 || N < 1 || K < 1) return 0;
    const size_t planes = align256((size_t)M * K * 2 * sizeof(uint16_t));
    const int n_sm = sm_count();
    const TcPlan p = tc_plan(M, N, K, n_sm, (size_t)-1);
    return planes + align256((size_t)p.splits * M * N * sizeof(float));
}

sp_status sp_debug_gemm_plan(int M, int N, int K, int n_sm, int lo, int schedule,
                             size_t capacity_bytes, sp_gemm_plan *out) {
    if (M < 1 || N < 1 || K < 1 || n_sm < 1 || !out || (lo != 0 && lo != 1) || schedule < 0 ||
        schedule > 2)
        return fail(SP_ERR_INVALID_ARG, "bad plan query");
    if (!tc_supported(N, K)) return fail(SP_ERR_UNSUPPORTED, "no tensor path for N %d, K %d", N, K);
    const TcPlan p = tc_plan(M, N, K, n_sm, capacity_bytes, lo != 0, schedule);
    out->rows_per_tile = p.bn;
    out->m_tiles = p.m_tiles;
    out->n_tiles = p.n_tiles;
    out->n_kblocks = p.n_kb;
    out->tiles_per_cta = p.persistent ? 1 : p.nt;
    out->persistent = p.persistent ? 1 : 0;
    out->kblocks_per_cta = p.units_per_cta;
    out->splits = p.splits;
    out->grid = p.grid;
    return SP_OK;
}

sp_status sp_project(sp_stream stream, int M, int N, int K, const float *d_x, const void *d_w,
                     float *d_y, int path, void *d_workspace, size_t workspace_bytes) {
    if (M < 1 || N < 1 || K < 1) return fail(SP_ERR_INVALID_ARG, "M, N, K must be >= 1");
    if (!d_x || !d_w || !d_y) return fail(SP_ERR_INVALID_ARG, "a required pointer is NULL");
    if ((((uintptr_t)d_x) | ((uintptr_t)d_w)) & 15)
        return fail(SP_ERR_INVALID_ARG, "X and W must be 16-byte aligned");
    if (path < 0 || path > 2) return fail(SP_ERR_INVALID_ARG, "bad path");
    cudaStream_t st = (cudaStream_t)stream;
    const bool tc_ok = tc_supported(N, K);
    if (path == 2 && !tc_ok)
        return fail(SP_ERR_UNSUPPORTED, "tensor path needs N %% 128 == 0 and K %% 64 == 0");
    if (path == 1 || !tc_ok) {
        SP_CUDA(launch_gemm_simt(1, d_x, d_w, d_y, M, N, K, st));
        return SP_OK;
    }
    if (!d_workspace || ((uintptr_t)d_workspace & 255))
        return fail(SP_ERR_INVALID_ARG, "workspace must be non-NULL and 256-byte aligned");
    const size_t planes = align256((size_t)M * K * 2 * sizeof(uint16_t));
    if (workspace_bytes < planes + 256) return fail(SP_ERR_INVALID_ARG, "workspace too small");
    WeightMat w;
    init_weight(w, d_w, N, K, 1);
    ActBuf x;
    init_act(x, d_workspace, M, K, true);
    if (!w.tc || !x.maps) return fail(SP_ERR_CUDA, "tensor map encoding failed");
    float *part = (float *)((char *)d_workspace + planes);
    const TcPlan p = tc_plan(M, N, K, sm_count(), workspace_bytes - planes);
    SP_CUDA(launch_to_act(d_x, (size_t)M * K, x.out(true), st));
    const int bi = bn_index(p.bn);
    SP_CUDA(launch_gemm_tc(w.map, x.hi[bi], x.lo[bi], p, M, N, K, part, nullptr, st));
    SP_CUDA(launch_sum_partials(PartIn{part, p.splits, (size_t)M * N}, (size_t)M * N, d_y, st));
    return SP_OK;
}

}  // extern "C"
