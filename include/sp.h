/*
 * sp.h -- C ABI of the Speculative Probing classify path (libsp.so).
 *
 * Speculative Probing (Sec. 3.2) classifies a sequence by appending k learned
 * soft-prompt rows after it and running the frozen single decoder layer of the
 * speculative-decoding draft head (Sec. 3.1) over those rows.  Their attention
 * reads the sequence's keys/values already resident in the draft head's cache
 * (Sec. 3.3, Eq. 1-3); a linear head then reads class logits from the pooled
 * outputs (Sec. 3.2, "Classification head").  This library evaluates that path
 * on one GPU, in hand-written CUDA for sm_103a.
 *
 * Per row r = 0..k-1 of sequence b (cached length L_b, position L_b + r):
 *   x_hat = RMSNorm(x_r; g_in)
 *   q, k', v' = W_q x_hat, W_k x_hat, W_v x_hat; q, k' rotated at L_b + r
 *   o = softmax(q [K_cache ; k'_0..r]^T / sqrt(dh)) [V_cache ; v'_0..r]
 *   h1 = x_r + W_o o ;  n = RMSNorm(h1; g_post)
 *   h2_r = h1 + W_down (silu(W_gate n) * W_up n)
 * logits_b = W_head pool_r(h2_r) + head_b      (pool: mean over r, or r = k-1)
 * Query head h reads KV head h / (n_q_heads / n_kv_heads).  Rotation is the
 * rotate-half form: pair (i, i + dh/2) turns by (L_b + r) * theta^(-2i/dh).
 *
 * Conventions for every entry point:
 *  - Host pointers are named h_*, device pointers d_*; the stream argument is a
 *    cudaStream_t (NULL = the legacy default stream).
 *  - Calls that take a stream are asynchronous on it unless stated otherwise;
 *    they neither synchronise nor allocate.
 *  - Arguments are validated on the host before any launch; a rejected call
 *    returns SP_ERR_INVALID_ARG or SP_ERR_UNSUPPORTED and launches nothing.
 *  - Problems only the device can see (a sequence id or cached length out of
 *    range, a page id outside the pool) never fault: the kernels skip the bad
 *    access, treat it as masked, and set bits of a device status word that
 *    sp_check_status() returns as SP_ERR_DEVICE_STATUS.
 *  - sp_last_error() returns a per-thread description of the last failure.
 *  - The caches passed in are only read, never written (Sec. 3.3, "Monitoring
 *    does not disturb speculative decoding"): the k new keys/values go to
 *    library-owned scratch memory.
 */
#ifndef SP_H
#define SP_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define SP_API __attribute__((visibility("default")))
#else
#define SP_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef struct sp_handle sp_handle;
typedef struct CUstream_st *sp_stream; /* identical to cudaStream_t */

typedef enum sp_status {
    SP_OK = 0,
    SP_ERR_INVALID_ARG = 1,   /* bad pointer, size or enum; nothing launched        */
    SP_ERR_UNSUPPORTED = 2,   /* valid but not implemented (e.g. head_dim 96)       */
    SP_ERR_CUDA = 3,          /* a CUDA runtime/driver call failed                  */
    SP_ERR_OOM = 4,           /* device allocation failed in sp_create              */
    SP_ERR_DEVICE_STATUS = 5  /* the device reported bad ids/lengths/pages          */
} sp_status;

enum { SP_F32 = 0, SP_BF16 = 1 };              /* element types                  */
enum { SP_POOL_MEAN = 0, SP_POOL_LAST = 1 };   /* which outputs the head reads   */
enum { SP_KV_CONTIGUOUS = 0, SP_KV_PAGED = 1 };/* cache addressing               */

/* Device status bits (OR-ed together). */
enum {
    SP_DEV_BAD_SEQ_ID = 1,    /* a sequence id was outside [0, n_seqs)               */
    SP_DEV_BAD_LENGTH = 2,    /* a cached length was < 0 or > max_seq_len            */
    SP_DEV_BAD_PAGE = 4,      /* a page-table entry was outside [0, n_pages)         */
    SP_DEV_TIMEOUT = 8        /* a tensor-core kernel gave up waiting on a copy or an
                                 MMA (its outputs are invalid; the context is intact) */
};

/* Shapes of the frozen layer and of the probe (Sec. 3.1, 3.2). */
typedef struct sp_config {
    int d_model;      /* hidden size d; multiple of 8                                */
    int n_q_heads;    /* query heads Hq; a multiple of n_kv_heads                    */
    int n_kv_heads;   /* key/value heads Hkv (grouped-query attention)               */
    int head_dim;     /* dh: 32, 64 or 128                                           */
    int d_ff;         /* SwiGLU intermediate size; multiple of 8                     */
    int k_rows;       /* soft-prompt rows k appended per sequence, 1..32             */
    int n_classes;    /* C >= 1 rows of the linear head                              */
    float rope_theta; /* rotary base theta                                           */
    float rms_eps;    /* RMSNorm epsilon (added to the mean square)                  */
    int pool;         /* SP_POOL_MEAN or SP_POOL_LAST                                */
    int w_dtype;      /* SP_F32 or SP_BF16: layer matrices, soft prompt, input rows  */
    int kv_dtype;     /* SP_F32 or SP_BF16: cached keys/values                       */
    int max_batch;    /* largest batch passed to sp_classify (sizes the scratch)     */
    int max_seq_len;  /* largest cached length L_b (sizes the split plan)            */
    int n_tasks;      /* T probes sharing one pass over the cache (Sec. 3.3: several
                         classifiers with their own soft prompt and head on the same
                         draft-head KV cache); 0 or 1 = one task.  Task t's k rows sit
                         at positions L_b..L_b+k-1 and attend to the cache and to the
                         task's own new rows only; the soft prompt is [T][k][d], the
                         head [T][C][d] (+ bias [T][C]), per-sequence rows [B][T][k][d],
                         logits [B][T][C].  G * T * k <= 128 keeps the tensor-core
                         attention; recursive probing needs T = 1                  */
} sp_config;

/* Layer and probe parameters: HOST pointers, read once by sp_create and
 * copied to the device (the caller may free them afterwards).  Matrices are
 * row-major [out][in] in w_dtype (bf16 as raw 16-bit patterns):
 *   w_q [Hq*dh][d], w_k [Hkv*dh][d], w_v [Hkv*dh][d], w_o [d][Hq*dh],
 *   w_gate [d_ff][d], w_up [d_ff][d], w_down [d][d_ff],
 *   soft_prompt [k][d] (w_dtype), g_in [d], g_post [d] (float),
 *   head_w [C][d] (float), head_b [C] (float, may be NULL = zero bias).
 * Optional input fusion of an MTP draft layer (Sec. 3.1: the base model's
 * hidden state and the input embedding are RMS-normalised, concatenated and
 * projected by W_fc): w_fc [d][2d] (w_dtype; columns [0, d) act on the
 * normalised hidden state, [d, 2d) on the normalised embedding), g_h [d] and
 * g_e [d] (float) the two norm gains.  All three NULL: no fusion (then
 * sp_classify_hidden returns SP_ERR_INVALID_ARG).
 * Optional LM-head readout (Sec. 5 ablation, "Classification head": the frozen
 * lm_head read at label tokens such as yes/no): g_final [d] (float) is the
 * head's final RMSNorm gain, applied to the pooled state before head_w, whose
 * rows are then the label tokens' lm_head rows (logits[yes] - logits[no] is the
 * binary logit).  NULL = the plain linear head. */
typedef struct sp_weights {
    const void *w_q, *w_k, *w_v, *w_o, *w_gate, *w_up, *w_down;
    const float *g_in, *g_post;
    const void *soft_prompt;
    const float *head_w, *head_b;
    const void *w_fc;
    const float *g_h, *g_e;
    const float *g_final;
} sp_weights;

/* A resident key/value cache (Sec. 3.3): DEVICE pointers, borrowed for the
 * duration of the stream work of one call and never written.  Keys are stored
 * already rotated at their own positions 0..L_b-1.
 *  SP_KV_CONTIGUOUS: k_seq/v_seq are DEVICE arrays of n_seqs device pointers;
 *    sequence s is token-major [L_s][Hkv][dh] in kv_dtype.
 *  SP_KV_PAGED: k_pool/v_pool hold n_pages pages laid out
 *    [page][Hkv][page_size][dh]; page_table is a DEVICE int32 array
 *    [n_seqs][max_pages_per_seq]; token t of sequence s sits in page
 *    page_table[s][t / page_size], slot t % page_size.  Entries past
 *    ceil(L_s / page_size) are never read; a length that would need more than
 *    max_pages_per_seq pages is reported as SP_DEV_BAD_PAGE and the excess is
 *    masked.  page_size: 16, 32 or 64.
 *  A contiguous buffer must hold min(L_s, max_seq_len) tokens: its size is not
 *  known to the library, so a length beyond it cannot be detected.
 *  Every sequence pointer and both pools must be 16-byte aligned: the kernels
 *  copy 16-byte vectors.  The pools are checked on the host
 *  (SP_ERR_INVALID_ARG); the per-sequence pointers live in device memory and
 *  are the caller's to get right. */
typedef struct sp_kv_cache {
    int layout;
    const void *const *k_seq;
    const void *const *v_seq;
    const void *k_pool;
    const void *v_pool;
    const int *page_table;
    int page_size;
    int n_pages;
    int max_pages_per_seq;
    int n_seqs;
} sp_kv_cache;

/* Build a handle on the current CUDA device: validates the shapes, copies the
 * weights, precomputes the projections of the shared soft prompt and sizes all
 * scratch memory for cfg->max_batch.  The handle owns every device buffer it
 * allocates.  One handle serves one stream at a time (its scratch is shared by
 * consecutive calls).  Returns SP_OK and *out, or an error with *out = NULL. */
SP_API sp_status sp_create(const sp_config *cfg, const sp_weights *w, sp_handle **out);

/* Free a handle and everything it owns; waits for the device to go idle first.
 * NULL is accepted and ignored. */
SP_API sp_status sp_destroy(sp_handle *h);

/* The classify path (Sec. 3.2-3.3): logits for `batch` sequences of a resident
 * cache, enqueued on `stream`, no synchronisation, no allocation.
 *   d_seq_ids  [batch] int32 device: which cache sequences to classify
 *              (NULL: sequences 0..batch-1).
 *   d_seq_lens [kv->n_seqs] int32 device: cached length of every sequence;
 *              only the entries of the classified ids are read.
 *   kv         the cache (see sp_kv_cache); kv_dtype must match the handle.
 *   d_rows     [batch][k][d] device, w_dtype: the per-sequence input rows of
 *              the layer (e.g. an MTP head's fused inputs), or NULL: every
 *              sequence uses the handle's shared soft prompt rows.  Must be
 *              16-byte aligned (SP_ERR_INVALID_ARG otherwise).
 *   d_logits   [batch][C] float device, caller-owned: raw class logits.
 * 1 <= batch <= max_batch.  Device-side range problems are reported through
 * sp_check_status(). */
SP_API sp_status sp_classify(sp_handle *h, sp_stream stream, int batch, const int *d_seq_ids,
                      const int *d_seq_lens, const sp_kv_cache *kv, const void *d_rows,
                      float *d_logits);

/* sp_classify from HOST buffers: copies h_seq_ids [batch] (NULL = 0..batch-1),
 * h_seq_lens [batch] (the cached length of each classified sequence, in batch
 * order) and h_rows [batch][k][d] (NULL = shared prompt) to
 * handle-owned device staging, runs the path, copies the logits back to
 * h_logits [batch][C] and synchronises `stream`.  The cache stays on the
 * device.  Also returns any device status as SP_ERR_DEVICE_STATUS.  Pinned host
 * buffers make the copies asynchronous DMA transfers. */
SP_API sp_status sp_classify_host(sp_handle *h, sp_stream stream, int batch, const int *h_seq_ids,
                           const int *h_seq_lens, const sp_kv_cache *kv, const void *h_rows,
                           float *h_logits);

/* The classify path fed by base hidden states (Sec. 3.2, single-step probing:
 * the soft prompt replaces the next token's embedding in the MTP input): the
 * k input rows of sequence b are
 *   x_{b,r} = W_fc [RMSNorm(h_b; g_h) ; RMSNorm(soft_prompt_r; g_e)],  r < k,
 * evaluated in parallel at positions L_b..L_b+k-1 like sp_classify's rows.
 *   d_hidden [batch][d] device, w_dtype, 16-byte aligned: the base model's
 *            last hidden state of each classified sequence.
 * Other arguments as sp_classify.  The handle must have been created with
 * w_fc, g_h and g_e (SP_ERR_INVALID_ARG otherwise).  Enqueued on `stream`, no
 * synchronisation, no allocation. */
SP_API sp_status sp_classify_hidden(sp_handle *h, sp_stream stream, int batch,
                                    const int *d_seq_ids, const int *d_seq_lens,
                                    const sp_kv_cache *kv, const void *d_hidden, float *d_logits);

/* sp_classify_hidden from HOST buffers (ids, lengths as in sp_classify_host;
 * h_hidden [batch][d] w_dtype), logits copied back to h_logits; synchronises
 * `stream` and returns any device status as SP_ERR_DEVICE_STATUS. */
SP_API sp_status sp_classify_hidden_host(sp_handle *h, sp_stream stream, int batch,
                                         const int *h_seq_ids, const int *h_seq_lens,
                                         const sp_kv_cache *kv, const void *h_hidden,
                                         float *h_logits);

/* Synchronise `stream`, read and clear the handle's device status word.
 * Returns SP_OK, or SP_ERR_DEVICE_STATUS with the SP_DEV_* bits in *bits. */
SP_API sp_status sp_check_status(sp_handle *h, sp_stream stream, int *bits);

/* Per-thread text describing the last failure of any entry point. */
SP_API const char *sp_last_error(void);

/* Options (tests and benchmarks).  Returns SP_ERR_INVALID_ARG for an unknown
 * key or value. */
enum {
    SP_OPT_SPLIT_TOKENS = 1,  /* attention tokens per split-KV work unit (multiple
                                 of 64), 0 = automatic plan; a finer plan than
                                 sp_create sized for grows the handle's scratch
                                 here (the only allocation after sp_create)      */
    SP_OPT_GEMM_PATH = 2,     /* 0 = automatic, 1 = CUDA-core kernels only,
                                 2 = tensor-core kernels wherever supported       */
    SP_OPT_ATTN_PATH = 3,     /* 0 = automatic, 1 = CUDA-core kernel only,
                                 2 = tensor-core kernel wherever supported        */
    SP_OPT_PROFILE = 4,       /* 1 = record CUDA events around every stage of
                                 sp_classify on its stream (as external event
                                 nodes when the call is captured in a graph),
                                 0 = off (default)                              */
    SP_OPT_RECURSIVE = 5,     /* 1 = sp_classify_hidden runs recursive probing
                                 SP-k (Sec. 3.2): k steps of one row each, step i
                                 fusing step i-1's output with soft-prompt row i
                                 (no per-stage event markers); 0 = the parallel
                                 form (default)                                   */
    SP_OPT_ATTN_SEG_COST = 6, /* tensor-core attention: the cost of a segment
                                 boundary, in 64-token tiles, that the cuts
                                 between CTA shares balance (-1..1024); -1 = the
                                 built-in default (12 for paged caches, 28 for
                                 contiguous ones).  Changes the work split only,
                                 never the result beyond rounding order          */
    SP_OPT_ACT_PRECISION = 7, /* activations fed to the tensor-core
                                 projections: 0 = automatic (gate/up and down
                                 take plain bf16 when pool is SP_POOL_MEAN and
                                 at least 8 rows per task are pooled, else bf16
                                 hi + lo planes, ~16 mantissa bits; Q/K/V and
                                 output take hi + lo), 1 = hi + lo always, 2 =
                                 plain bf16 for gate/up and down, 3 = plain bf16
                                 always, 4 = plain bf16 except Q/K/V            */
    SP_OPT_DEBUG_STALL = 8,   /* test of the failure path: 1 = in the next
                                 sp_classify only, the first CTA of the output
                                 projection (when it runs on the one-CTA-per-tile
                                 schedule) never loads its first k-block, so its
                                 tensor-core wait runs out; that launch's waits
                                 give up after 1 ms, the kernel drains its copies,
                                 frees TMEM and returns, and sp_check_status
                                 reports SP_DEV_TIMEOUT (that call's logits are
                                 invalid, the handle stays usable).  Resets
                                 itself after that call                          */
    SP_OPT_GEMM_SCHEDULE = 9, /* tensor-core projections: 0 = automatic, 1 = one
                                 CTA per (weight tile, K split), 2 = persistent
                                 stream-K (one CTA per SM, an even share of the
                                 (tile, k-block) units each) wherever its partial
                                 planes fit the handle's scratch.  Changes the
                                 work split only, never the result beyond the
                                 order of the fp32 partial sums                 */
    SP_OPT_ATTN_MERGE = 10,   /* tensor-core attention: where the partials of a
                                 (sequence, kv head) split over several CTAs are
                                 merged: 0 = automatic, 1 = inside the attention
                                 kernel (by the CTA that completes the pair),
                                 2 = in a second kernel over (head, sequence,
                                 query row).  Both merge in segment order        */
    SP_OPT_QUERY_PRECISION = 11 /* tensor-core attention: queries as 0 =
                                 automatic (plain bf16 when pool is
                                 SP_POOL_MEAN and at least 16 rows per task are
                                 pooled, else hi + lo), 1 = bf16 hi + lo (two
                                 score MMAs per step), 2 = plain bf16 (one)     */
};

/* Stages of sp_classify, in launch order. */
enum {
    SP_STAGE_INPUT_NORM = 0,  /* a1: RMSNorm of per-sequence rows                    */
    SP_STAGE_QKV = 1,         /* a2: Q/K/V projection (skipped for the shared prompt) */
    SP_STAGE_ROPE = 2,        /* a2: rotation at L_b + r, new keys to scratch (not
                                 a stage of its own when the Q/K/V projection's
                                 epilogue rotates: reported as -1 then)           */
    SP_STAGE_ATTN = 3,        /* a3: split-KV attention over [cache ; new keys]      */
    SP_STAGE_MERGE = 4,       /* a3: log-sum-exp merge of the splits                 */
    SP_STAGE_O_PROJ = 5,      /* a4: output projection                               */
    SP_STAGE_POST_NORM = 6,   /* a4: residual + post-norm                            */
    SP_STAGE_GATE_UP = 7,     /* a5: gate/up projection                              */
    SP_STAGE_SWIGLU = 8,      /* a5: SwiGLU (-1 when the gate/up projection's
                                 epilogue applies it)                             */
    SP_STAGE_DOWN = 9,        /* a6: down projection                                 */
    SP_STAGE_READOUT = 10,    /* a6-a7: residual, pooling, linear head               */
    SP_STAGE_FUSION = 11,     /* input fusion: hidden-state norm and its W_fc
                                 projection (sp_classify_hidden only)             */
    SP_N_STAGES = 12
};

/* With SP_OPT_PROFILE on: synchronise on the last call's events and write the
 * device time (ms) of each stage of that call to ms[0..n-1] (-1 for a stage the
 * call did not run).  Returns SP_ERR_INVALID_ARG when profiling is off. */
SP_API sp_status sp_stage_times(sp_handle *h, float *ms, int n);
SP_API sp_status sp_set_option(sp_handle *h, int key, int value);

/* Number of kernel launches the last sp_classify enqueued. */
SP_API int sp_last_launch_count(const sp_handle *h);

/* Test hook: record the physical page ids the attention step of every later
 * sp_classify / sp_classify_hidden reads (paged caches only).  d_out is a
 * DEVICE int32 buffer of `capacity` entries, caller-owned, laid out
 * [batch][kv->max_pages_per_seq]: entry [i][j] receives the page id read for
 * logical page j of the i-th classified sequence (entries it did not read are
 * left untouched).  A call whose batch * max_pages_per_seq exceeds capacity
 * returns SP_ERR_INVALID_ARG before any launch.  d_out = NULL stops the
 * recording.  The ids let a test check the page-table walk bit-exactly (the
 * pages of sequence b are page_table[b][0 .. ceil(L_b / page_size))). */
SP_API sp_status sp_debug_gathered_pages(sp_handle *h, int *d_out, size_t capacity);

/* ------------------------------------------------------------------------- */
/* The attention step alone (Eq. 1-3), for step-level checks and for callers  */
/* that run their own projections.                                            */
/* ------------------------------------------------------------------------- */
typedef struct sp_attn_dims {
    int n_q_heads, n_kv_heads, head_dim; /* as in sp_config                         */
    int k_rows;                          /* query rows per sequence (k), 1..32      */
    int kv_dtype;                        /* SP_F32 or SP_BF16                       */
    int max_seq_len;                     /* bound on the cached lengths             */
    int split_tokens;                    /* tokens per split-KV work unit (multiple
                                            of 64), 0 = automatic plan              */
    int path;                            /* 0 = automatic, 1 = CUDA-core kernel,
                                            2 = tensor-core kernel (head_dim 128,
                                            bf16 cache, G * k <= 128; else
                                            SP_ERR_UNSUPPORTED)                     */
} sp_attn_dims;

/* Bytes of device scratch sp_attend needs for `batch` sequences (256-byte
 * aligned start required); 0 for invalid dims. */
SP_API size_t sp_attend_workspace_bytes(const sp_attn_dims *dims, int batch);

/* Attention of k rotated query rows per sequence over [cache ; new keys]:
 *   d_q     [batch][k][Hq][dh] float device (already rotated)
 *   d_k_new [batch][k][Hkv][dh] float device (already rotated), d_v_new same
 *   d_out   [batch][k][Hq][dh], float (out_dtype SP_F32) or bf16 (SP_BF16)
 * Row r of sequence b sees the L_b cached tokens and new tokens 0..r.
 * d_q, d_k_new, d_v_new and d_out must be 16-byte aligned (SP_ERR_INVALID_ARG
 * otherwise): the kernels move whole 16-byte vectors.
 * d_workspace: caller-allocated, >= sp_attend_workspace_bytes(dims, batch).
 * d_status: optional device int (OR-ed SP_DEV_* bits), NULL = not recorded.
 * d_gathered_pages: optional device int32 [batch][kv->max_pages_per_seq]
 *   (paged caches only): entry [i][j] receives the physical page id the kernel
 *   read for logical page j of the i-th sequence; entries it did not read are
 *   left untouched.  NULL = not recorded. */
SP_API sp_status sp_attend(sp_stream stream, const sp_attn_dims *dims, int batch, const int *d_seq_ids,
                    const int *d_seq_lens, const sp_kv_cache *kv, const float *d_q,
                    const float *d_k_new, const float *d_v_new, void *d_out, int out_dtype,
                    void *d_workspace, size_t workspace_bytes, int *d_status,
                    int *d_gathered_pages);

/* sp_attend for callers that cannot allocate device memory; the paper has no
 * counterpart to this entry point.  A monitor on the decoding hot path must not
 * call cudaMalloc (it can synchronise the device and stall decoding), and some
 * serving frameworks give a library no device memory of its own to allocate.
 * This call takes its split-KV scratch from a 32 MiB array inside the library
 * (a static device object that every GPU loading the library holds until the
 * process exits) and allocates nothing; the caller passes the same inputs and
 * outputs as to sp_attend, without a workspace.
 *  - A batch whose scratch (sp_attend_workspace_bytes) exceeds 32 MiB is
 *    rejected with SP_ERR_INVALID_ARG before any launch.
 *  - The first call on each device looks up the array's device address, with
 *    that device current, and caches it.  With lazy module loading (CUDA's
 *    default) that first call also loads the module holding the array, which
 *    commits its 32 MiB on the device: make the first call at set-up time,
 *    before any stream capture.  Later calls allocate nothing.  The cached
 *    address does not survive cudaDeviceReset.
 *  - Invalid dims or batch (those sp_attend_workspace_bytes rejects) return
 *    SP_ERR_INVALID_ARG.
 *  - Every call shares the one array and leaves its contents behind: calls
 *    whose work overlaps on the GPU (other streams, other threads) race on it
 *    and must be serialised by the caller.  Nothing in it needs clearing: each
 *    call writes every value it later reads. */
SP_API sp_status sp_attend_static(sp_stream stream, const sp_attn_dims *dims, int batch,
                                  const int *d_seq_ids, const int *d_seq_lens,
                                  const sp_kv_cache *kv, const float *d_q, const float *d_k_new,
                                  const float *d_v_new, void *d_out, int out_dtype, int *d_status,
                                  int *d_gathered_pages);

/* ------------------------------------------------------------------------- */
/* The projection step alone: one of the decoder layer's linear maps (Sec. 3.1)*/
/* ------------------------------------------------------------------------- */
/* Bytes of device scratch sp_project needs for an M x N x K product. */
SP_API size_t sp_project_workspace_bytes(int M, int N, int K);

/* Y[M][N] = X[M][K] W[N][K]^T with X and Y fp32 row-major and W bf16 row-major
 * [N][K] (raw 16-bit patterns), all DEVICE pointers (X, W 16-byte aligned,
 * SP_ERR_INVALID_ARG otherwise).
 * path: 1 = CUDA cores, 2 = tensor cores (needs N % 128 == 0 and K % 64 == 0;
 * SP_ERR_UNSUPPORTED otherwise), 0 = tensor cores when supported.  The tensor
 * path splits X into bf16 hi + lo parts and may split K across CTAs; both live
 * in d_workspace (>= sp_project_workspace_bytes, 256-byte aligned). */
/* Test hook, host only (needs no GPU): the launch plan of the tensor-core
 * projection y[M][N] = x[M][K] W^T on n_sm SMs, as sp_classify and sp_project
 * would choose it.  lo: 1 = hi + lo bf16 activation planes, 0 = plain bf16;
 * schedule: an SP_OPT_GEMM_SCHEDULE value (0 automatic, 1 tile kernel,
 * 2 persistent stream-K); capacity_bytes: room for fp32 partial planes
 * [splits][M][N] (SIZE_MAX: unbounded).  Fills *out; SP_ERR_INVALID_ARG for
 * M, N, K or n_sm < 1, a NULL out or a bad lo / schedule; SP_ERR_UNSUPPORTED
 * when the shape has no tensor path (N % 128 or K % 64 nonzero). */
typedef struct sp_gemm_plan {
    int rows_per_tile;   /* activation rows per tile (16, 32, 64, 128 or 256)  */
    int m_tiles;         /* ceil(M / rows_per_tile)                            */
    int n_tiles;         /* N / 128 weight tiles                               */
    int n_kblocks;       /* K / 64                                             */
    int tiles_per_cta;   /* tile kernel: 1, or 2 weight tiles sharing each
                            activation block                                   */
    int persistent;      /* 1: stream-K kernel over (tile, k-block) units      */
    int kblocks_per_cta; /* tile kernel: k-blocks per K split; persistent:
                            units per CTA                                      */
    int splits;          /* fp32 partial planes written                        */
    int grid;            /* CTAs launched                                      */
} sp_gemm_plan;
SP_API sp_status sp_debug_gemm_plan(int M, int N, int K, int n_sm, int lo, int schedule,
                                    size_t capacity_bytes, sp_gemm_plan *out);

SP_API sp_status sp_project(sp_stream stream, int M, int N, int K, const float *d_x,
                            const void *d_w, float *d_y, int path, void *d_workspace,
                            size_t workspace_bytes);

#ifdef __cplusplus
}
#endif
#endif /* SP_H */
