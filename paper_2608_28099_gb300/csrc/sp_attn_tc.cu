// Split-KV attention of the k appended rows over [cached ; new] keys
// (Sec. 3.3, Eq. 1-3) on tcgen05 tensor cores, for head_dim 128, bf16 caches
// and up to 128 query rows per (sequence, kv head).
//
// Work balance: the keys of every sequence b are cut into 64-token tiles, and
// the tiles of all sequences, in order, form one list of T tiles per kv head.
// The persistent grid holds n groups of Hkv CTAs (n Hkv <= SMs); CTA (j, g)
// attends kv head g over the equal share [j T / n, (j+1) T / n) of the list,
// whatever the mix of lengths, so a ragged batch keeps every SM streaming
// until the end, and the Hkv heads of a token range are read at the same time
// (a token's keys of all heads sit together in the cache: whole cache rows or
// pages are read while they are open).  A share crosses sequence boundaries:
// each piece of a sequence inside it is a segment.  A (sequence, kv head) pair
// that lies inside one share is finished there (normalised output); otherwise
// each of its segments leaves an unnormalised partial (max, sum, O) in slot
// (j + b) Hkv + g (unique: segments are ordered by both j and b), and the CTA
// that completes the pair's last segment (a counter per pair, zero before the
// launch) combines the partials in the exp2 domain, in segment order: in that
// segment's epilogue, or, when it is the last segment of the CTA's share (the
// usual case: such segments end with the kernel), after every role has
// finished, by all 384 threads, with the partials staged through the idle K/V
// ring in one round of copies.  The cuts between shares weigh every sequence
// start as a number of tiles (the cost of a segment boundary), so shares with
// more boundaries hold fewer tiles.
//
// All R = G * k query rows of the KV head's group share every K/V tile: the
// GQA group and the k soft-prompt rows together form the M side of the MMA.
// Per 64-token tile i of a segment (w = i & 1):
//   S_i   = Q K_i^T           M = 128 query rows, N = 64 tokens, K = 128 dims,
//                             Q held in TMEM (the MMA's A operand) as bf16 hi +
//                             lo (two MMAs per step) or, when the head pools at
//                             least 16 rows, plain bf16 (one), into TMEM buffer
//                             S_w
//   softmax                   warpgroup w (tiles alternate between two
//                             warpgroups), one query row per thread; a row's
//                             running max only moves when its max grows by
//                             more than 2^8, and O_w is rescaled in TMEM then
//   O_w  += P_i V_i           P written as bf16 over the first half of S_w (A
//                             operand from TMEM), V read in place from shared
//                             memory as an MN-major B operand
// At the end of a segment the two warpgroups swap their (max, sum) through
// shared memory; each then combines both O accumulators (they sit on the same
// TMEM lanes) over half of the columns, writes that half of the output or the
// partial, and loads half of the next segment's queries into TMEM.  The even and odd
// tiles form two independent pipelines, each with its own MMA issuing warp:
// one thread issuing small-N MMAs back to back leaves the tensor pipe idle
// between them, two keep it busy.
// Tiles come from a 6-stage ring that runs across segment boundaries (the K/V
// stream never drains): TMA for whole cache tiles of a paged pool (one box per
// (page, kv head) block of K and of V, issued by two lead warps taking
// alternate tiles), cp.async for contiguous caches, plain loads for the tile
// holding the sequence end and the new keys.  A page id outside the pool is
// never dereferenced: its block is zero-filled and the status word records it.
//
// Tile layout in shared memory (K and V alike, 64 tokens x 128 dims bf16):
// [8-token group][dim half][8 tokens][64 dims], 128-byte swizzle, so that a
// (page, head) block of 16/32/64 tokens is one TMA box and both MMAs read the
// tile with uniform strides (8-token groups 2048 B apart, dim halves 1024 B).
//
// Warps 0-3 and 4-7: the two softmax warpgroups (+ epilogue, merge); warps 8
// and 11: producers; warp 9: TMEM owner and MMA issuer of even tiles; warp 10:
// MMA issuer of odd tiles.  Softmax warps that own no query row (R <= 96)
// join the producers.  Every wait is time-limited (SP_DEV_TIMEOUT).
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
constexpr int KV_TILE = TT * DH * 2;           // K or V of one tile, 16 KB
constexpr int KV_STAGE = 2 * KV_TILE;          // K then V
constexpr uint32_t GROUP_STRIDE = 2048;        // 8-token groups
constexpr uint32_t HALF_STRIDE = 1024;         // 64-dim halves within a group
constexpr int MAX_B = 2048;                    // sequences per launch (tile prefix in smem)
constexpr int OFF_KV = 0;
constexpr int OFF_PREFIX = OFF_KV + STG * KV_STAGE;
constexpr int MAX_GRP = 256;                   // groups (cuts table in smem)
constexpr int OFF_CUTS = OFF_PREFIX + (MAX_B + 4) * 4;
constexpr int OFF_BAR = OFF_CUTS + (MAX_GRP + 4) * 4;
constexpr int OFF_ML = OFF_BAR + 512;           // both warpgroups' (max, sum) per row, 2 KB
// each sequence's cache id and length, resolved once at the start (the segment
// loops then make no global round trip for them)
constexpr int OFF_SEQ = OFF_ML + 2048;
// + 1 KB: the kernel rounds the dynamic shared window's start up to 1024 bytes
constexpr int SMEM_BYTES = OFF_SEQ + MAX_B * 8 + 1024;
constexpr int THREADS = 384;                   // 2 softmax warpgroups, 2 producers, 2 MMA
constexpr int PRODUCER_WARP = 8, MMA_WARP = 9, MMA_WARP1 = 10, PRODUCER_WARP1 = 11;
constexpr float RESCALE_LOG2 = 8.f;            // tolerate p <= 2^8 before rescaling O
constexpr int kStagedSegs = 4;                 // most partials merged through the idle ring
// TMEM columns: S0 [0,64) S1 [64,128) O0 [128,256) O1 [256,384) Qhi [384,448) Qlo [448,512)
// (Qlo unused with plain queries);
// P_w (64 bf16 per row) overwrites the first 32 columns of S_w once S_w is read.
constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t O_COL = 128, QHI_COL = 384, QLO_COL = 448;
// named barriers (id 0 is __syncthreads): the epilogue and the segment start,
// both over the softmax warps of the two warpgroups
constexpr int BAR_EPI = 1, BAR_SEG = 2;

static_assert(OFF_BAR % 16 == 0 && SMEM_BYTES <= 227 * 1024, "shared memory layout");

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

__device__ __forceinline__ void named_sync(int id, int n) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory");
}

struct Bars {
    uint64_t kv_full[STG], kv_empty[STG], s_full[2], p_full[2], pv_done[2], fin, q_full;  // fin: 2 arrivals
    uint32_t tmem;
    int abort;
    int merge_now;             // this segment completed its pair: merge it in the epilogue
    int fm_merge, fm_b, fm_nseg;  // the share's last segment completed its pair: merged at the end
    long long fm_slot0;           // partial slot of the pair's first segment
    int wsum[THREADS / 32];    // tile-prefix scan
};
static_assert(sizeof(Bars) <= 512, "barrier block");

// A CTA's piece of one sequence: tiles [t_a, t_a + n) of sequence b, which
// starts at tile xp of the list and has nt tiles.
struct Seg {
    int b, t_a, n, nt, xp;
};

// Segment holding tile x (x < x_end <= T), clipped at x_end.  prefix[b] is the
// first tile of sequence b; it grows strictly (every sequence has a tile for
// its new keys).
__device__ __forceinline__ Seg seg_at(const int *prefix, int B, int x, int x_end) {
    int lo = 0, hi = B - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (prefix[mid] <= x) lo = mid;
        else hi = mid - 1;
    }
    Seg s;
    s.b = lo;
    s.xp = prefix[lo];
    s.nt = prefix[lo + 1] - s.xp;
    s.t_a = x - s.xp;
    s.n = min(s.nt - s.t_a, x_end - x);
    return s;
}

// First tile of group j's share.  A segment boundary inside a share costs the
// consumers a pipeline drain, the epilogue and the next queries' load, worth
// about `c` tiles of streaming, so the shares balance tiles + c per sequence:
// every sequence b gets c virtual tiles in front of its own, the virtual list
// (T + c B long) is cut evenly, and a cut that lands in a sequence's virtual
// part moves to that sequence's first tile.  A cut within delta = min(share /
// 4, SNAP) tiles of a sequence start then moves onto it (a short piece of a
// sequence would pay a whole boundary).  c falls back to 0 when a share is
// shorter than c + 1 virtual tiles, which keeps the cuts strictly increasing
// (snapping moves them by at most a quarter share).  Evaluated once per group
// into a table (cuts[0..n]).
constexpr int SNAP = 4;
__device__ __forceinline__ int share_start(const int *prefix, int B, int T, int n, int j, int c) {
    if (j <= 0) return 0;
    if (j >= n) return T;
    if ((long long)T + (long long)c * B < (long long)n * (c + 1)) c = 0;
    const long long V = (long long)T + (long long)c * B;
    const long long v = (long long)j * V / n;
    int lo = 0, hi = B - 1;  // last sequence whose virtual start vpre(b) = prefix[b] + c b is <= v
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if ((long long)prefix[mid] + (long long)c * mid <= v) lo = mid;
        else hi = mid - 1;
    }
    const long long off = v - ((long long)prefix[lo] + (long long)c * lo);
    int x = off < c ? prefix[lo] : (int)min((long long)prefix[lo] + off - c, (long long)prefix[lo + 1] - 1);
    const int delta = min(T / n / 4, SNAP);
    if (delta == 0) return x;
    lo = 0, hi = B - 1;  // last sequence starting at or before x
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (prefix[mid] <= x) lo = mid;
        else hi = mid - 1;
    }
    const int c0 = prefix[lo], c1 = prefix[lo + 1];
    const int best = (x - c0 <= c1 - x) ? c0 : c1;
    return abs(best - x) <= delta ? best : x;
}

// Group whose share holds tile x (0 <= x < T): the largest j with cuts[j] <= x.
__device__ __forceinline__ int group_of(const int *cuts, int n, int x) {
    int lo = 0, hi = n - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (cuts[mid] <= x) lo = mid;
        else hi = mid - 1;
    }
    return lo;
}

__global__ void __launch_bounds__(THREADS, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap map_k,
                   const __grid_constant__ CUtensorMap map_v, AttnArgs a) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    Bars *bars = (Bars *)(smem + OFF_BAR);
    int *prefix = (int *)(smem + OFF_PREFIX);
    volatile int *abort = &bars->abort;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int R = a.R, k = a.k, B = a.B, Hkv = a.Hkv;
    const int kns = a.kn_stride ? a.kn_stride : k;  // rows per sequence of k_new / v_new
    const bool paged = a.kv.layout == SP_KV_PAGED;
    const int act_warps = (R + 31) / 32;  // softmax warps that own real query rows
    pdl_trigger();

    // ---- the tile list: prefix[b] = sum_{b' < b} ceil((L_b' + k) / TT).
    // Lengths and ids come from the caller, not from the previous kernel, so
    // this runs before pdl_wait.
    int2 *seqs = (int2 *)(smem + OFF_SEQ);  // (sid, len) of sequence b
    {
        const int per = (B + THREADS - 1) / THREADS;
        const int b0 = min(B, (int)threadIdx.x * per), b1 = min(B, b0 + per);
        int sum = 0;
        for (int bb = b0; bb < b1; ++bb) {
            const SeqRef sq = resolve_seq(a.seq_ids, a.seq_lens, a.lens_by_batch, bb, a.kv.n_seqs,
                                          a.max_seq_len, blockIdx.x == 0 ? a.status : nullptr);
            seqs[bb] = make_int2(sq.sid, sq.len);
            const int v = ceil_div(sq.len + a.r0 + k, TT);
            prefix[bb] = v;
            sum += v;
        }
        int incl = sum;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int v = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += v;
        }
        if (lane == 31) bars->wsum[warp] = incl;
        __syncthreads();
        int run = incl - sum;
        for (int w = 0; w < warp; ++w) run += bars->wsum[w];
        for (int bb = b0; bb < b1; ++bb) {
            const int v = prefix[bb];
            prefix[bb] = run;
            run += v;
        }
        if (threadIdx.x == 0) {
            int tot = 0;
            for (int w = 0; w < THREADS / 32; ++w) tot += bars->wsum[w];
            prefix[B] = tot;
        }
    }
    __syncthreads();
    const int T = prefix[B];
    const int n_grp = min((int)gridDim.x / Hkv, ceil_div(T, max(1, a.tc_min_tiles)));
    const int grp = blockIdx.x / Hkv, g = blockIdx.x - grp * Hkv;
    if (grp >= n_grp) {  // uniform over the CTA: no tile for this one
        if (threadIdx.x == 0 && a.l2_next)
            prefetch_l2_share(a.l2_next, a.l2_next_bytes, blockIdx.x, gridDim.x);
        return;
    }
    int *cuts = (int *)(smem + OFF_CUTS);
    for (int j = threadIdx.x; j <= n_grp; j += THREADS) cuts[j] = share_start(prefix, B, T, n_grp, j, a.tc_seg_cost);
    __syncthreads();
    const int x0 = cuts[grp], x1 = cuts[grp + 1];

    // producers: warps 8 and 11, plus the softmax warps that own no rows (they
    // help with the cp.async and plain-load tiles; warps 8 and 11 issue TMA)
    const int n_prod = 2 + 2 * (4 - act_warps);
    const bool is_producer = warp == PRODUCER_WARP || warp == PRODUCER_WARP1 ||
                             (warp < 8 && (warp & 3) >= act_warps);
    const int pidx = warp == PRODUCER_WARP    ? 0
                     : warp == PRODUCER_WARP1 ? 1
                                              : 2 + (warp >> 2) * (4 - act_warps) + ((warp & 3) - act_warps);
    const int n_cons = 64 * act_warps;  // softmax threads of both warpgroups

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
        bars->merge_now = 0;
        bars->fm_merge = 0;
        fence_mbar_init();
        if (paged) {
            prefetch_tmap(&map_k);
            prefetch_tmap(&map_v);
        }
    }
    if (warp == MMA_WARP) {
        tmem_alloc(&bars->tmem, TMEM_COLS);
        tmem_relinquish();
    }
    // No griddepcontrol.wait here: the cache, page table and lengths belong to the
    // caller, so the producers start streaming cache tiles while the previous
    // kernel (which writes the rotated queries and new keys) drains.  Every
    // thread that reads its output, or writes memory an earlier kernel may still
    // read, calls pdl_wait() first: producers before a tile with new keys, the
    // softmax warps before the first queries they load.
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = bars->tmem;
    const int P = a.kv.page_size;

    if (is_producer) {
        // ------------------------------------------------------------ producers
        const int ptid = pidx * 32 + lane, pstride = 32 * n_prod;
        const uint64_t pol_kv = policy_evict_first();
        const int npg = paged ? TT / P : 0;  // pages per tile
        int ci = 0;                          // CTA-local tile counter (ring position)
        int bad = 0;
        bool stop = false, waited = false;
        for (int x = x0; x < x1 && !stop;) {
            const Seg sg = seg_at(prefix, B, x, x1);
            x += sg.n;
            const int b = sg.b;
            const int2 sq2 = seqs[b];
            const SeqRef sq = {sq2.x, sq2.y};
            const int L = sq.len, total = L + a.r0 + k;
            const int *ptab = paged ? a.kv.page_table + (size_t)max(sq.sid, 0) * a.kv.max_pages : nullptr;
            for (int i = 0; i < sg.n; ++i, ++ci) {
                const int st = ci % STG;
                const int t0 = (sg.t_a + i) * TT;
                const bool lead = pidx == (ci & 1);
                const bool pure = t0 + TT <= L;  // cache tokens only (TMA when paged)
                // this tile's page ids, requested before the ring wait hides their latency
                int page = -1;
                const int lp = t0 / max(P, 1) + lane;
                if (pure && paged && lead && lane < npg) page = lp < a.kv.max_pages ? ptab[lp] : -1;
                // warp-uniform verdict: the lead warp's collectives below need every lane
                if (!__all_sync(0xffffffffu, mbar_wait(&bars->kv_empty[st], ((ci / STG) & 1) ^ 1, abort))) {
                    stop = true;
                    break;
                }
                uint8_t *K = smem + OFF_KV + st * KV_STAGE;
                uint8_t *V = K + KV_TILE;
                if (pure && paged) {
                    if (!lead) {
                        mbar_arrive(&bars->kv_full[st]);
                    } else {
                        // one TMA box per lane: lane = 2 * page + (K, V), each the
                        // (page, head) block of P tokens; a page outside the pool
                        // is zero-filled instead.  Lane 0 registers the stage's
                        // bytes before any box is issued.
                        const bool ok = lane < npg && page >= 0 && page < a.kv.n_pages;
                        const unsigned okm = __ballot_sync(0xffffffffu, ok);
                        if (ok && a.gathered) a.gathered[(size_t)b * a.kv.max_pages + lp] = page;
                        if (lane == 0)
                            mbar_arrive_expect_tx(&bars->kv_full[st], (uint32_t)__popc(okm) * 2u * P * DH * 2u);
                        __syncwarp();
                        const int j = (lane >> 1) & 3, part = lane & 1;
                        const int pj = __shfl_sync(0xffffffffu, page, j);
                        if (lane < 2 * npg && ((okm >> j) & 1)) {
                            const int grp = (pj * Hkv + g) * (P / 8);
                            // the cache is read once: evict-first keeps the queries and
                            // the partials of the merges resident in L2
                            tma_load_4d_hint((part ? V : K) + j * P * 256, part ? &map_v : &map_k,
                                             &bars->kv_full[st], 0, 0, 0, grp, pol_kv);
                        }
                        const unsigned want = (1u << npg) - 1u;
                        if ((okm & want) != want) {
                            bad = 1;
                            for (int jj = 0; jj < npg; ++jj) {
                                if ((okm >> jj) & 1) continue;
                                for (int e = lane; e < P * 16; e += 32) {
                                    st_shared_v4(K + jj * P * 256 + e * 16, 0, 0, 0, 0);
                                    st_shared_v4(V + jj * P * 256 + e * 16, 0, 0, 0, 0);
                                }
                            }
                            fence_proxy_async();
                        }
                        if (lane != 0) mbar_arrive(&bars->kv_full[st]);
                    }
                } else {
                    // cp.async tiles: cache rows (a contiguous cache, or the sequence-end
                    // tile of a paged one) copied 16 bytes at a time, the k new keys and
                    // values converted to bf16 through registers, rows past the end
                    // zero-filled.  This thread's arrival on kv_full fires when its
                    // copies have landed; the MMA warps fence the async proxy after
                    // their wait.
                    const int n_cache = max(0, min(TT, L - t0));             // rows [0, n_cache)
                    const int n_new = max(0, min(TT, total - t0)) - n_cache;  // then new keys
                    if (n_new > 0 && !waited) {
                        pdl_wait();  // the new keys come from the previous kernel
                        waited = true;
                    }
                    if (n_cache > 0 && paged) {
                        // this tile's page ids: lane j loads logical page t0 / P + j
                        int mine = -1;
                        if (lane < npg) {
                            const int lpt = t0 / P + lane;
                            mine = lpt < a.kv.max_pages ? ptab[lpt] : -1;
                            if (pidx == 0 && a.gathered && lane * P < n_cache && mine >= 0 &&
                                mine < a.kv.n_pages)
                                a.gathered[(size_t)b * a.kv.max_pages + lpt] = mine;
                        }
                        const int pg0 = __shfl_sync(0xffffffffu, mine, 0);
                        const int pg1 = __shfl_sync(0xffffffffu, mine, 1);
                        const int pg2 = __shfl_sync(0xffffffffu, mine, 2);
                        const int pg3 = __shfl_sync(0xffffffffu, mine, 3);
                        for (int idx = ptid; idx < n_cache * 16; idx += pstride) {
                            const int row = idx >> 4, c16 = idx & 15, q = row / P;
                            const uint32_t dst = kv_off(row, c16);
                            const int pg = q == 0 ? pg0 : q == 1 ? pg1 : q == 2 ? pg2 : pg3;
                            if (pg >= 0 && pg < a.kv.n_pages) {
                                const size_t o = (((size_t)pg * Hkv + g) * P + (t0 + row) % P) * DH + c16 * 8;
                                cp_async16(K + dst, (const bf16 *)a.kv.k_pool + o);
                                cp_async16(V + dst, (const bf16 *)a.kv.v_pool + o);
                            } else {
                                st_shared_v4(K + dst, 0, 0, 0, 0);
                                st_shared_v4(V + dst, 0, 0, 0, 0);
                                bad = 1;
                            }
                        }
                    } else if (n_cache > 0) {
                        // contiguous: token-major rows of 256 B
                        const bf16 *kb = (const bf16 *)a.kv.k_seq[sq.sid];
                        const bf16 *vb = (const bf16 *)a.kv.v_seq[sq.sid];
                        for (int idx = ptid; idx < n_cache * 16; idx += pstride) {
                            const int row = idx >> 4, c16 = idx & 15;
                            const size_t src = ((size_t)(t0 + row) * Hkv + g) * DH + c16 * 8;
                            const uint32_t dst = kv_off(row, c16);
                            cp_async16(K + dst, kb + src);
                            cp_async16(V + dst, vb + src);
                        }
                    }
                    // new keys/values [B][k][Hkv][dh] fp32: two chunks per thread in flight
                    for (int idx = ptid; idx < n_new * 16; idx += 2 * pstride) {
                        float4 kf[2][2], vf[2][2];
#pragma unroll
                        for (int u = 0; u < 2; ++u) {
                            const int j = idx + u * pstride;
                            if (j < n_new * 16) {
                                const int rr = (t0 + n_cache + (j >> 4)) - L, c16 = j & 15;
                                const size_t o = (((size_t)b * kns + rr) * Hkv + g) * DH + c16 * 8;
                                kf[u][0] = *(const float4 *)(a.k_new + o);
                                kf[u][1] = *(const float4 *)(a.k_new + o + 4);
                                vf[u][0] = *(const float4 *)(a.v_new + o);
                                vf[u][1] = *(const float4 *)(a.v_new + o + 4);
                            }
                        }
#pragma unroll
                        for (int u = 0; u < 2; ++u) {
                            const int j = idx + u * pstride;
                            if (j >= n_new * 16) continue;
                            const uint32_t dst = kv_off(n_cache + (j >> 4), j & 15);
                            st_shared_v4(K + dst, pack_bf16(kf[u][0].x, kf[u][0].y), pack_bf16(kf[u][0].z, kf[u][0].w),
                                         pack_bf16(kf[u][1].x, kf[u][1].y), pack_bf16(kf[u][1].z, kf[u][1].w));
                            st_shared_v4(V + dst, pack_bf16(vf[u][0].x, vf[u][0].y), pack_bf16(vf[u][0].z, vf[u][0].w),
                                         pack_bf16(vf[u][1].x, vf[u][1].y), pack_bf16(vf[u][1].z, vf[u][1].w));
                        }
                    }
                    const int n_fill = n_cache + n_new;
                    for (int idx = ptid; idx < (TT - n_fill) * 16; idx += pstride) {
                        const uint32_t dst = kv_off(n_fill + (idx >> 4), idx & 15);
                        st_shared_v4(K + dst, 0, 0, 0, 0);
                        st_shared_v4(V + dst, 0, 0, 0, 0);
                    }
                    fence_proxy_async();  // this thread's shared-memory stores
                    cp_async_mbar_arrive(&bars->kv_full[st]);
                }
            }
        }
        asm volatile("cp.async.wait_all;" ::: "memory");  // nothing lands after the CTA is gone
        if (pidx < 2 && lane == 0) {
            // drain TMA writes still in flight (only possible after an abort)
            for (int jd = ci > STG ? ci - STG : 0; jd < ci; ++jd)
                if ((jd & 1) == pidx) mbar_wait_drain(&bars->kv_full[jd % STG], (jd / STG) & 1);
        }
        bad = __any_sync(0xffffffffu, bad);
        if (bad && lane == 0 && a.status) atomicOr(a.status, SP_DEV_BAD_PAGE);
    } else if (warp == MMA_WARP || warp == MMA_WARP1) {
        // ------------------------------------------------------------ MMA issuers
        // Pipeline w = warp - MMA_WARP takes the tiles i = w, w + 2, ... of each
        // segment: S_w once the segment's queries are in TMEM, then per tile i:
        // PV_i (after softmax i) and S_{i+2} (reusing S buffer w).  PV_i does not
        // wait for any later tile's data, so stage i is released as soon as its
        // softmax is done.
        const int w = warp - MMA_WARP;
        if (lane == 0) {
            constexpr uint32_t idesc_s = idesc_bf16_f32(128, TT);
            constexpr uint32_t idesc_o = idesc_bf16_f32_bmn(128, DH);
            const uint32_t s_tmem = tmem + (uint32_t)(w * TT);  // S_w; P_w over its first half
            const uint32_t o_tmem = tmem + O_COL + (uint32_t)(w * DH);
            auto issue_s = [&](int cst) {
                const uint8_t *K = smem + OFF_KV + cst * KV_STAGE;
#pragma unroll
                for (int kk = 0; kk < DH / 16; ++kk) {
                    // 16 dims = 32 B along a 128-byte row of dim half kk / 4
                    const uint64_t bk =
                        sw128_kmajor_desc_sbo(K + (kk >> 2) * HALF_STRIDE, GROUP_STRIDE) +
                        (uint64_t)((kk & 3) * 2);
                    // 16 dims of Q = 8 TMEM columns
                    mma_bf16_ts(s_tmem, tmem + QHI_COL + (uint32_t)(kk * 8), bk, idesc_s,
                                kk > 0 ? 1u : 0u);
                    if (!a.tc_q_plain)
                        mma_bf16_ts(s_tmem, tmem + QLO_COL + (uint32_t)(kk * 8), bk, idesc_s, 1u);
                }
                mma_commit(&bars->s_full[w]);
            };
            bool ok = true;
            int ci0 = 0, kw = 0, j = 0;
            for (int x = x0; ok && x < x1; ++j) {
                const Seg sg = seg_at(prefix, B, x, x1);
                x += sg.n;
                if (!mbar_wait(&bars->q_full, (uint32_t)(j & 1), abort)) break;
                tc_fence_after();
                if (w < sg.n) {
                    const int cw = ci0 + w;
                    ok = mbar_wait(&bars->kv_full[cw % STG], (cw / STG) & 1, abort);
                    if (ok) {
                        tc_fence_after();
                        fence_proxy_async();  // cp.async data -> tensor-core reads
                        issue_s(cw % STG);
                    }
                }
                for (int i = w; ok && i < sg.n; i += 2, ++kw) {
                    if (!mbar_wait(&bars->p_full[w], (uint32_t)(kw & 1), abort)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const int cst = (ci0 + i) % STG;
                    const uint8_t *V = smem + OFF_KV + cst * KV_STAGE + KV_TILE;
#pragma unroll
                    for (int kk = 0; kk < TT / 16; ++kk) {
                        // 16 tokens of P = 8 TMEM columns; 16 tokens of V = two 8-token groups
                        mma_bf16_ts(o_tmem, s_tmem + (uint32_t)(kk * 8),
                                    sw128_mnmajor_desc2(V + kk * 2 * GROUP_STRIDE, HALF_STRIDE, GROUP_STRIDE),
                                    idesc_o, (i >= 2 || kk > 0) ? 1u : 0u);
                    }
                    mma_commit(&bars->kv_empty[cst]);
                    mma_commit(&bars->pv_done[w]);
                    if (i + 2 < sg.n) {
                        // S buffer w is free: softmax i has read it (p_full above)
                        const int cn = ci0 + i + 2;
                        if (!mbar_wait(&bars->kv_full[cn % STG], (cn / STG) & 1, abort)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        fence_proxy_async();  // cp.async data -> tensor-core reads
                        issue_s(cn % STG);
                    }
                }
                ci0 += sg.n;
            }
            mma_commit(&bars->fin);  // completes when every MMA of this issuer is done
        }
        __syncwarp();
    } else if (warp < 8 && (warp & 3) < act_warps) {
        // ------------------------------------------------------------ softmax + epilogue
        const int wg = warp >> 2;           // warpgroup: tiles i with (i & 1) == wg
        const int row = threadIdx.x & 127;  // == TMEM lane
        const int ct = wg * 32 * act_warps + (warp & 3) * 32 + lane;  // 0 .. n_cons-1
        const bool active = row < R;
        const int r_soft = row % k;
        const uint32_t lane_base = tmem + ((uint32_t)((warp & 3) * 32) << 16);
        const uint32_t s_col = (uint32_t)(wg * TT), o_col = O_COL + (uint32_t)(wg * DH);
        float *sm_ml = (float *)(smem + OFF_ML);
        // The queries of sequence b for kv head g -> bf16 hi/lo in TMEM (row rr =
        // hl*k + r on lane rr; zero past R), scaled to log2 units.  Warpgroup wg
        // converts dims [64 wg, 64 wg + 64): TMEM columns [32 wg, 32 wg + 32) of
        // the hi and of the lo block (two bf16 per column).  Both warpgroups'
        // warps w and w + 4 reach the same TMEM lanes.
        auto load_q = [&](int b) {
            const float4 *src = nullptr;
            if (active) {
                const int hl = row / k, r = row - hl * k;
                src = (const float4 *)(a.q + (((size_t)b * k + r) * a.Hq + g * a.G + hl) * DH) + wg * 16;
            }
            uint32_t hi[32], lo[32];
            float4 xs[16];
#pragma unroll
            for (int c4 = 0; c4 < 16; ++c4) xs[c4] = src ? src[c4] : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
            for (int c4 = 0; c4 < 16; ++c4) {
                const float v[4] = {xs[c4].x * a.scale_log2, xs[c4].y * a.scale_log2,
                                    xs[c4].z * a.scale_log2, xs[c4].w * a.scale_log2};
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
            tmem_st32u(lane_base + QHI_COL + wg * 32, hi);
            if (!a.tc_q_plain) tmem_st32u(lane_base + QLO_COL + wg * 32, lo);
            tc_fence_before();
        };
        pdl_wait();  // the rotated queries come from the previous kernel
        load_q(seg_at(prefix, B, x0, x1).b);
        bool ok = true;
        int k0 = 0, k1 = 0;  // tiles done so far by pipeline 0 / 1 (barrier phases)
        for (int x = x0; x < x1;) {
            const int xs = x;  // segment start (its other fields are recomputed after the tiles)
            int n_tiles, lim_rel, lo_rel, new_rel;
            {
                const Seg sg = seg_at(prefix, B, x, x1);
                n_tiles = sg.n;
                const int2 sq2 = seqs[sg.b];
                const SeqRef sq = {sq2.x, sq2.y};
                // this row sees tokens t < L + r0 + r + 1 except the new rows of
                // other tasks before its own, [L, L + lo); relative to the segment start:
                lim_rel = sq.len + a.r0 + r_soft + 1 - sg.t_a * TT;
                lo_rel = sq.len + (a.k_task ? (r_soft / a.k_task) * a.k_task : 0) - sg.t_a * TT;
                new_rel = sq.len - sg.t_a * TT;
            }
            x += n_tiles;
            // this segment's queries are written, and the previous epilogue is complete
            named_sync(BAR_SEG, n_cons);
            if (ct == 0) mbar_arrive(&bars->q_full);

            float m = -INFINITY, l = 0.f;
            int kw = wg ? k1 : k0;
            for (int i = wg; ok && i < n_tiles; i += 2, ++kw) {
                // warp-uniform verdicts: the TMEM loads and stores are warp-collective
                if (!__all_sync(0xffffffffu, mbar_wait(&bars->s_full[wg], (uint32_t)(kw & 1), abort))) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                float sv[TT];
                {
                    float t32[32];
                    tmem_ld32(lane_base + s_col, t32);
#pragma unroll
                    for (int jj = 0; jj < 32; ++jj) sv[jj] = t32[jj];
                    tmem_ld32(lane_base + s_col + 32, t32);
#pragma unroll
                    for (int jj = 0; jj < 32; ++jj) sv[32 + jj] = t32[jj];
                }
                const int t0 = i * TT;  // relative to the segment start
                if (t0 + TT > new_rel) {  // the tile holds new rows: causal and task masks
#pragma unroll
                    for (int jj = 0; jj < TT; ++jj) {
                        const int t = t0 + jj;
                        if (t >= lim_rel || (t >= new_rel && t < lo_rel)) sv[jj] = -INFINITY;
                    }
                }
                // tile max as an 8-way tree
                float mx[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) mx[e] = fmaxf(sv[e], sv[e + 8]);
#pragma unroll
                for (int jj = 16; jj < TT; jj += 8)
#pragma unroll
                    for (int e = 0; e < 8; ++e) mx[e] = fmaxf(mx[e], sv[jj + e]);
                const float mt = fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])),
                                       fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7])));
                const bool grow = active && (mt > m + RESCALE_LOG2 || (m == -INFINITY && mt != -INFINITY));
                const float m_new = grow ? mt : m;
                const float alpha = grow ? (m == -INFINITY ? 0.f : fast_exp2(m - m_new)) : 1.f;
                // O_wg and P_wg were last used by PV of this pipeline's previous tile
                if (i >= 2) {
                    if (!__all_sync(0xffffffffu, mbar_wait(&bars->pv_done[wg], (uint32_t)((kw - 1) & 1), abort))) {
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
                            for (int jj = 0; jj < 32; ++jj) o32[jj] *= alpha;
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
                for (int jj = 0; jj < TT; jj += 2) {
                    const float p0 = fast_exp2(sv[jj] - mu);
                    const float p1 = fast_exp2(sv[jj + 1] - mu);
                    ps[(jj >> 1) & 7] += p0 + p1;
                    pk[jj >> 1] = pack_bf16(p0, p1);
                }
                l += ((ps[0] + ps[1]) + (ps[2] + ps[3])) + ((ps[4] + ps[5]) + (ps[6] + ps[7]));
                tmem_st32u(lane_base + s_col, pk);  // P_i over the first half of S_i
                tc_fence_before();
                mbar_arrive(&bars->p_full[wg]);
            }
            const int n0 = (n_tiles + 1) >> 1, n1 = n_tiles >> 1;  // tiles of pipeline 0 / 1
            k0 += n0;
            k1 += n1;

            // ---- epilogue, shared by the two warpgroups: each hands its (max, sum)
            // to the other through shared memory, combines (max, sum, O) of both
            // pipelines over its half of the columns, writes the pair's output
            // (whole pair in this CTA's share) or this segment's partial, and loads
            // its half of the next segment's queries
            const Seg sg = seg_at(prefix, B, xs, x1);
            const int b = sg.b;
            const int j_first = group_of(cuts, n_grp, sg.xp);
            const int j_last = group_of(cuts, n_grp, sg.xp + sg.nt - 1);
            const bool whole = j_first == j_last;
            const bool mine = wg == 0 || n1 > 0;  // pipeline 0 has >= 1 tile, pipeline 1 may have none
            sm_ml[wg * 256 + row] = mine ? m : -INFINITY;
            sm_ml[wg * 256 + 128 + row] = mine ? l : 0.f;
            // both warpgroups are past their last S of the segment: Q may be rewritten
            named_sync(BAR_EPI, n_cons);
            const float m0 = sm_ml[row], l0 = sm_ml[128 + row];
            const float m1 = sm_ml[256 + row], l1 = sm_ml[384 + row];
            const float mc = fmaxf(m0, m1);
            const float a0 = (m0 == -INFINITY) ? 0.f : fast_exp2(m0 - mc);
            const float a1 = (m1 == -INFINITY) ? 0.f : fast_exp2(m1 - mc);
            const float lsum = a0 * l0 + a1 * l1;
            bool have = ok && mbar_wait(&bars->pv_done[0], (uint32_t)((k0 - 1) & 1), abort);
            if (have && n1 > 0) have = mbar_wait(&bars->pv_done[1], (uint32_t)((k1 - 1) & 1), abort);
            have = __all_sync(0xffffffffu, have);  // the TMEM loads below are warp-collective
            if (!have) ok = false;
            const size_t slot = ((size_t)grp + b) * Hkv + g;
            float *po = a.part_o + (slot * R + row) * DH;
            const float inv = lsum > 0.f ? 1.f / lsum : 0.f;
            const int hl = row / k, r = row - hl * k;
            const size_t out0 = (((size_t)b * k + r) * a.Hq + g * a.G + hl) * DH;
            if (have) {
                tc_fence_after();
#pragma unroll 1
                for (int c0 = wg * (DH / 2); c0 < (wg + 1) * (DH / 2); c0 += 32) {
                    float o0[32], o1[32];
                    tmem_ld32(lane_base + O_COL + c0, o0);
                    if (n1 > 0) {
                        tmem_ld32(lane_base + O_COL + DH + c0, o1);
                    } else {
#pragma unroll
                        for (int jj = 0; jj < 32; ++jj) o1[jj] = 0.f;
                    }
                    if (active && whole) {
#pragma unroll
                        for (int jj = 0; jj < 32; jj += 4)
                            act_store4(a.out, out0 + c0 + jj,
                                       make_float4((a0 * o0[jj] + a1 * o1[jj]) * inv,
                                                   (a0 * o0[jj + 1] + a1 * o1[jj + 1]) * inv,
                                                   (a0 * o0[jj + 2] + a1 * o1[jj + 2]) * inv,
                                                   (a0 * o0[jj + 3] + a1 * o1[jj + 3]) * inv));
                    } else if (active) {
#pragma unroll
                        for (int jj = 0; jj < 32; jj += 4)
                            *(float4 *)(po + c0 + jj) =
                                make_float4(a0 * o0[jj] + a1 * o1[jj], a0 * o0[jj + 1] + a1 * o1[jj + 1],
                                            a0 * o0[jj + 2] + a1 * o1[jj + 2],
                                            a0 * o0[jj + 3] + a1 * o1[jj + 3]);
                    }
                }
                if (active && !whole && wg == 0) {
                    a.part_ml[(slot * R + row) * 2] = mc;
                    a.part_ml[(slot * R + row) * 2 + 1] = lsum;
                }
            }
            if (!whole && !a.tc_merge_kernel) {
                // count this segment; the one completing the pair merges all of its
                // partials here, in segment order (the result does not depend on
                // which CTA finishes last), while its own are still in L2
                const int n_seg = j_last - j_first + 1;
                const int staged_max = min(kStagedSegs, (STG * KV_STAGE) / (R * (DH * 4 + 8)));
                __threadfence();  // this segment's partial is visible before it is counted
                named_sync(BAR_EPI, n_cons);
                if (ct == 0) {
                    const int done_before = atomicAdd(a.counters + b * Hkv + g, 1);
                    const int last = done_before == n_seg - 1;
                    if (last) a.counters[b * Hkv + g] = 0;  // ready for the next launch
                    bars->merge_now = last;
                }
                named_sync(BAR_EPI, n_cons);
                const size_t slot0 = ((size_t)j_first + b) * Hkv + g;  // segment e: + e Hkv
                if (bars->merge_now && x >= x1 && n_seg <= staged_max) {
                    // the share's last segment: merged by the whole CTA once every
                    // role is done (below), through the idle K/V ring
                    if (ct == 0) {
                        bars->fm_b = b;
                        bars->fm_nseg = n_seg;
                        bars->fm_slot0 = (long long)slot0;
                        bars->fm_merge = 1;
                    }
                } else if (bars->merge_now && have && active) {
                    __threadfence();  // the other segments' partials are read after their count
#pragma unroll 1
                    for (int c0 = wg * (DH / 2); c0 < (wg + 1) * (DH / 2); c0 += 32) {
                        float acc[32], mm = -INFINITY, ll = 0.f;
#pragma unroll
                        for (int jj = 0; jj < 32; ++jj) acc[jj] = 0.f;
                        for (int e0 = 0; e0 < n_seg; e0 += 2) {
                            float2 ml[2];
                            float4 ov[2][8];
#pragma unroll
                            for (int e = 0; e < 2; ++e) {  // both segments' loads in flight together
                                const bool in = e0 + e < n_seg;
                                const size_t sl = slot0 + (size_t)(e0 + e) * Hkv;
                                ml[e] = in ? __ldcg((const float2 *)(a.part_ml + (sl * R + row) * 2))
                                           : make_float2(-INFINITY, 0.f);
                                const float4 *src = (const float4 *)(a.part_o + (sl * R + row) * DH + c0);
#pragma unroll
                                for (int q4 = 0; q4 < 8; ++q4)
                                    ov[e][q4] = in ? __ldcg(src + q4) : make_float4(0.f, 0.f, 0.f, 0.f);
                            }
#pragma unroll
                            for (int e = 0; e < 2; ++e) {
                                const float mn = fmaxf(mm, ml[e].x);
                                if (mn == -INFINITY) continue;
                                const float al = mm == -INFINITY ? 0.f : exp2f(mm - mn);
                                const float wt = ml[e].x == -INFINITY ? 0.f : exp2f(ml[e].x - mn);
                                ll = ll * al + wt * ml[e].y;
#pragma unroll
                                for (int q4 = 0; q4 < 8; ++q4) {
                                    acc[4 * q4] = acc[4 * q4] * al + wt * ov[e][q4].x;
                                    acc[4 * q4 + 1] = acc[4 * q4 + 1] * al + wt * ov[e][q4].y;
                                    acc[4 * q4 + 2] = acc[4 * q4 + 2] * al + wt * ov[e][q4].z;
                                    acc[4 * q4 + 3] = acc[4 * q4 + 3] * al + wt * ov[e][q4].w;
                                }
                                mm = mn;
                            }
                        }
                        const float il = ll > 0.f ? 1.f / ll : 0.f;
#pragma unroll
                        for (int jj = 0; jj < 32; jj += 4)
                            act_store4(a.out, out0 + c0 + jj,
                                       make_float4(acc[jj] * il, acc[jj + 1] * il, acc[jj + 2] * il,
                                                   acc[jj + 3] * il));
                    }
                }
            }
            if (x < x1) load_q(seg_at(prefix, B, x, x1).b);
        }
    }
    // every MMA must be finished before TMEM and shared memory go away
    mbar_wait_drain(&bars->fin, 0);
    tc_fence_before();
    __syncthreads();
    if (threadIdx.x == 0 && *abort && a.status) atomicOr(a.status, SP_DEV_TIMEOUT);
    if (bars->fm_merge) {
        // Merge of the pair completed by this share's last segment, by all 384
        // threads: every partial of the pair lands in the idle K/V ring in one
        // round of cp.async copies (O of segment e as [e][row][dh], then (max,
        // sum) as [e][row]), then thread (row, c) combines 16-byte units c, c + 8,
        // c + 16, c + 24 of its row in segment order, in the arithmetic of the
        // register merge above, so the bits do not depend on which path ran.
        // Shared-memory reads are conflict-free and eight lanes store 64
        // contiguous bytes per plane.  Loads through registers would need a
        // dependent round trip per two segments, each waiting behind the other
        // SMs' cache streams.
        const int b = bars->fm_b, n_seg = bars->fm_nseg;
        const size_t slot0 = (size_t)bars->fm_slot0;
        const bool good = !*abort;  // every wait is over: uniform
        __threadfence();            // the other segments' partials are read after their count
        uint8_t *stage = smem + OFF_KV;
        float2 *st_ml = (float2 *)(stage + (size_t)n_seg * R * DH * 4);
        const int units = R * (DH / 4);  // 16-byte units of one segment's O
        for (int idx = threadIdx.x; idx < n_seg * units; idx += THREADS) {
            const int e = idx / units, rem = idx - e * units;
            cp_async16(stage + (size_t)idx * 16, a.part_o + (slot0 + (size_t)e * Hkv) * R * DH + (size_t)rem * 4);
        }
        for (int idx = threadIdx.x; idx < n_seg * R; idx += THREADS) {
            const int e = idx / R, rr = idx - e * R;
            st_ml[idx] = __ldcg((const float2 *)(a.part_ml + ((slot0 + (size_t)e * Hkv) * R + rr) * 2));
        }
        asm volatile("cp.async.wait_all;" ::: "memory");
        __syncthreads();
        if (good) {
            for (int item = threadIdx.x; item < R * 8; item += THREADS) {
                const int rr = item >> 3, c = item & 7;
                float2 ml[kStagedSegs];
                float4 ov[kStagedSegs][4];
#pragma unroll
                for (int e = 0; e < kStagedSegs; ++e) {
                    const int ee = min(e, n_seg - 1);
                    ml[e] = st_ml[ee * R + rr];
#pragma unroll
                    for (int q = 0; q < 4; ++q)
                        ov[e][q] = ld_shared_v4f(stage + (((size_t)ee * R + rr) * (DH / 4) + c + 8 * q) * 16);
                }
                float acc[16], mm = -INFINITY, ll = 0.f;
#pragma unroll
                for (int j = 0; j < 16; ++j) acc[j] = 0.f;
#pragma unroll
                for (int e = 0; e < kStagedSegs; ++e) {
                    if (e >= n_seg) break;
                    const float mn = fmaxf(mm, ml[e].x);
                    if (mn == -INFINITY) continue;
                    const float al = mm == -INFINITY ? 0.f : exp2f(mm - mn);
                    const float wt = ml[e].x == -INFINITY ? 0.f : exp2f(ml[e].x - mn);
                    ll = ll * al + wt * ml[e].y;
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        acc[4 * q] = acc[4 * q] * al + wt * ov[e][q].x;
                        acc[4 * q + 1] = acc[4 * q + 1] * al + wt * ov[e][q].y;
                        acc[4 * q + 2] = acc[4 * q + 2] * al + wt * ov[e][q].z;
                        acc[4 * q + 3] = acc[4 * q + 3] * al + wt * ov[e][q].w;
                    }
                    mm = mn;
                }
                const float il = ll > 0.f ? 1.f / ll : 0.f;
                const int hl = rr / k, r = rr - hl * k;
                const size_t o0 = (((size_t)b * k + r) * a.Hq + g * a.G + hl) * DH;
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    act_store4(a.out, o0 + (size_t)(c + 8 * q) * 4,
                               make_float4(acc[4 * q] * il, acc[4 * q + 1] * il, acc[4 * q + 2] * il,
                                           acc[4 * q + 3] * il));
            }
        }
    }
    // the cache stream of the slower CTAs leaves DRAM time for the next
    // projection's weights: this CTA's share goes to L2 (the K/V tiles were
    // loaded evict-first, so the weights stay)
    if (threadIdx.x == 0 && a.l2_next)
        prefetch_l2_share(a.l2_next, a.l2_next_bytes, blockIdx.x, gridDim.x);
    if (warp == MMA_WARP) tmem_dealloc(tmem, TMEM_COLS);
}

// Merge of the partial segments for small batches (a few long sequences, each
// spread over many groups): one block per (kv head g, sequence b, query row),
// one thread per dim, the pair's segments combined in the exp2 domain in
// chunks of eight with their loads issued together.  Pairs inside one share
// were finished by the attention kernel.
__global__ void __launch_bounds__(DH) attn_tc_merge_kernel(AttnArgs a) {
    pdl_trigger();
    __shared__ int prefix[MAX_B + 1];
    __shared__ int cuts[MAX_GRP + 1];
    const int g = blockIdx.x, b = blockIdx.y, rr = blockIdx.z, c = threadIdx.x;
    const int B = a.B, Hkv = a.Hkv, R = a.R, k = a.k;
    if (threadIdx.x == 0) {
        int run = 0;
        for (int bb = 0; bb < B; ++bb) {
            prefix[bb] = run;
            const SeqRef sq = resolve_seq(a.seq_ids, a.seq_lens, a.lens_by_batch, bb, a.kv.n_seqs,
                                          a.max_seq_len, nullptr);
            run += ceil_div(sq.len + a.r0 + k, TT);
        }
        prefix[B] = run;
    }
    __syncthreads();
    const int T = prefix[B];
    const int n_grp = min(a.tc_ctas / Hkv, ceil_div(T, max(1, a.tc_min_tiles)));
    for (int j = threadIdx.x; j <= n_grp; j += blockDim.x) cuts[j] = share_start(prefix, B, T, n_grp, j, a.tc_seg_cost);
    __syncthreads();
    const int j0 = group_of(cuts, n_grp, prefix[b]);
    const int j1 = group_of(cuts, n_grp, prefix[b + 1] - 1);
    if (j0 == j1) return;  // written by the attention kernel
    pdl_wait();            // the partials come from the attention kernel
    const int ns = j1 - j0 + 1;
    float mm = -INFINITY, l = 0.f, o = 0.f;
    for (int e0 = 0; e0 < ns; e0 += 8) {
        float mv[8], lv[8], ov[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const bool in = e0 + e < ns;
            const size_t sl = ((size_t)j0 + e0 + e + b) * Hkv + g;
            mv[e] = in ? __ldcg(a.part_ml + (sl * R + rr) * 2) : -INFINITY;
            lv[e] = in ? __ldcg(a.part_ml + (sl * R + rr) * 2 + 1) : 0.f;
            ov[e] = in ? __ldcg(a.part_o + (sl * R + rr) * DH + c) : 0.f;
        }
        float mn = mm;
#pragma unroll
        for (int e = 0; e < 8; ++e) mn = fmaxf(mn, mv[e]);
        if (mn == -INFINITY) continue;
        const float al = mm == -INFINITY ? 0.f : exp2f(mm - mn);
        l *= al;
        o *= al;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const float w = mv[e] == -INFINITY ? 0.f : exp2f(mv[e] - mn);
            l += w * lv[e];
            o += w * ov[e];
        }
        mm = mn;
    }
    const int hl = rr / k, r = rr - hl * k;
    act_store(a.out, (((size_t)b * k + r) * a.Hq + g * a.G + hl) * DH + c, l > 0.f ? o / l : 0.f);
}

}  // namespace

bool attention_tc_supported(const AttnArgs &a) {
    return a.dh == DH && a.kv_bf16 && a.R >= 1 && a.R <= 128 && a.B >= 1 && a.B <= MAX_B &&
           a.tc_ctas / a.Hkv <= MAX_GRP &&
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
    cudaError_t e = launch_k(attn_tc_kernel, dim3(a.tc_ctas), dim3(THREADS), SMEM_BYTES, st,
                             map_k ? *map_k : dummy, map_v ? *map_v : dummy, a);
    if (e != cudaSuccess || !a.tc_merge_kernel) return e;
    return launch_k(attn_tc_merge_kernel, dim3(a.Hkv, a.B, a.R), dim3(DH), 0, st, a);
}

}  // namespace sp
