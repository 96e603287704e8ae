"""CUDA path vs the fp64 oracle on seeded inputs (all named workloads, edge
cases) and invariants of the GPU path.  Every call goes through the C ABI."""
import hashlib

import numpy as np
import pytest

import oracle.sp_oracle as so
import paper_2608_28099_gb300 as sp
from paper_2608_28099_gb300 import workloads as wl
from gpu_util import ATOL, RTOL, GpuRun, compare, ensure_built, oracle_logits, torch_dev

pytestmark = pytest.mark.gpu


# --------------------------------------------------------------------------- #
# named workloads
# --------------------------------------------------------------------------- #
def test_tiny_fp32_matches_oracle_tightly():
    w = wl.generate(wl.named("tiny"))
    run = GpuRun(w)
    gpu = run.logits()
    ref = oracle_logits(w)
    # fp32 weights and cache: a much tighter bound than the bf16 one
    scale = float(np.max(np.abs(ref)))
    assert np.max(np.abs(gpu - ref)) <= 1e-5 * scale + 1e-7, (gpu, ref)
    compare(gpu, ref, label="tiny")
    run.close()


@pytest.mark.parametrize("name", ["4b", "8b_paged", "27b_long"])
def test_named_workload_matches_oracle(name):
    w = wl.generate(wl.named(name, rows_per_seq=True))
    run = GpuRun(w)
    for use_rows in (True, False):
        gpu = run.logits(use_rows=use_rows)
        ref = oracle_logits(w, use_rows=use_rows)
        assert np.all(np.isfinite(gpu))
        # logits are O(0.1-1) here, so the bound is not vacuous
        assert np.max(np.abs(ref)) > 0.05
        compare(gpu, ref, label=f"{name} rows={use_rows}")
    run.close()


SWEEP_SAMPLE = ["sweep_B1_L512_k1_C2", "sweep_B8_L2048_k4_C16", "sweep_B32_L8192_k16_C2",
                "sweep_B8_L16384_k32_C16", "sweep_B128_L512_k32_C2", "sweep_B256_L512_k1_C16"]


@pytest.mark.parametrize("name", SWEEP_SAMPLE)
def test_sweep_point_matches_oracle_on_a_subset(name):
    w = wl.generate(wl.named(name))
    run = GpuRun(w)
    gpu = run.logits()
    sub = np.random.default_rng(0).choice(len(w.seq_ids), size=min(8, len(w.seq_ids)),
                                          replace=False)
    ref = oracle_logits(w, ids=np.sort(sub))
    compare(gpu[np.sort(sub)], ref, label=name)
    run.close()


# --------------------------------------------------------------------------- #
# edge cases on small shapes (several tiles, ragged tails)
# --------------------------------------------------------------------------- #
SMALL_BF16 = wl.Shape(256, 8, 2, 128, 512, 4, 3)
EDGE_LENS = [0, 1, 15, 16, 17, 63, 64, 65, 127, 300]


@pytest.mark.parametrize("layout", [wl.LAYOUT_CONTIGUOUS, wl.LAYOUT_PAGED])
@pytest.mark.parametrize("rows", [False, True])
def test_edge_lengths(layout, rows):
    w = wl.custom(SMALL_BF16, EDGE_LENS, layout, 31, rows_per_seq=rows, head_bias=True)
    run = GpuRun(w)
    compare(run.logits(), oracle_logits(w), label="edge")
    run.close()


@pytest.mark.parametrize("shape", [
    wl.Shape(128, 4, 4, 64, 256, 1, 2),            # MHA (G=1), k=1
    wl.Shape(256, 8, 1, 32, 256, 32, 5),           # MQA, k=32, head_dim 32
    wl.Shape(512, 8, 2, 128, 1024, 7, 2, pool=wl.POOL_LAST),
    wl.Shape(384, 12, 4, 64, 768, 5, 16, w_dtype=wl.F32, kv_dtype=wl.F32),
])
def test_shape_variants(shape):
    w = wl.custom(shape, [5, 40, 129, 257], wl.LAYOUT_PAGED, 41, rows_per_seq=True)
    run = GpuRun(w)
    gpu = run.logits()
    ref = oracle_logits(w)
    if shape.w_dtype == wl.F32:
        assert np.max(np.abs(gpu - ref)) <= 1e-4 * max(1.0, np.max(np.abs(ref)))
    compare(gpu, ref, label=str(shape))
    run.close()


def test_sequence_ids_select_and_permute():
    w = wl.custom(SMALL_BF16, [10, 200, 33, 0, 90, 64], wl.LAYOUT_PAGED, 51)
    run = GpuRun(w, max_batch=6)
    ids = [4, 1, 1, 5]
    compare(run.logits(ids=ids, use_rows=False), oracle_logits(w, use_rows=False, ids=ids))
    run.close()


# --------------------------------------------------------------------------- #
# invariants
# --------------------------------------------------------------------------- #
def _sha(t):
    return hashlib.sha256(t.cpu().numpy().tobytes()).hexdigest()


def test_cache_is_never_written():
    w = wl.custom(SMALL_BF16, [100, 257], wl.LAYOUT_PAGED, 61, rows_per_seq=True)
    run = GpuRun(w)
    before = (_sha(run.cache.k_pool), _sha(run.cache.v_pool), _sha(run.cache.page_table))
    run.logits()
    run.logits(use_rows=False)
    assert before == (_sha(run.cache.k_pool), _sha(run.cache.v_pool), _sha(run.cache.page_table))
    run.close()


def test_layouts_and_page_permutation_agree_bitwise():
    base = wl.custom(SMALL_BF16, [70, 300, 1, 128], wl.LAYOUT_CONTIGUOUS, 71, rows_per_seq=True)
    outs = []
    for cache in (base.cache, wl.contiguous_to_paged(base.cache, 16, 1),
                  wl.contiguous_to_paged(base.cache, 16, 2)):
        w = wl.Workload(base.spec, base.weights, cache, base.seq_ids, base.rows)
        run = GpuRun(w, options={sp.SP_OPT_SPLIT_TOKENS: 128})
        outs.append(run.logits())
        run.close()
    assert np.array_equal(outs[0], outs[1]) and np.array_equal(outs[1], outs[2])


@pytest.mark.parametrize("attn_path", [1, 2])
def test_split_plan_does_not_change_results(attn_path):
    w = wl.custom(SMALL_BF16, [1000, 2000, 37], wl.LAYOUT_PAGED, 81)
    res = []
    for split in (64, 256, 2048 + 64):
        run = GpuRun(w, options={sp.SP_OPT_SPLIT_TOKENS: split, sp.SP_OPT_ATTN_PATH: attn_path})
        res.append(run.logits())
        run.close()
    # fp32 attention: only the merge order changes.  Tensor-core attention: the
    # split also moves where P is rounded to bf16.
    tol = 1e-5 if attn_path == 1 else 2e-3
    for r in res[1:]:
        np.testing.assert_allclose(r, res[0], rtol=tol, atol=tol)
    compare(res[0], oracle_logits(w))


def test_repeated_calls_are_bitwise_deterministic():
    w = wl.custom(SMALL_BF16, [500, 12, 1200], wl.LAYOUT_PAGED, 91, rows_per_seq=True)
    run = GpuRun(w)
    a, b = run.logits(), run.logits()
    assert np.array_equal(a, b)
    run.close()


def test_result_does_not_depend_on_batch_company():
    w = wl.custom(SMALL_BF16, [40, 700, 129, 5], wl.LAYOUT_PAGED, 101)
    run = GpuRun(w, max_batch=4)
    full = run.logits(use_rows=False)
    for i in range(4):
        one = run.logits(use_rows=False, ids=[i])
        # the batch size changes the split plans (rounding points), nothing else
        np.testing.assert_allclose(one[0], full[i], rtol=2e-3, atol=2e-3)
    run.close()


def test_shared_prompt_equals_rows_holding_the_prompt():
    w = wl.custom(SMALL_BF16, [33, 90], wl.LAYOUT_PAGED, 111)
    w.rows = np.stack([w.weights.soft_prompt] * 2)
    run = GpuRun(w)
    # fp32 projections of the shared prompt vs tensor-core projections of rows
    np.testing.assert_allclose(run.logits(use_rows=True), run.logits(use_rows=False),
                               rtol=2e-3, atol=2e-3)
    run.close()


def test_host_entry_point_matches_device_entry_point():
    torch = torch_dev()
    w = wl.custom(SMALL_BF16, [50, 260, 3], wl.LAYOUT_PAGED, 121, rows_per_seq=True)
    run = GpuRun(w)
    dev = run.logits()
    out = np.zeros((3, SMALL_BF16.n_classes), dtype=np.float32)
    lens = np.ascontiguousarray(w.cache.seq_lens[w.seq_ids], dtype=np.int32)
    ids = np.ascontiguousarray(w.seq_ids, dtype=np.int32)
    sp.sp_classify_host(run.model.handle, torch.cuda.current_stream(), 3, ids, lens,
                        run.cache.desc, np.ascontiguousarray(w.rows), out)
    assert np.array_equal(out.astype(np.float64), dev)
    run.close()


# --------------------------------------------------------------------------- #
# the attention step alone and its page gather
# --------------------------------------------------------------------------- #
def _attend(shape, w, q, kn, vn, path, split=128):
    torch = torch_dev()
    lens = [int(x) for x in w.cache.seq_lens]
    B, k = len(lens), shape.k_rows
    cache = sp.DeviceCache(w.cache)
    dims = sp.sp_attn_dims(shape.n_q_heads, shape.n_kv_heads, shape.head_dim, k, shape.kv_dtype,
                           max(lens), split, path)
    ws_bytes = sp.sp_attend_workspace_bytes(dims, B)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device="cuda")
    out = torch.full(q.shape, float("nan"), dtype=torch.float32, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    gathered = None
    if w.cache.layout == wl.LAYOUT_PAGED:
        gathered = torch.full((B, w.cache.max_pages), -7, dtype=torch.int32, device="cuda")
    sp.sp_attend(torch.cuda.current_stream(), dims, B, None, cache.seq_lens, cache.desc,
                 torch.from_numpy(q).cuda(), torch.from_numpy(kn).cuda(), torch.from_numpy(vn).cuda(),
                 out, sp.SP_F32, ws, ws_bytes, status, gathered)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    return out.cpu().numpy(), (None if gathered is None else gathered.cpu().numpy())


ATTN_CASES = [
    # kv dtype, head_dim, layout, q heads, kv heads, k rows, page size, path
    (wl.F32, 64, wl.LAYOUT_PAGED, 8, 2, 5, 16, 1),
    (wl.BF16, 64, wl.LAYOUT_PAGED, 8, 2, 5, 16, 1),
    (wl.BF16, 128, wl.LAYOUT_PAGED, 8, 2, 5, 16, 2),
    (wl.BF16, 128, wl.LAYOUT_CONTIGUOUS, 8, 2, 5, 16, 2),
    (wl.BF16, 128, wl.LAYOUT_PAGED, 8, 2, 32, 16, 2),     # 128 query rows per kv head
    (wl.BF16, 128, wl.LAYOUT_PAGED, 10, 2, 16, 32, 2),    # G=5 as in the 27B shape, 32-token pages
    (wl.BF16, 128, wl.LAYOUT_PAGED, 4, 4, 1, 64, 2),      # MHA, k=1, 64-token pages
    (wl.BF16, 128, wl.LAYOUT_CONTIGUOUS, 16, 2, 9, 16, 2),
]


@pytest.mark.parametrize("case", ATTN_CASES, ids=lambda c: "-".join(map(str, c)))
def test_attention_step_and_gathered_pages(case):
    ensure_built()
    kv_dtype, dh, layout, hq, hkv, k, P, path = case
    shape = wl.Shape(256, hq, hkv, dh, 256, k, 2, kv_dtype=kv_dtype, page_size=P)
    lens = [0, 16, 17, 250, 1000, 64, 127]
    w = wl.custom(shape, lens, layout, 131)
    rng = np.random.default_rng(7)
    B = len(lens)
    q = rng.standard_normal((B, k, hq, dh)).astype(np.float32)
    kn = rng.standard_normal((B, k, hkv, dh)).astype(np.float32)
    vn = rng.standard_normal((B, k, hkv, dh)).astype(np.float32)
    ref = so.attention_step(shape, w.cache, w.seq_ids, q.astype(np.float64), kn.astype(np.float64),
                            vn.astype(np.float64))
    out, g = _attend(shape, w, q, kn, vn, path)
    # CUDA cores: fp32 throughout.  Tensor cores: Q as bf16 hi+lo, P and the new
    # keys/values as bf16, fp32 accumulation.
    tol = 1e-4 if path == 1 else 1e-2
    np.testing.assert_allclose(out, ref, rtol=tol, atol=tol)
    if g is not None:
        for b, L in enumerate(lens):
            npg = (L + P - 1) // P
            assert np.array_equal(g[b, :npg], w.cache.page_table[b, :npg])  # bit-exact ids
            assert np.all(g[b, npg:] == -7)                                 # nothing else read


@pytest.mark.parametrize("layout", [wl.LAYOUT_PAGED, wl.LAYOUT_CONTIGUOUS])
def test_attention_tensor_and_cuda_core_kernels_agree(layout):
    ensure_built()
    shape = wl.Shape(256, 32, 8, 128, 256, 8, 2)
    lens = [3000, 70, 1025, 0, 4096]
    w = wl.custom(shape, lens, layout, 137)
    rng = np.random.default_rng(8)
    B = len(lens)
    q = (rng.standard_normal((B, 8, 32, 128))).astype(np.float32)
    kn = rng.standard_normal((B, 8, 8, 128)).astype(np.float32)
    vn = rng.standard_normal((B, 8, 8, 128)).astype(np.float32)
    tc, _ = _attend(shape, w, q, kn, vn, 2, split=0)
    ref, _ = _attend(shape, w, q, kn, vn, 1, split=0)
    np.testing.assert_allclose(tc, ref, rtol=1e-2, atol=1e-2)
    assert np.sqrt(np.mean((tc - ref) ** 2)) < 2e-3


# --------------------------------------------------------------------------- #
# device-side status (bad ids, lengths, pages never fault; they are reported)
# --------------------------------------------------------------------------- #
def test_device_status_reports_bad_inputs():
    torch = torch_dev()
    w = wl.custom(SMALL_BF16, [20, 40], wl.LAYOUT_PAGED, 141)
    run = GpuRun(w, max_batch=2, max_seq_len=64)
    h = run.model.handle
    out = torch.empty((2, SMALL_BF16.n_classes), dtype=torch.float32, device="cuda")
    st = torch.cuda.current_stream()
    bad_ids = torch.tensor([0, 9], dtype=torch.int32, device="cuda")
    sp.sp_classify(h, st, 2, bad_ids, run.cache.seq_lens, run.cache.desc, None, out)
    assert sp.sp_check_status(h) & sp.SP_DEV_BAD_SEQ_ID
    bad_lens = torch.tensor([20, 65], dtype=torch.int32, device="cuda")
    sp.sp_classify(h, st, 2, None, bad_lens, run.cache.desc, None, out)
    assert sp.sp_check_status(h) & sp.SP_DEV_BAD_LENGTH
    pt = run.cache.page_table.clone()
    pt[1, 1] = 10_000
    desc = sp.sp_kv_cache(sp.SP_KV_PAGED, None, None, run.cache.k_pool.data_ptr(),
                          run.cache.v_pool.data_ptr(), pt.data_ptr(), 16, w.cache.n_pages,
                          w.cache.max_pages, 2)
    sp.sp_classify(h, st, 2, None, run.cache.seq_lens, desc, None, out)
    assert sp.sp_check_status(h) & sp.SP_DEV_BAD_PAGE
    # the context is still usable and a clean call reports nothing
    good = run.logits(use_rows=False)
    compare(good, oracle_logits(w, use_rows=False))
    run.close()


def test_empty_and_oversized_batches_are_refused_before_any_launch():
    # batch must lie in 1..max_batch: an empty batch and one beyond the handle's
    # max_batch are refused on the host (nothing is enqueued), and the handle
    # stays usable
    torch = torch_dev()
    w = wl.custom(SMALL_BF16, [20, 40], wl.LAYOUT_PAGED, 141)
    run = GpuRun(w, max_batch=2, max_seq_len=64)
    h = run.model.handle
    out = torch.full((3, SMALL_BF16.n_classes), 7.0, dtype=torch.float32, device="cuda")
    st = torch.cuda.current_stream()
    for batch in (0, 3):
        with pytest.raises(sp.SpError) as e:
            sp.sp_classify(h, st, batch, None, run.cache.seq_lens, run.cache.desc, None, out)
        assert e.value.status == sp.SP_ERR_INVALID_ARG
    torch.cuda.synchronize()
    assert bool((out == 7.0).all())
    compare(run.logits(use_rows=False), oracle_logits(w, use_rows=False))
    run.close()


@pytest.mark.parametrize("prec", [0, 1, 2, 3, 4])
def test_mlp_activation_precision_options(prec):
    # automatic (bf16 MLP inputs here: mean over 8 rows), hi + lo, plain bf16
    # for the MLP, plain bf16 for every projection, for all but Q/K/V: all
    # inside the tolerance on a multi-tile shape
    shape = wl.Shape(512, 8, 2, 128, 1024, 8, 4)
    w = wl.custom(shape, [5, 40, 129, 257, 700, 1024, 64, 3], wl.LAYOUT_PAGED, 81,
                  rows_per_seq=True)
    run = GpuRun(w, options={sp.SP_OPT_ACT_PRECISION: prec})
    compare(run.logits(), oracle_logits(w), label=f"precision option {prec}")
    run.close()


@pytest.mark.parametrize("opts", [
    {sp.SP_OPT_GEMM_SCHEDULE: 1}, {sp.SP_OPT_GEMM_SCHEDULE: 2},
    {sp.SP_OPT_ATTN_MERGE: 1}, {sp.SP_OPT_ATTN_MERGE: 2},
    {sp.SP_OPT_QUERY_PRECISION: 1}, {sp.SP_OPT_QUERY_PRECISION: 2},
], ids=["gemm-tile", "gemm-persistent", "merge-in-kernel", "merge-kernel", "query-hi-lo",
        "query-plain"])
def test_work_split_and_query_precision_options(opts):
    # every projection schedule, both places of the attention merge and both
    # query precisions stay inside the tolerance: 16 pooled rows (plain bf16
    # queries by default here), 8 ragged sequences over many tiles
    shape = wl.Shape(512, 8, 2, 128, 1024, 16, 4)
    w = wl.custom(shape, [5, 40, 129, 257, 700, 1024, 64, 3], wl.LAYOUT_PAGED, 83,
                  rows_per_seq=True)
    run = GpuRun(w, options=opts)
    compare(run.logits(), oracle_logits(w), label=str(opts))
    run.close()


def test_wide_model_takes_the_two_pass_norms():
    # d > 8192 rows do not fit the register-resident norm kernels; the two-pass
    # kernels serve them (input norm, residual + post-norm)
    shape = wl.Shape(8448, 8, 2, 128, 1024, 8, 2)
    w = wl.custom(shape, [64, 300, 1000], wl.LAYOUT_PAGED, 91, rows_per_seq=True)
    run = GpuRun(w)
    compare(run.logits(), oracle_logits(w), label="d = 8448")
    run.close()


def test_tensor_core_wait_timeout_is_reported_and_the_handle_recovers():
    # the failure path of the bounded waits: one CTA of the output projection
    # never receives its first k-block, its MMA warp gives up after 1 ms, the
    # kernel drains, frees TMEM and reports SP_DEV_TIMEOUT; nothing faults
    torch = torch_dev()
    w = wl.custom(SMALL_BF16, [20, 300, 64, 5], wl.LAYOUT_PAGED, 151, rows_per_seq=True)
    run = GpuRun(w)
    h = run.model.handle
    out = torch.empty((4, SMALL_BF16.n_classes), dtype=torch.float32, device="cuda")
    sp.sp_set_option(h, sp.SP_OPT_DEBUG_STALL, 1)
    sp.sp_classify(h, torch.cuda.current_stream(), 4, run.ids, run.cache.seq_lens, run.cache.desc,
                   run.rows, out)
    assert sp.sp_check_status(h) & sp.SP_DEV_TIMEOUT
    # the option was one-shot: the next call on the same handle is clean and exact
    compare(run.logits(), oracle_logits(w), label="after timeout")
    run.close()


def test_classify_records_the_gathered_pages_bit_exact():
    # the page-table walk of the full call on the 8b paged configuration
    # (K/V values drawn on the device; lengths and page table as the host draw)
    torch = torch_dev()
    ensure_built()
    spec = wl.named("8b_paged", rows_per_seq=True)
    dw = wl.generate_on_device(spec)
    cache = sp.DevicePagedCache(dw)
    B = spec.batch
    model = sp.Model(spec.shape, dw.weights, B, int(dw.seq_lens.max()))
    h = model.handle
    max_pages = dw.page_table.shape[1]
    rec = torch.full((B, max_pages), -1, dtype=torch.int32, device="cuda")
    sp.sp_debug_gathered_pages(h, rec)
    rows = torch.from_numpy(np.ascontiguousarray(dw.rows).view(np.int16)).cuda()
    ids = torch.arange(B, dtype=torch.int32, device="cuda")
    out = torch.empty((B, spec.shape.n_classes), dtype=torch.float32, device="cuda")
    sp.sp_classify(h, torch.cuda.current_stream(), B, ids, cache.seq_lens, cache.desc, rows, out)
    assert sp.sp_check_status(h) == 0
    got = rec.cpu().numpy()
    for b in range(B):
        npg = (int(dw.seq_lens[b]) + 15) // 16
        assert np.array_equal(got[b, :npg], dw.page_table[b, :npg])
        assert np.all(got[b, npg:] == -1)  # pages past the length are never read
    sp.sp_debug_gathered_pages(h, None)
    model.close()
