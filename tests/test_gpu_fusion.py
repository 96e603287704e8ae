"""The classify path fed by base hidden states (MTP input fusion, Sec. 3.1 and
Sec. 3.2 single-step probing) through the C ABI, against the fp64 oracle."""
import numpy as np
import pytest

import oracle.sp_oracle as so
import paper_2608_28099_gb300 as sp
from paper_2608_28099_gb300 import workloads as wl
from gpu_util import GpuRun, compare, rows_tensor, torch_dev

pytestmark = pytest.mark.gpu

SMALL_BF16 = wl.Shape(256, 8, 2, 128, 512, 4, 3)


def hidden_logits(run: GpuRun, hidden, host=False):
    torch = run.torch
    B = len(run.w.seq_ids)
    out = torch.empty((B, run.w.shape.n_classes), dtype=torch.float32, device="cuda")
    if host:
        res = np.zeros((B, run.w.shape.n_classes), dtype=np.float32)
        lens = np.ascontiguousarray(run.w.cache.seq_lens[run.w.seq_ids], dtype=np.int32)
        ids = np.ascontiguousarray(run.w.seq_ids, dtype=np.int32)
        h = np.ascontiguousarray(hidden)
        sp.sp_classify_hidden_host(run.model.handle, torch.cuda.current_stream(), B, ids, lens,
                                   run.cache.desc, h.view(np.int16) if h.dtype == np.uint16 else h,
                                   res)
        return res.astype(np.float64)
    sp.sp_classify_hidden(run.model.handle, torch.cuda.current_stream(), B, run.ids,
                          run.cache.seq_lens, run.cache.desc, rows_tensor(torch, hidden), out)
    torch.cuda.synchronize()
    assert sp.sp_check_status(run.model.handle) == 0, sp.sp_last_error()
    return out.cpu().numpy().astype(np.float64)


def oracle_hidden(w):
    return so.classify(so.Layer(w.shape, w.weights), w.cache, w.seq_ids, hidden=w.hidden)


CASES = [
    ("paged_ragged", SMALL_BF16, [0, 17, 300, 1000, 64], wl.LAYOUT_PAGED),
    ("contiguous", SMALL_BF16, [5, 129, 700], wl.LAYOUT_CONTIGUOUS),
    ("k1", wl.Shape(256, 8, 2, 128, 512, 1, 2), [40, 2000], wl.LAYOUT_PAGED),
    ("head_dim_64", wl.Shape(256, 8, 4, 64, 512, 3, 2), [90, 33], wl.LAYOUT_PAGED),
    # 64 sequences x 8 rows and 48 heads: the Q/K/V projection runs one CTA per
    # head with no K split, so the rotation happens in its epilogue
    ("rotation_in_projection", wl.Shape(256, 32, 8, 128, 512, 8, 2),
     [int(v) for v in np.random.default_rng(5).integers(0, 100, size=64)], wl.LAYOUT_PAGED),
]


@pytest.mark.parametrize("name,shape,lens,layout", CASES, ids=[c[0] for c in CASES])
def test_fused_input_matches_oracle(name, shape, lens, layout):
    w = wl.with_fusion(wl.custom(shape, lens, layout, 201))
    run = GpuRun(w)
    gpu = hidden_logits(run, w.hidden)
    ref = oracle_hidden(w)
    assert np.all(np.isfinite(gpu))
    assert np.max(np.abs(ref)) > 0.05
    compare(gpu, ref, label=name)
    run.close()


def test_fused_tiny_fp32_matches_oracle_tightly():
    w = wl.generate(wl.named("tiny", fused=True))
    run = GpuRun(w)
    gpu = hidden_logits(run, w.hidden)
    ref = oracle_hidden(w)
    scale = float(np.max(np.abs(ref)))
    assert np.max(np.abs(gpu - ref)) <= 1e-5 * scale + 1e-7, (gpu, ref)
    run.close()


def test_fused_4b_workload_matches_oracle():
    w = wl.generate(wl.named("4b", fused=True))
    run = GpuRun(w)
    gpu = hidden_logits(run, w.hidden)
    ref = oracle_hidden(w)
    assert np.max(np.abs(ref)) > 0.05
    compare(gpu, ref, label="4b fused")
    run.close()


def test_fused_host_entry_equals_device_entry():
    w = wl.with_fusion(wl.custom(SMALL_BF16, [70, 3, 520], wl.LAYOUT_PAGED, 202))
    run = GpuRun(w)
    dev = hidden_logits(run, w.hidden)
    host = hidden_logits(run, w.hidden, host=True)
    assert np.array_equal(dev, host)
    run.close()


def test_fused_rows_equal_the_row_path_given_the_same_rows():
    # the fused inputs computed by the oracle, passed as explicit rows, give the
    # same logits through sp_classify (the fusion stage is the only difference)
    w = wl.with_fusion(wl.custom(SMALL_BF16, [300, 45], wl.LAYOUT_PAGED, 203))
    layer = so.Layer(w.shape, w.weights)
    k = w.shape.k_rows
    rows = np.stack([layer.fuse(np.repeat(so.to_f64(w.hidden[i], w.shape.w_dtype)[None], k, axis=0),
                                layer.soft_prompt) for i in range(2)])
    w.rows = wl.f32_to_bf16_bits(rows.astype(np.float32))
    run = GpuRun(w)
    via_rows = run.logits(use_rows=True)
    fused = hidden_logits(run, w.hidden)
    # rows rounded to bf16 vs fused rows kept in fp32: within the bf16 tolerance
    compare(fused, via_rows, label="fused vs rows")
    run.close()


def test_hidden_entry_needs_fusion_weights():
    torch = torch_dev()
    w = wl.custom(SMALL_BF16, [10, 20], wl.LAYOUT_PAGED, 204)
    run = GpuRun(w)
    hidden = torch.zeros((2, SMALL_BF16.d_model), dtype=torch.int16, device="cuda")
    out = torch.empty((2, SMALL_BF16.n_classes), device="cuda")
    with pytest.raises(sp.SpError) as e:
        sp.sp_classify_hidden(run.model.handle, None, 2, run.ids, run.cache.seq_lens,
                              run.cache.desc, hidden, out)
    assert e.value.status == sp.SP_ERR_INVALID_ARG
    run.close()


# --------------------------------------------------------------------------- #
# recursive probing SP-k (SP_OPT_RECURSIVE)
# --------------------------------------------------------------------------- #
REC_CASES = [
    ("paged_k4", SMALL_BF16, [0, 17, 300, 1000, 64], wl.LAYOUT_PAGED, wl.POOL_MEAN),
    ("contiguous_last", wl.Shape(256, 8, 2, 128, 512, 3, 2, pool=wl.POOL_LAST), [5, 129, 700],
     wl.LAYOUT_CONTIGUOUS, wl.POOL_LAST),
    ("k1", wl.Shape(256, 8, 2, 128, 512, 1, 2), [40, 2000], wl.LAYOUT_PAGED, wl.POOL_MEAN),
    ("head_dim_64", wl.Shape(256, 8, 4, 64, 512, 5, 2), [90, 33, 250], wl.LAYOUT_PAGED,
     wl.POOL_MEAN),
]


@pytest.mark.parametrize("name,shape,lens,layout,pool", REC_CASES, ids=[c[0] for c in REC_CASES])
def test_recursive_probing_matches_oracle(name, shape, lens, layout, pool):
    w = wl.with_fusion(wl.custom(shape, lens, layout, 211))
    run = GpuRun(w, options={sp.SP_OPT_RECURSIVE: 1})
    gpu = hidden_logits(run, w.hidden)
    ref = so.classify_recursive(so.Layer(w.shape, w.weights), w.cache, w.seq_ids, w.hidden)
    assert np.all(np.isfinite(gpu))
    assert np.max(np.abs(ref)) > 0.05
    compare(gpu, ref, label=f"recursive {name}")
    # the parallel form of the same inputs differs for k > 1 (a real recursion ran)
    if shape.k_rows > 1:
        par = oracle_hidden(w)
        assert np.max(np.abs(par - ref)) > 1e-3
    run.close()


def test_recursive_tiny_fp32_matches_oracle_tightly():
    w = wl.generate(wl.named("tiny", fused=True))
    run = GpuRun(w, options={sp.SP_OPT_RECURSIVE: 1})
    gpu = hidden_logits(run, w.hidden)
    ref = so.classify_recursive(so.Layer(w.shape, w.weights), w.cache, w.seq_ids, w.hidden)
    scale = float(np.max(np.abs(ref)))
    assert np.max(np.abs(gpu - ref)) <= 1e-5 * scale + 1e-7, (gpu, ref)
    run.close()


def test_recursive_then_parallel_on_one_handle():
    # switching the option back restores the parallel form exactly
    w = wl.with_fusion(wl.custom(SMALL_BF16, [80, 400], wl.LAYOUT_PAGED, 212))
    run = GpuRun(w)
    first = hidden_logits(run, w.hidden)
    sp.sp_set_option(run.model.handle, sp.SP_OPT_RECURSIVE, 1)
    rec = hidden_logits(run, w.hidden)
    sp.sp_set_option(run.model.handle, sp.SP_OPT_RECURSIVE, 0)
    again = hidden_logits(run, w.hidden)
    assert np.array_equal(first, again)
    assert np.max(np.abs(first - rec)) > 1e-3
    run.close()
