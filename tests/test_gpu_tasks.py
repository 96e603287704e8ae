"""Several probes over one pass of the cache (Sec. 3.3: classifiers with their own
soft prompt and head sharing the draft head's KV cache) through the C ABI,
against the fp64 oracle's task-by-task classification."""

import numpy as np
import pytest

import oracle.sp_oracle as so
import paper_2608_28099_gb300 as sp
from paper_2608_28099_gb300 import workloads as wl
from gpu_util import GpuRun, compare, rows_tensor

pytestmark = pytest.mark.gpu

SHAPE = wl.Shape(256, 8, 2, 128, 512, 4, 3)   # G = 4: T = 3 tasks give 48 query rows


def task_logits(run: GpuRun, use_rows=True, hidden=None):
    torch = run.torch
    w = run.w
    B, T, C = len(w.seq_ids), w.shape.n_tasks, w.shape.n_classes
    out = torch.empty((B, T, C), dtype=torch.float32, device="cuda")
    stream = torch.cuda.current_stream()
    if hidden is not None:
        sp.sp_classify_hidden(run.model.handle, stream, B, run.ids, run.cache.seq_lens,
                              run.cache.desc, rows_tensor(torch, hidden), out)
    else:
        sp.sp_classify(run.model.handle, stream, B, run.ids, run.cache.seq_lens, run.cache.desc,
                       run.rows if use_rows else None, out)
    torch.cuda.synchronize()
    assert sp.sp_check_status(run.model.handle) == 0, sp.sp_last_error()
    return out.cpu().numpy().astype(np.float64)


def oracle_tasks(w, use_rows=True, hidden=None):
    prompts, heads, biases, rows = wl.task_views(w)
    return so.classify_tasks(so.Layer(w.shape, w.weights), w.cache, w.seq_ids, prompts, heads,
                             biases, rows if use_rows else None, hidden=hidden)


@pytest.mark.parametrize("layout", [wl.LAYOUT_PAGED, wl.LAYOUT_CONTIGUOUS])
def test_tasks_match_oracle(layout):
    w = wl.with_tasks(wl.custom(SHAPE, [0, 40, 700, 1500], layout, 301, rows_per_seq=True,
                                head_bias=True), 3)
    run = GpuRun(w)
    for use_rows in (True, False):
        gpu = task_logits(run, use_rows)
        ref = oracle_tasks(w, use_rows)
        assert np.max(np.abs(ref)) > 0.05
        for t in range(3):
            compare(gpu[:, t], ref[:, t], label=f"task {t} rows={use_rows}")
    run.close()


def test_task_zero_of_many_equals_the_single_task_handle():
    base = wl.custom(SHAPE, [33, 500, 1200], wl.LAYOUT_PAGED, 302, rows_per_seq=True)
    many = wl.with_tasks(base, 4)
    one = GpuRun(base)
    run = GpuRun(many)
    single = one.logits()
    multi = task_logits(run)
    # the same task through different batch shapes of the projections and
    # attention: equal within rounding, not bitwise
    np.testing.assert_allclose(multi[:, 0], single, rtol=2e-3, atol=2e-3)
    one.close()
    run.close()


def test_other_tasks_do_not_touch_a_task_bitwise():
    w = wl.with_tasks(wl.custom(SHAPE, [64, 300, 1000], wl.LAYOUT_PAGED, 303, rows_per_seq=True), 3)
    run = GpuRun(w)
    a = task_logits(run)
    rows = w.rows.copy()
    k = SHAPE.k_rows
    rows[:, k:2 * k] = rows[:, k:2 * k][:, ::-1]          # task 1's rows reversed
    run.rows = rows_tensor(run.torch, rows)
    b = task_logits(run)
    assert np.array_equal(a[:, 0], b[:, 0]) and np.array_equal(a[:, 2], b[:, 2])
    assert np.max(np.abs(a[:, 1] - b[:, 1])) > 1e-4
    run.close()


def test_tasks_fp32_tiny_on_cuda_cores():
    w = wl.generate(wl.named("tiny", n_tasks=2))
    run = GpuRun(w)
    gpu = task_logits(run, use_rows=False)
    ref = oracle_tasks(w, use_rows=False)
    scale = float(np.max(np.abs(ref)))
    assert np.max(np.abs(gpu - ref)) <= 1e-5 * scale + 1e-7, (gpu, ref)
    run.close()


def test_tasks_with_input_fusion():
    w = wl.with_fusion(wl.with_tasks(wl.custom(SHAPE, [20, 900], wl.LAYOUT_PAGED, 304), 2))
    run = GpuRun(w)
    gpu = task_logits(run, hidden=w.hidden)
    ref = oracle_tasks(w, use_rows=False, hidden=w.hidden)
    for t in range(2):
        compare(gpu[:, t], ref[:, t], label=f"fused task {t}")
    run.close()


def test_recursive_probing_rejects_several_tasks():
    w = wl.with_fusion(wl.with_tasks(wl.custom(SHAPE, [20, 90], wl.LAYOUT_PAGED, 305), 2))
    run = GpuRun(w, options={sp.SP_OPT_RECURSIVE: 1})
    with pytest.raises(sp.SpError) as e:
        task_logits(run, hidden=w.hidden)
    assert e.value.status == sp.SP_ERR_UNSUPPORTED
    run.close()
