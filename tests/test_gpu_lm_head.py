"""The LM-head readout (Sec. 5 ablation, "Classification head": the frozen
lm_head at the label tokens after the head's final RMSNorm) through the C ABI,
against the fp64 oracle, in every form of the path."""
import numpy as np
import pytest

import oracle.sp_oracle as so
import paper_2608_28099_gb300 as sp
from paper_2608_28099_gb300 import workloads as wl
from gpu_util import GpuRun, compare, oracle_logits, rows_tensor

pytestmark = pytest.mark.gpu

SHAPE = wl.Shape(256, 8, 2, 128, 512, 4, 2)


@pytest.mark.parametrize("pool", [wl.POOL_MEAN, wl.POOL_LAST])
@pytest.mark.parametrize("layout", [wl.LAYOUT_PAGED, wl.LAYOUT_CONTIGUOUS])
def test_lm_head_readout_matches_oracle(pool, layout):
    sh = wl.Shape(256, 8, 2, 128, 512, 4, 2, pool=pool)
    w = wl.with_lm_head(wl.custom(sh, [0, 300, 1100], layout, 401, rows_per_seq=True))
    run = GpuRun(w)
    for use_rows in (True, False):
        gpu = run.logits(use_rows=use_rows)
        ref = oracle_logits(w, use_rows=use_rows)
        # unit-RMS pooled state times 0.02-scale rows: logits of O(0.1-1)
        assert np.max(np.abs(ref)) > 0.05
        compare(gpu, ref, label=f"lm head rows={use_rows}")
        # the yes/no difference, the binary logit the paper reads
        np.testing.assert_allclose(gpu[:, 1] - gpu[:, 0], ref[:, 1] - ref[:, 0],
                                   atol=2e-2, rtol=1e-2)
    run.close()


def test_lm_head_readout_tiny_fp32_tightly():
    w = wl.with_lm_head(wl.generate(wl.named("tiny")))
    run = GpuRun(w)
    gpu = run.logits(use_rows=False)
    ref = oracle_logits(w, use_rows=False)
    scale = float(np.max(np.abs(ref)))
    assert np.max(np.abs(gpu - ref)) <= 1e-5 * scale + 1e-7, (gpu, ref)
    run.close()


def test_lm_head_readout_recursive_and_tasks():
    base = wl.with_fusion(wl.custom(SHAPE, [40, 900], wl.LAYOUT_PAGED, 402))
    w = wl.with_lm_head(base)
    run = GpuRun(w, options={sp.SP_OPT_RECURSIVE: 1})
    torch = run.torch
    out = torch.empty((2, SHAPE.n_classes), dtype=torch.float32, device="cuda")
    sp.sp_classify_hidden(run.model.handle, torch.cuda.current_stream(), 2, run.ids,
                          run.cache.seq_lens, run.cache.desc, rows_tensor(torch, w.hidden), out)
    torch.cuda.synchronize()
    gpu = out.cpu().numpy().astype(np.float64)
    ref = so.classify_recursive(so.Layer(w.shape, w.weights), w.cache, w.seq_ids, w.hidden)
    compare(gpu, ref, label="recursive lm head")
    run.close()
    wt = wl.with_lm_head(wl.with_tasks(wl.custom(SHAPE, [70, 500], wl.LAYOUT_PAGED, 403), 3))
    run = GpuRun(wt)
    out = torch.empty((2, 3, SHAPE.n_classes), dtype=torch.float32, device="cuda")
    sp.sp_classify(run.model.handle, torch.cuda.current_stream(), 2, run.ids, run.cache.seq_lens,
                   run.cache.desc, None, out)
    torch.cuda.synchronize()
    gpu = out.cpu().numpy().astype(np.float64)
    prompts, heads, biases, _ = wl.task_views(wt)
    ref = so.classify_tasks(so.Layer(wt.shape, wt.weights), wt.cache, wt.seq_ids, prompts, heads,
                            biases)
    for t in range(3):
        compare(gpu[:, t], ref[:, t], label=f"task {t} lm head")
    run.close()
