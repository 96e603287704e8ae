"""sp_attend_static: the attention step for callers that cannot allocate device
memory (a monitor on the decoding hot path must not call cudaMalloc, which can
synchronise the device; some serving frameworks give a library no device memory
of its own).  It must give the same result as sp_attend with a caller-provided
workspace, call after call, although every call reuses one static array."""
import gc

import numpy as np
import pytest

import paper_2608_28099_gb300 as sp
from paper_2608_28099_gb300 import workloads as wl
from gpu_util import ensure_built, torch_dev

pytestmark = pytest.mark.gpu


def _inputs(torch, lens, seed, kv_dtype=wl.BF16):
    shape = wl.Shape(256, 8, 2, 128, 256, 6, 2, kv_dtype=kv_dtype)
    w = wl.custom(shape, lens, wl.LAYOUT_PAGED, seed)
    rng = np.random.default_rng(seed)
    B, k = len(lens), shape.k_rows
    mk = lambda h: torch.from_numpy(
        rng.standard_normal((B, k, h, shape.head_dim)).astype(np.float32)).cuda()
    q, kn, vn = mk(shape.n_q_heads), mk(shape.n_kv_heads), mk(shape.n_kv_heads)
    cache = sp.DeviceCache(w.cache)
    dims = sp.sp_attn_dims(shape.n_q_heads, shape.n_kv_heads, shape.head_dim, k, kv_dtype,
                           max(lens), 0)
    return shape, cache, dims, q, kn, vn


def _with_workspace(torch, dims, cache, q, kn, vn):
    B = q.shape[0]
    nbytes = sp.sp_attend_workspace_bytes(dims, B)
    ws = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    out = torch.empty(q.shape, dtype=torch.float32, device="cuda")
    sp.sp_attend(torch.cuda.current_stream(), dims, B, None, cache.seq_lens, cache.desc, q, kn,
                 vn, out, sp.SP_F32, ws, nbytes)
    return out


def _static(torch, dims, cache, q, kn, vn):
    out = torch.full(q.shape, float("nan"), dtype=torch.float32, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    sp.sp_attend_static(torch.cuda.current_stream(), dims, q.shape[0], None, cache.seq_lens,
                        cache.desc, q, kn, vn, out, sp.SP_F32, status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    return out


def test_static_scratch_matches_workspace_entry_point_on_consecutive_calls():
    torch = torch_dev()
    ensure_built()
    # two calls in a row with different lengths, so the second finds the
    # first call's partials left in the shared array
    for lens, seed in (([700, 3, 1500, 64], 11), ([17, 2100, 0], 12)):
        shape, cache, dims, q, kn, vn = _inputs(torch, lens, seed)
        ref = _with_workspace(torch, dims, cache, q, kn, vn).cpu().numpy()
        got = _static(torch, dims, cache, q, kn, vn).cpu().numpy()
        assert np.all(np.isfinite(got))
        np.testing.assert_allclose(got, ref, rtol=1e-4, atol=1e-4)


def test_static_scratch_rejects_batches_that_do_not_fit():
    torch = torch_dev()
    ensure_built()
    shape, cache, dims, q, kn, vn = _inputs(torch, [40, 50], 13)
    big = sp.sp_attn_dims(shape.n_q_heads, shape.n_kv_heads, shape.head_dim, shape.k_rows,
                          wl.BF16, 1 << 20, 64)          # a split plan far beyond 32 MiB
    assert sp.sp_attend_workspace_bytes(big, 2) > (32 << 20)
    with pytest.raises(sp.SpError) as e:
        sp.sp_attend_static(None, big, 2, None, cache.seq_lens, cache.desc, q, kn, vn,
                            torch.empty_like(q), sp.SP_F32)
    assert e.value.status == sp.SP_ERR_INVALID_ARG
    assert "static" in sp.sp_last_error()


def test_static_scratch_calls_after_the_first_allocate_nothing():
    torch = torch_dev()
    ensure_built()
    shape, cache, dims, q, kn, vn = _inputs(torch, [300, 1200, 5], 14)
    out = torch.empty(q.shape, dtype=torch.float32, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")

    def call():
        sp.sp_attend_static(torch.cuda.current_stream(), dims, q.shape[0], None, cache.seq_lens,
                            cache.desc, q, kn, vn, out, sp.SP_F32, status)

    call()  # the first call on the device may load the module holding the array
    torch.cuda.synchronize()
    gc.collect()  # tensors of earlier tests must not be freed inside the window
    free0, _ = torch.cuda.mem_get_info()
    alloc0 = torch.cuda.memory_allocated()
    for _ in range(3):
        call()
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    # neither torch's allocator nor the driver gave out memory for these calls
    assert torch.cuda.memory_allocated() <= alloc0
    assert free1 >= free0
    assert int(status.item()) == 0
