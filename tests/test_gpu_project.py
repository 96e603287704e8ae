"""The projection step (Y = X W^T, the decoder layer's linear maps) through the
C ABI, tensor-core and CUDA-core paths, against a plain fp64 matmul."""
import numpy as np
import pytest

import paper_2608_28099_gb300 as sp
from paper_2608_28099_gb300 import workloads as wl
from gpu_util import ensure_built, torch_dev

pytestmark = pytest.mark.gpu

SHAPES = [(1, 128, 64), (5, 256, 192), (16, 128, 2560), (17, 384, 640), (64, 128, 128),
          (100, 256, 4096), (128, 6144, 2560), (129, 128, 256), (300, 256, 1024),
          (1024, 512, 4096),
          # tile counts that fill the SMs badly take the persistent stream-K
          # schedule (two partial planes, zero-filled where a tile has one
          # segment; several row tiles)
          (1, 24576, 4096), (20, 20480, 256), (512, 6144, 4096),
          # partial warps of rows, one k-block, a gate/up-sized product
          (33, 2560, 9728), (127, 256, 64), (128, 19456, 2560)]


def run(M, N, K, path, seed):
    torch = torch_dev()
    ensure_built()
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((M, K)).astype(np.float32)
    wbits = wl.f32_to_bf16_bits((0.02 * rng.standard_normal((N, K))).astype(np.float32))
    ref = x.astype(np.float64) @ wl.bf16_bits_to_f32(wbits).astype(np.float64).T
    xt = torch.from_numpy(x).cuda()
    wt = torch.from_numpy(wbits.view(np.int16)).cuda()
    yt = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
    nbytes = sp.sp_project_workspace_bytes(M, N, K)
    ws = torch.empty(max(nbytes, 256), dtype=torch.uint8, device="cuda")
    sp.sp_project(torch.cuda.current_stream(), M, N, K, xt, wt, yt, path, ws, nbytes)
    torch.cuda.synchronize()
    return yt.cpu().numpy().astype(np.float64), ref


@pytest.mark.parametrize("M,N,K", SHAPES)
def test_tensor_core_projection(M, N, K):
    y, ref = run(M, N, K, 2, M * 7 + N + K)
    scale = np.max(np.abs(ref))
    assert np.all(np.isfinite(y))
    # bf16 hi+lo activations carry ~16 mantissa bits; fp32 accumulation
    assert np.max(np.abs(y - ref)) <= 2e-5 * scale * max(1.0, np.sqrt(K / 256)), \
        np.max(np.abs(y - ref)) / scale


@pytest.mark.parametrize("M,N,K", SHAPES[:6])
def test_cuda_core_projection(M, N, K):
    y, ref = run(M, N, K, 1, M + N + K)
    assert np.max(np.abs(y - ref)) <= 1e-5 * np.max(np.abs(ref)) * max(1.0, np.sqrt(K / 256))


def test_tensor_path_rejects_unsupported_shapes():
    torch = torch_dev()
    ensure_built()
    x = torch.zeros((4, 96), device="cuda")
    w = torch.zeros((100, 96), dtype=torch.int16, device="cuda")
    y = torch.zeros((4, 100), device="cuda")
    with pytest.raises(sp.SpError) as e:
        sp.sp_project(None, 4, 100, 96, x, w, y, 2, None, 0)
    assert e.value.status == sp.SP_ERR_UNSUPPORTED
