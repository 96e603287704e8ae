"""Helpers shared by the GPU tests: run a seeded workload through the C ABI and
through the fp64 oracle, and compare them."""
from __future__ import annotations

import functools

import numpy as np

import oracle.sp_oracle as so
import paper_2608_28099_gb300 as sp
from paper_2608_28099_gb300 import build_lib
from paper_2608_28099_gb300 import workloads as wl

# Tolerance for bf16 inputs with fp32 accumulation: |gpu - oracle| <= ATOL + RTOL |oracle|.
ATOL, RTOL = 2e-2, 1e-2


@functools.lru_cache(maxsize=None)
def ensure_built():
    build_lib.build()
    return sp.load_library()


def torch_dev():
    import torch
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return torch


def rows_tensor(torch, rows):
    if rows is None:
        return None
    a = np.ascontiguousarray(rows)
    if a.dtype == np.uint16:
        a = a.view(np.int16)
    return torch.from_numpy(a).cuda()


class GpuRun:
    """A model + uploaded cache for one workload, callable repeatedly."""

    def __init__(self, w: wl.Workload, max_batch=None, max_seq_len=None, options=None):
        ensure_built()
        torch = torch_dev()
        self.torch = torch
        self.w = w
        lens = w.cache.seq_lens
        self.model = sp.Model(w.shape, w.weights, max_batch or len(w.seq_ids),
                              max_seq_len if max_seq_len is not None else int(lens.max(initial=0)))
        for k, v in (options or {}).items():
            sp.sp_set_option(self.model.handle, k, v)
        self.cache = sp.DeviceCache(w.cache)
        self.ids = torch.from_numpy(np.ascontiguousarray(w.seq_ids, dtype=np.int32)).cuda()
        self.rows = rows_tensor(torch, w.rows)

    def logits(self, use_rows=True, ids=None, lens=None):
        torch = self.torch
        B = len(self.w.seq_ids) if ids is None else len(ids)
        ids_t = self.ids if ids is None else torch.as_tensor(np.asarray(ids, np.int32)).cuda()
        out = torch.empty((B, self.w.shape.n_classes), dtype=torch.float32, device="cuda")
        sp.sp_classify(self.model.handle, torch.cuda.current_stream(), B, ids_t,
                       self.cache.seq_lens if lens is None else lens, self.cache.desc,
                       self.rows if use_rows else None, out)
        torch.cuda.synchronize()
        bits = sp.sp_check_status(self.model.handle)
        assert bits == 0, f"device status {bits}: {sp.sp_last_error()}"
        return out.cpu().numpy().astype(np.float64)

    def close(self):
        self.model.close()


def oracle_logits(w: wl.Workload, use_rows=True, ids=None) -> np.ndarray:
    layer = so.Layer(w.shape, w.weights)
    seq_ids = w.seq_ids if ids is None else np.asarray(ids)
    rows = w.rows if (use_rows and w.rows is not None) else None
    if rows is not None and ids is not None:
        rows = rows[np.asarray(ids)]
    return so.classify(layer, w.cache, seq_ids, rows)


def compare(gpu: np.ndarray, ref: np.ndarray, atol=ATOL, rtol=RTOL, label=""):
    """Element-wise tolerance plus argmax agreement away from near-ties."""
    err = np.abs(gpu - ref)
    bound = atol + rtol * np.abs(ref)
    worst = np.unravel_index(np.argmax(err - bound), err.shape)
    assert np.all(err <= bound), (f"{label}: max err {err.max():.3e} at {worst} "
                                  f"(gpu {gpu[worst]:.6f} ref {ref[worst]:.6f})")
    if ref.shape[1] > 1:
        srt = np.sort(ref, axis=1)
        margin = srt[:, -1] - srt[:, -2]
        decisive = margin > 2 * (atol + rtol * np.abs(srt[:, -1]))
        agree = np.argmax(gpu, axis=1) == np.argmax(ref, axis=1)
        assert np.all(agree[decisive]), f"{label}: argmax disagrees on a decisive row"
        return float(err.max()), float(np.mean(agree))
    return float(err.max()), 1.0
