"""Python binding of libsp.so, the Speculative Probing classify path on GB300.

Argument marshalling only: every step of the path runs in the library's CUDA
kernels.  The functions carry the C names (``sp_create``, ``sp_classify``,
``sp_classify_host``, ``sp_attend`` ...).  PyTorch provides device memory and
streams; tensors are passed by ``data_ptr()``.  There is no fallback: if the
library has not been built, every call raises.
"""
from __future__ import annotations

import ctypes as C
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "_build", "libsp.so")

SP_OK, SP_ERR_INVALID_ARG, SP_ERR_UNSUPPORTED, SP_ERR_CUDA, SP_ERR_OOM, SP_ERR_DEVICE_STATUS = range(6)
SP_F32, SP_BF16 = 0, 1
SP_POOL_MEAN, SP_POOL_LAST = 0, 1
SP_KV_CONTIGUOUS, SP_KV_PAGED = 0, 1
SP_DEV_BAD_SEQ_ID, SP_DEV_BAD_LENGTH, SP_DEV_BAD_PAGE, SP_DEV_TIMEOUT = 1, 2, 4, 8
SP_OPT_SPLIT_TOKENS, SP_OPT_GEMM_PATH, SP_OPT_ATTN_PATH, SP_OPT_PROFILE = 1, 2, 3, 4
SP_OPT_RECURSIVE = 5
SP_OPT_ATTN_SEG_COST = 6
SP_OPT_ACT_PRECISION = 7
SP_OPT_DEBUG_STALL = 8
SP_OPT_GEMM_SCHEDULE = 9
SP_OPT_ATTN_MERGE = 10
SP_OPT_QUERY_PRECISION = 11
STAGES = ["input_norm", "qkv", "rope", "attention", "merge", "o_proj", "post_norm", "gate_up",
          "swiglu", "down", "readout", "fusion"]

EXPORTED = ["sp_create", "sp_destroy", "sp_classify", "sp_classify_host", "sp_check_status",
            "sp_last_error", "sp_set_option", "sp_last_launch_count", "sp_attend_workspace_bytes",
            "sp_attend", "sp_stage_times", "sp_project_workspace_bytes", "sp_project",
            "sp_attend_static", "sp_classify_hidden", "sp_classify_hidden_host",
            "sp_debug_gathered_pages", "sp_debug_gemm_plan"]


class sp_config(C.Structure):
    _fields_ = [("d_model", C.c_int), ("n_q_heads", C.c_int), ("n_kv_heads", C.c_int),
                ("head_dim", C.c_int), ("d_ff", C.c_int), ("k_rows", C.c_int),
                ("n_classes", C.c_int), ("rope_theta", C.c_float), ("rms_eps", C.c_float),
                ("pool", C.c_int), ("w_dtype", C.c_int), ("kv_dtype", C.c_int),
                ("max_batch", C.c_int), ("max_seq_len", C.c_int), ("n_tasks", C.c_int)]


class sp_weights(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in ("w_q", "w_k", "w_v", "w_o", "w_gate", "w_up", "w_down",
                                           "g_in", "g_post", "soft_prompt", "head_w", "head_b",
                                           "w_fc", "g_h", "g_e", "g_final")]


class sp_kv_cache(C.Structure):
    _fields_ = [("layout", C.c_int), ("k_seq", C.c_void_p), ("v_seq", C.c_void_p),
                ("k_pool", C.c_void_p), ("v_pool", C.c_void_p), ("page_table", C.c_void_p),
                ("page_size", C.c_int), ("n_pages", C.c_int), ("max_pages_per_seq", C.c_int),
                ("n_seqs", C.c_int)]


class sp_gemm_plan(C.Structure):
    _fields_ = [(n, C.c_int) for n in ("rows_per_tile", "m_tiles", "n_tiles", "n_kblocks",
                                       "tiles_per_cta", "persistent", "kblocks_per_cta", "splits",
                                       "grid")]


class sp_attn_dims(C.Structure):
    _fields_ = [("n_q_heads", C.c_int), ("n_kv_heads", C.c_int), ("head_dim", C.c_int),
                ("k_rows", C.c_int), ("kv_dtype", C.c_int), ("max_seq_len", C.c_int),
                ("split_tokens", C.c_int), ("path", C.c_int)]


class SpError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__(f"status {status}: {msg}")
        self.status = status


_lib = None


def load_library(path: str | None = None):
    """Load libsp.so (built in-tree by build_lib.build()); raises if absent."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = path or LIB_PATH
    if not os.path.exists(p):
        raise RuntimeError(f"{p} is missing: build the CUDA library first "
                           "(python -c 'import __graft_entry__ as g; g.build()')")
    lib = C.CDLL(p)
    vp, ip, i = C.c_void_p, C.POINTER(C.c_int), C.c_int
    lib.sp_create.argtypes = [C.POINTER(sp_config), C.POINTER(sp_weights), C.POINTER(C.c_void_p)]
    lib.sp_destroy.argtypes = [vp]
    lib.sp_classify.argtypes = [vp, vp, i, vp, vp, C.POINTER(sp_kv_cache), vp, vp]
    lib.sp_classify_host.argtypes = [vp, vp, i, vp, vp, C.POINTER(sp_kv_cache), vp, vp]
    lib.sp_classify_hidden.argtypes = [vp, vp, i, vp, vp, C.POINTER(sp_kv_cache), vp, vp]
    lib.sp_classify_hidden_host.argtypes = [vp, vp, i, vp, vp, C.POINTER(sp_kv_cache), vp, vp]
    lib.sp_check_status.argtypes = [vp, vp, ip]
    lib.sp_last_error.restype = C.c_char_p
    lib.sp_last_error.argtypes = []
    lib.sp_set_option.argtypes = [vp, i, i]
    lib.sp_last_launch_count.argtypes = [vp]
    lib.sp_last_launch_count.restype = C.c_int
    lib.sp_attend_workspace_bytes.argtypes = [C.POINTER(sp_attn_dims), i]
    lib.sp_attend_workspace_bytes.restype = C.c_size_t
    lib.sp_stage_times.argtypes = [vp, C.POINTER(C.c_float), i]
    lib.sp_project_workspace_bytes.argtypes = [i, i, i]
    lib.sp_project_workspace_bytes.restype = C.c_size_t
    lib.sp_project.argtypes = [vp, i, i, i, vp, vp, vp, i, vp, C.c_size_t]
    lib.sp_attend_static.argtypes = [vp, C.POINTER(sp_attn_dims), i, vp, vp,
                                     C.POINTER(sp_kv_cache), vp, vp, vp, vp, i, vp, vp]
    lib.sp_attend.argtypes = [vp, C.POINTER(sp_attn_dims), i, vp, vp, C.POINTER(sp_kv_cache), vp,
                              vp, vp, vp, i, vp, C.c_size_t, vp, vp]
    lib.sp_debug_gathered_pages.argtypes = [vp, vp, C.c_size_t]
    lib.sp_debug_gemm_plan.argtypes = [i, i, i, i, i, i, C.c_size_t, C.POINTER(sp_gemm_plan)]
    for name in EXPORTED:
        if name not in ("sp_last_error", "sp_last_launch_count", "sp_attend_workspace_bytes",
                        "sp_project_workspace_bytes"):
            getattr(lib, name).restype = C.c_int
    if path is None:
        _lib = lib
    return lib


def _check(status: int):
    if status != SP_OK:
        raise SpError(status, load_library().sp_last_error().decode())
    return status


def _ptr(t):
    """Device/host pointer of a torch tensor, numpy array, int or None."""
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if hasattr(t, "data_ptr"):
        return t.data_ptr()
    if hasattr(t, "ctypes"):
        return t.ctypes.data
    raise TypeError(type(t))


def _stream(stream):
    if stream is None:
        return None
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


# --------------------------------------------------------------------------- #
# the C entry points under their own names
# --------------------------------------------------------------------------- #
def sp_create(cfg: sp_config, weights: sp_weights) -> int:
    h = C.c_void_p()
    _check(load_library().sp_create(C.byref(cfg), C.byref(weights), C.byref(h)))
    return h.value


def sp_destroy(handle: int):
    _check(load_library().sp_destroy(handle))


def sp_classify(handle, stream, batch, seq_ids, seq_lens, kv: sp_kv_cache, rows, logits):
    _check(load_library().sp_classify(handle, _stream(stream), int(batch), _ptr(seq_ids),
                                      _ptr(seq_lens), C.byref(kv), _ptr(rows), _ptr(logits)))


def sp_classify_host(handle, stream, batch, seq_ids, seq_lens, kv: sp_kv_cache, rows, logits):
    _check(load_library().sp_classify_host(handle, _stream(stream), int(batch), _ptr(seq_ids),
                                           _ptr(seq_lens), C.byref(kv), _ptr(rows), _ptr(logits)))


def sp_classify_hidden(handle, stream, batch, seq_ids, seq_lens, kv: sp_kv_cache, hidden, logits):
    _check(load_library().sp_classify_hidden(handle, _stream(stream), int(batch), _ptr(seq_ids),
                                             _ptr(seq_lens), C.byref(kv), _ptr(hidden),
                                             _ptr(logits)))


def sp_classify_hidden_host(handle, stream, batch, seq_ids, seq_lens, kv: sp_kv_cache, hidden,
                            logits):
    _check(load_library().sp_classify_hidden_host(handle, _stream(stream), int(batch),
                                                  _ptr(seq_ids), _ptr(seq_lens), C.byref(kv),
                                                  _ptr(hidden), _ptr(logits)))


def sp_check_status(handle, stream=None) -> int:
    bits = C.c_int(0)
    st = load_library().sp_check_status(handle, _stream(stream), C.byref(bits))
    if st not in (SP_OK, SP_ERR_DEVICE_STATUS):
        _check(st)
    return bits.value


def sp_set_option(handle, key, value):
    _check(load_library().sp_set_option(handle, int(key), int(value)))


def sp_last_launch_count(handle) -> int:
    return load_library().sp_last_launch_count(handle)


def sp_debug_gathered_pages(handle, out=None):
    """Record the page ids the attention step of later classify calls reads
    into the int32 device tensor `out` ([batch][max_pages_per_seq]); None stops."""
    if out is None:
        _check(load_library().sp_debug_gathered_pages(handle, None, 0))
    else:
        _check(load_library().sp_debug_gathered_pages(handle, _ptr(out), out.numel()))


def sp_stage_times(handle) -> dict:
    ms = (C.c_float * len(STAGES))()
    _check(load_library().sp_stage_times(handle, ms, len(STAGES)))
    return {name: float(ms[i]) for i, name in enumerate(STAGES) if ms[i] >= 0}


def sp_attend_static(stream, dims, batch, seq_ids, seq_lens, kv, q, k_new, v_new, out, out_dtype,
                     status=None, gathered_pages=None):
    _check(load_library().sp_attend_static(_stream(stream), C.byref(dims), int(batch),
                                           _ptr(seq_ids), _ptr(seq_lens), C.byref(kv), _ptr(q),
                                           _ptr(k_new), _ptr(v_new), _ptr(out), int(out_dtype),
                                           _ptr(status), _ptr(gathered_pages)))


def sp_project_workspace_bytes(M, N, K) -> int:
    return load_library().sp_project_workspace_bytes(int(M), int(N), int(K))


def sp_debug_gemm_plan(M, N, K, n_sm, lo, schedule=0, capacity_bytes=None) -> dict:
    """The tensor-core projection plan for y[M][N] = x[M][K] W^T (host only)."""
    plan = sp_gemm_plan()
    cap = C.c_size_t(-1).value if capacity_bytes is None else int(capacity_bytes)
    _check(load_library().sp_debug_gemm_plan(int(M), int(N), int(K), int(n_sm), int(lo),
                                             int(schedule), cap, C.byref(plan)))
    return {name: getattr(plan, name) for name, _ in sp_gemm_plan._fields_}


def sp_project(stream, M, N, K, x, w, y, path, workspace, workspace_bytes):
    _check(load_library().sp_project(_stream(stream), int(M), int(N), int(K), _ptr(x), _ptr(w),
                                     _ptr(y), int(path), _ptr(workspace), int(workspace_bytes)))


def sp_last_error() -> str:
    return load_library().sp_last_error().decode()


def sp_attend_workspace_bytes(dims: sp_attn_dims, batch: int) -> int:
    return load_library().sp_attend_workspace_bytes(C.byref(dims), int(batch))


def sp_attend(stream, dims, batch, seq_ids, seq_lens, kv, q, k_new, v_new, out, out_dtype,
              workspace, workspace_bytes, status=None, gathered_pages=None):
    _check(load_library().sp_attend(_stream(stream), C.byref(dims), int(batch), _ptr(seq_ids),
                                    _ptr(seq_lens), C.byref(kv), _ptr(q), _ptr(k_new), _ptr(v_new),
                                    _ptr(out), int(out_dtype), _ptr(workspace),
                                    int(workspace_bytes), _ptr(status), _ptr(gathered_pages)))


# --------------------------------------------------------------------------- #
# marshalling helpers for the seeded workloads
# --------------------------------------------------------------------------- #
def make_config(shape, max_batch: int, max_seq_len: int) -> sp_config:
    return sp_config(shape.d_model, shape.n_q_heads, shape.n_kv_heads, shape.head_dim, shape.d_ff,
                     shape.k_rows, shape.n_classes, float(shape.rope_theta), float(shape.rms_eps),
                     shape.pool, shape.w_dtype, shape.kv_dtype, int(max_batch), int(max_seq_len),
                     int(getattr(shape, "n_tasks", 1)))


class Model:
    """An sp_handle built from host weight arrays (workloads.Weights)."""

    def __init__(self, shape, weights, max_batch: int, max_seq_len: int):
        import numpy as np
        self.shape = shape
        arrs = {}
        for name in ("w_q", "w_k", "w_v", "w_o", "w_gate", "w_up", "w_down", "soft_prompt"):
            arrs[name] = np.ascontiguousarray(getattr(weights, name))
        for name in ("g_in", "g_post", "head_w"):
            arrs[name] = np.ascontiguousarray(getattr(weights, name), dtype=np.float32)
        arrs["head_b"] = (None if weights.head_b is None
                          else np.ascontiguousarray(weights.head_b, dtype=np.float32))
        fc = getattr(weights, "w_fc", None)
        arrs["w_fc"] = None if fc is None else np.ascontiguousarray(fc)
        for name in ("g_h", "g_e"):
            arrs[name] = (None if fc is None
                          else np.ascontiguousarray(getattr(weights, name), dtype=np.float32))
        gf = getattr(weights, "g_final", None)
        arrs["g_final"] = None if gf is None else np.ascontiguousarray(gf, dtype=np.float32)
        self._arrs = arrs  # host copies stay alive for the handle's lifetime (read at create)
        w = sp_weights(*[None if arrs[n] is None else arrs[n].ctypes.data for n in (
            "w_q", "w_k", "w_v", "w_o", "w_gate", "w_up", "w_down", "g_in", "g_post",
            "soft_prompt", "head_w", "head_b", "w_fc", "g_h", "g_e", "g_final")])
        self.cfg = make_config(shape, max_batch, max_seq_len)
        self.handle = sp_create(self.cfg, w)

    def close(self):
        if self.handle:
            sp_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class DeviceCache:
    """A workloads.KVCache uploaded to torch device tensors, plus its sp_kv_cache."""

    def __init__(self, cache, device="cuda"):
        import numpy as np
        import torch
        self.host = cache

        def up(a):
            a = np.ascontiguousarray(a)
            if a.dtype == np.uint16:
                a = a.view(np.int16)
            return torch.from_numpy(a).to(device)

        self.seq_lens = torch.from_numpy(np.ascontiguousarray(cache.seq_lens, dtype=np.int32)).to(device)
        if cache.layout == SP_KV_CONTIGUOUS:
            self.k_flat = up(cache.k_flat)
            self.v_flat = up(cache.v_flat)
            es = 2 if cache.dtype == SP_BF16 else 4
            row = cache.k_flat.shape[1] * cache.k_flat.shape[2] * es
            kp = [self.k_flat.data_ptr() + int(o) * row for o in cache.offsets]
            vp = [self.v_flat.data_ptr() + int(o) * row for o in cache.offsets]
            self.k_ptrs = torch.tensor(kp, dtype=torch.int64, device=device)
            self.v_ptrs = torch.tensor(vp, dtype=torch.int64, device=device)
            self.desc = sp_kv_cache(SP_KV_CONTIGUOUS, self.k_ptrs.data_ptr(), self.v_ptrs.data_ptr(),
                                    None, None, None, cache.page_size, 0, 0, cache.n_seqs)
        else:
            self.k_pool = up(cache.k_pool)
            self.v_pool = up(cache.v_pool)
            self.page_table = torch.from_numpy(np.ascontiguousarray(cache.page_table)).to(device)
            self.desc = sp_kv_cache(SP_KV_PAGED, None, None, self.k_pool.data_ptr(),
                                    self.v_pool.data_ptr(), self.page_table.data_ptr(),
                                    cache.page_size, cache.n_pages, cache.max_pages, cache.n_seqs)

    def nbytes(self) -> int:
        ts = ([self.k_flat, self.v_flat] if self.host.layout == SP_KV_CONTIGUOUS
              else [self.k_pool, self.v_pool])
        return sum(t.numel() * t.element_size() for t in ts)


class DevicePagedCache:
    """sp_kv_cache over a workloads.DeviceWorkload's device-resident pools."""

    def __init__(self, dw, device="cuda"):
        import numpy as np
        import torch
        self.host = dw
        self.seq_lens = torch.from_numpy(np.ascontiguousarray(dw.seq_lens, dtype=np.int32)).to(device)
        self.page_table = torch.from_numpy(np.ascontiguousarray(dw.page_table)).to(device)
        self.k_pool, self.v_pool = dw.k_pool, dw.v_pool
        self.desc = sp_kv_cache(SP_KV_PAGED, None, None, self.k_pool.data_ptr(),
                                self.v_pool.data_ptr(), self.page_table.data_ptr(),
                                dw.shape.page_size, max(dw.n_pages, 1), dw.page_table.shape[1],
                                len(dw.seq_lens))

    def nbytes(self) -> int:
        return sum(t.numel() * t.element_size() for t in (self.k_pool, self.v_pool))
