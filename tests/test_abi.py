"""The C-ABI library builds, loads without a GPU, exports every symbol that
include/sp.h declares, and rejects bad arguments on the host before touching
the device."""
import ctypes as C
import os
import re

import numpy as np
import pytest

import paper_2608_28099_gb300 as sp
from paper_2608_28099_gb300 import build_lib
from paper_2608_28099_gb300 import workloads as wl

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_symbols():
    names = []
    for h in os.listdir(os.path.join(ROOT, "include")):
        if h.endswith(".h"):
            text = open(os.path.join(ROOT, "include", h)).read()
            names += re.findall(r"^SP_API\s+[\w\s\*]*?\b(sp_\w+)\s*\(", text, flags=re.M)
    return sorted(set(names))


@pytest.fixture(scope="module")
def lib():
    build_lib.build()
    return sp.load_library()


def header_constants():
    """Every `SP_NAME = value` of the enums in include/sp.h."""
    text = open(os.path.join(ROOT, "include", "sp.h")).read()
    text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
    return {m.group(1): int(m.group(2)) for m in re.finditer(r"\b(SP_[A-Z0-9_]+)\s*=\s*(-?\d+)", text)}


def test_binding_constants_match_the_header():
    consts = header_constants()
    assert len(consts) > 30
    for name, value in consts.items():
        if name.startswith(("SP_OPT_", "SP_STAGE_", "SP_DEV_", "SP_ERR_", "SP_OK", "SP_POOL_",
                            "SP_KV_", "SP_F32", "SP_BF16")) and name != "SP_N_STAGES":
            assert hasattr(sp, name) or name.startswith("SP_STAGE_"), name
            if hasattr(sp, name):
                assert getattr(sp, name) == value, name
    stages = sorted((v, n) for n, v in consts.items() if n.startswith("SP_STAGE_"))
    header_names = [n[len("SP_STAGE_"):].lower() for _, n in stages]
    assert [{"attn": "attention"}.get(x, x) for x in header_names] == sp.STAGES
    assert consts["SP_N_STAGES"] == len(sp.STAGES)


def test_every_declared_symbol_is_exported(lib):
    names = declared_symbols()
    assert len(names) >= 10
    for n in names:
        assert hasattr(lib, n), n
    assert set(sp.EXPORTED) <= set(names)


def _cfg(**over):
    shape = wl.named("tiny").shape
    c = sp.make_config(shape, 4, 128)
    for k, v in over.items():
        setattr(c, k, v)
    return c


@pytest.mark.parametrize("field,value,status", [
    ("head_dim", 96, sp.SP_ERR_UNSUPPORTED),
    ("n_q_heads", 3, sp.SP_ERR_INVALID_ARG),
    ("k_rows", 0, sp.SP_ERR_INVALID_ARG),
    ("k_rows", 33, sp.SP_ERR_INVALID_ARG),
    ("d_model", 100, sp.SP_ERR_INVALID_ARG),
    ("max_batch", 0, sp.SP_ERR_INVALID_ARG),
    ("pool", 7, sp.SP_ERR_INVALID_ARG),
    ("kv_dtype", 5, sp.SP_ERR_INVALID_ARG),
])
def test_create_rejects_bad_config_on_host(lib, field, value, status):
    h = C.c_void_p(123)
    w = sp.sp_weights()
    st = lib.sp_create(C.byref(_cfg(**{field: value})), C.byref(w), C.byref(h))
    assert st == status
    assert h.value is None
    assert lib.sp_last_error()


def test_create_rejects_missing_weights_on_host(lib):
    h = C.c_void_p()
    w = sp.sp_weights()
    assert lib.sp_create(C.byref(_cfg()), C.byref(w), C.byref(h)) == sp.SP_ERR_INVALID_ARG
    assert b"weight" in lib.sp_last_error()


def test_null_handle_calls_fail_cleanly(lib):
    kv = sp.sp_kv_cache()
    assert lib.sp_classify(None, None, 1, None, None, C.byref(kv), None, None) == sp.SP_ERR_INVALID_ARG
    assert lib.sp_set_option(None, 1, 0) == sp.SP_ERR_INVALID_ARG
    assert lib.sp_destroy(None) == sp.SP_OK
    assert lib.sp_last_launch_count(None) == -1
    assert lib.sp_debug_gathered_pages(None, None, 0) == sp.SP_ERR_INVALID_ARG


def test_attend_rejects_bad_dims_on_host(lib):
    kv = sp.sp_kv_cache()
    dims = sp.sp_attn_dims(4, 3, 32, 4, sp.SP_F32, 64, 0)    # 4 q heads over 3 kv heads
    st = lib.sp_attend(None, C.byref(dims), 1, None, None, C.byref(kv), None, None, None, None, 0,
                       None, 0, None, None)
    assert st == sp.SP_ERR_INVALID_ARG
    dims = sp.sp_attn_dims(4, 2, 32, 4, sp.SP_F32, 64, 100)   # split not a multiple of 64
    assert lib.sp_attend_workspace_bytes(C.byref(dims), 1) == 0


@pytest.mark.parametrize("bad", ["q", "k_new", "v_new", "out"])
def test_attend_rejects_misaligned_vectors_on_host(lib, bad):
    # the kernels move whole 16-byte vectors: a pointer off by 4 bytes is refused
    # before any launch (the fake addresses are never dereferenced)
    kv = sp.sp_kv_cache()
    dims = sp.sp_attn_dims(4, 2, 128, 4, sp.SP_BF16, 64, 0)
    ptr = {n: C.c_void_p(0x100000 * (i + 1)) for i, n in enumerate(["q", "k_new", "v_new", "out"])}
    ptr[bad] = C.c_void_p(ptr[bad].value + 4)
    lens, ws = C.c_void_p(0x900000), C.c_void_p(0xA00000)
    st = lib.sp_attend(None, C.byref(dims), 1, None, lens, C.byref(kv), ptr["q"], ptr["k_new"],
                       ptr["v_new"], ptr["out"], sp.SP_F32, ws, 1 << 20, None, None)
    assert st == sp.SP_ERR_INVALID_ARG
    assert "16-byte aligned" in sp.sp_last_error()


@pytest.mark.parametrize("bad", ["x", "w"])
def test_project_rejects_misaligned_operands_on_host(lib, bad):
    # X and W are read by TMA when the tensor path runs: 16-byte aligned or refused
    x, w, y = C.c_void_p(0x100000), C.c_void_p(0x200000), C.c_void_p(0x300000)
    if bad == "x":
        x = C.c_void_p(x.value + 8)
    else:
        w = C.c_void_p(w.value + 8)
    st = lib.sp_project(None, 128, 256, 128, x, w, y, 0, C.c_void_p(0x400000), 1 << 24)
    assert st == sp.SP_ERR_INVALID_ARG
    assert "16-byte aligned" in sp.sp_last_error()


def test_attend_rejects_misaligned_pools_on_host(lib):
    kv = sp.sp_kv_cache(sp.SP_KV_PAGED, None, None, 0x600008, 0x700000, 0x500000, 16, 4, 4, 1)
    dims = sp.sp_attn_dims(4, 2, 128, 4, sp.SP_BF16, 64, 0)
    q, kn, vn, out = (C.c_void_p(0x100000 * i) for i in range(1, 5))
    st = lib.sp_attend(None, C.byref(dims), 1, None, C.c_void_p(0x900000), C.byref(kv), q, kn, vn,
                       out, sp.SP_F32, C.c_void_p(0xA00000), 1 << 20, None, None)
    assert st == sp.SP_ERR_INVALID_ARG
    assert "k_pool and v_pool" in sp.sp_last_error()


def test_attend_rejects_negative_max_seq_len_on_host(lib):
    # a negative bound would clamp lengths to a negative value on the device
    kv = sp.sp_kv_cache(sp.SP_KV_PAGED, None, None, 0x600000, 0x700000, 0x500000, 16, 4, 4, 1)
    dims = sp.sp_attn_dims(4, 2, 128, 4, sp.SP_BF16, -1, 0)
    q, kn, vn, out = (C.c_void_p(0x100000 * i) for i in range(1, 5))
    st = lib.sp_attend(None, C.byref(dims), 1, None, C.c_void_p(0x900000), C.byref(kv), q, kn, vn,
                       out, sp.SP_F32, C.c_void_p(0xA00000), 1 << 20, None, None)
    assert st == sp.SP_ERR_INVALID_ARG
    assert "max_seq_len" in sp.sp_last_error()
    assert lib.sp_attend_workspace_bytes(C.byref(dims), 1) == 0


def test_attend_static_rejects_invalid_dims_on_host(lib):
    kv = sp.sp_kv_cache(sp.SP_KV_PAGED, None, None, 0x600000, 0x700000, 0x500000, 16, 4, 4, 1)
    dims = sp.sp_attn_dims(4, 2, 128, 4, sp.SP_BF16, -1, 0)
    q, kn, vn, out = (C.c_void_p(0x100000 * i) for i in range(1, 5))
    st = lib.sp_attend_static(None, C.byref(dims), 1, None, C.c_void_p(0x900000), C.byref(kv), q,
                              kn, vn, out, sp.SP_F32, None, None)
    assert st == sp.SP_ERR_INVALID_ARG
    assert "invalid attention dims" in sp.sp_last_error()
