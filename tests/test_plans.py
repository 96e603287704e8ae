"""Host-side projection planning (no GPU): the launch plans sp_classify and
sp_project take, through the sp_debug_gemm_plan hook."""
import itertools

import pytest

import paper_2608_28099_gb300 as sp
from paper_2608_28099_gb300 import build_lib


@pytest.fixture(scope="module", autouse=True)
def lib():
    build_lib.build()
    return sp.load_library()


def cdiv(a, b):
    return -(-a // b)


SHAPES = list(itertools.product([1, 5, 16, 33, 64, 100, 128, 129, 300, 1024, 4096],
                                [128, 640, 2560, 5120, 7168, 24576, 34816],
                                [64, 192, 2560, 5120, 17408]))


@pytest.mark.parametrize("n_sm", [152, 148, 20])
@pytest.mark.parametrize("lo", [0, 1])
@pytest.mark.parametrize("schedule", [0, 1, 2])
def test_every_plan_covers_the_product_exactly_once(n_sm, lo, schedule):
    for M, N, K in SHAPES:
        p = sp.sp_debug_gemm_plan(M, N, K, n_sm, lo, schedule)
        rt = p["rows_per_tile"]
        assert rt in (16, 32, 64, 128, 256)
        assert rt != 256 or (lo == 0 and M >= 256)          # N = 512 exceeds one MMA with lo
        assert p["m_tiles"] == cdiv(M, rt)
        assert p["n_tiles"] == N // 128 and p["n_kblocks"] == K // 64
        tiles, nkb, kpc = p["m_tiles"] * p["n_tiles"], p["n_kblocks"], p["kblocks_per_cta"]
        assert p["splits"] >= 1 and kpc >= 1
        if p["persistent"]:
            assert schedule != 1
            units = tiles * nkb
            assert kpc >= 2
            assert p["grid"] * kpc >= units > (p["grid"] - 1) * kpc   # every unit, no idle CTA
            assert p["tiles_per_cta"] == 1
        else:
            # K splits: every k-block in exactly one split, no empty split
            assert kpc * (p["splits"] - 1) < nkb <= kpc * p["splits"]
            tpc = p["tiles_per_cta"]
            assert tpc in (1, 2)
            assert p["grid"] == p["m_tiles"] * (p["n_tiles"] // tpc) * p["splits"]
            if tpc == 2:
                assert schedule == 0 and lo == 0 and rt <= 128 and p["n_tiles"] % 2 == 0
                assert p["grid"] <= n_sm
            if p["splits"] > 1:
                assert p["grid"] <= n_sm        # K is split only to fill one wave
        if schedule == 2:
            assert p["persistent"] == 1


def test_partial_planes_respect_the_capacity():
    for M, N, K in SHAPES:
        one_plane = M * N * 4
        for lo in (0, 1):
            p = sp.sp_debug_gemm_plan(M, N, K, 152, lo, 0, one_plane)
            assert p["splits"] == 1
            q = sp.sp_debug_gemm_plan(M, N, K, 152, lo, 0, 3 * one_plane)
            assert q["splits"] <= 3


def test_named_layer_plans():
    # the plans the launch lists and kernel summaries describe (152 SMs)
    def plan(M, N, K, lo):
        p = sp.sp_debug_gemm_plan(M, N, K, 152, lo, 0)
        return (p["rows_per_tile"], p["tiles_per_cta"], p["persistent"], p["splits"], p["grid"])
    # 27B-class, 8 sequences x 16 rows: Q/K/V and output hi + lo, split over K
    assert plan(128, 7168, 5120, 1) == (128, 1, 0, 2, 112)
    assert plan(128, 5120, 5120, 1) == (128, 1, 0, 3, 120)
    # gate/up plain bf16: two weight tiles per CTA and no K split (the SwiGLU
    # epilogue's condition); down plain bf16 over three K splits
    assert plan(128, 34816, 5120, 0) == (128, 2, 0, 1, 136)
    assert plan(128, 5120, 17408, 0) == (128, 1, 0, 3, 120)
    # 8B-class at 1024 rows: Q/K/V one CTA per (row tile, head), no K split (the
    # rotation epilogue's condition); gate/up plain on 256-row tiles
    assert plan(1024, 6144, 4096, 1) == (128, 1, 0, 1, 384)
    assert plan(1024, 24576, 4096, 0)[:4] == (256, 1, 0, 1)
    # one row against a wide weight: the persistent stream-K schedule
    assert plan(1, 24576, 4096, 1)[2] == 1


def test_plan_query_rejects_bad_arguments():
    with pytest.raises(sp.SpError) as e:
        sp.sp_debug_gemm_plan(4, 100, 96, 152, 1)
    assert e.value.status == sp.SP_ERR_UNSUPPORTED
    for args in [(0, 128, 64, 152, 1), (4, 128, 64, 0, 1), (4, 128, 64, 152, 2),
                 (4, 128, 64, 152, 1, 3)]:
        with pytest.raises(sp.SpError) as e:
            sp.sp_debug_gemm_plan(*args)
        assert e.value.status == sp.SP_ERR_INVALID_ARG
