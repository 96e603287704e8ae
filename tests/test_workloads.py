"""Host logic of the seeded input generator (no method arithmetic)."""
import numpy as np
import pytest

from paper_2608_28099_gb300 import workloads as wl


def test_bf16_round_trip_and_rne():
    x = np.array([1.0, -2.5, 3.0e-3, 1.00390625, 1.01171875], dtype=np.float32)
    b = wl.f32_to_bf16_bits(x)
    y = wl.bf16_bits_to_f32(b)
    # exactly representable values survive; ties round to even mantissa
    assert y[0] == 1.0 and y[1] == -2.5
    assert y[3] == 1.0          # 1 + 2^-8 is a tie -> even (1.0)
    assert y[4] == 1.015625     # 1 + 3*2^-8 is a tie -> even (1 + 2^-6)
    assert abs(y[2] - 3.0e-3) <= 3.0e-3 * 2 ** -8


def test_generation_is_deterministic():
    a = wl.generate(wl.named("tiny"))
    b = wl.generate(wl.named("tiny"))
    assert np.array_equal(a.weights.w_q, b.weights.w_q)
    assert np.array_equal(a.cache.k_flat, b.cache.k_flat)
    assert a.cache.k_flat.shape == (64, 2, 32) and a.cache.k_flat.dtype == np.float32


def test_paged_layout_holds_the_logical_tokens():
    sh = wl.Shape(64, 4, 2, 16, 64, 2, 2)
    w = wl.custom(sh, [0, 3, 16, 17, 50], wl.LAYOUT_CONTIGUOUS, 3)
    p = wl.contiguous_to_paged(w.cache, 16, 9)
    assert p.page_table.shape == (5, 4)
    used = p.page_table[p.page_table >= 0]
    assert sorted(used.tolist()) == list(range(p.n_pages))       # a permutation
    for b, L in enumerate(w.cache.seq_lens):
        o = int(w.cache.offsets[b])
        for t in range(int(L)):
            page, slot = p.page_table[b, t // 16], t % 16
            assert np.array_equal(p.k_pool[page, :, slot, :], w.cache.k_flat[o + t])
            assert np.array_equal(p.v_pool[page, :, slot, :], w.cache.v_flat[o + t])
        assert np.all(p.page_table[b, (int(L) + 15) // 16:] == -1)


def test_named_shapes():
    s = wl.named("8b_paged")
    assert (s.batch, s.shape.d_model, s.shape.k_rows, s.shape.n_classes) == (64, 4096, 16, 4)
    s = wl.named("sweep_B8_L2048_k4_C16")
    assert (s.batch, s.len_lo, s.len_hi, s.shape.k_rows, s.shape.n_classes) == (8, 1536, 2560, 4, 16)
    assert len(wl.SWEEP_POINTS) == 160


def test_device_generator_matches_host_structure():
    """The device-drawn sweep inputs share lengths, page table, weights and rows
    with generate(); host_cache() hands back exactly the pooled pages."""
    torch = pytest.importorskip("torch")
    spec = wl.named("sweep_B8_L512_k4_C2", rows_per_seq=True)
    host = wl.generate(spec)
    dev = wl.generate_on_device(spec, device="cpu")
    assert np.array_equal(dev.seq_lens, host.cache.seq_lens)
    assert np.array_equal(dev.page_table, host.cache.page_table)
    assert dev.n_pages == host.cache.n_pages
    assert np.array_equal(dev.weights.w_down, host.weights.w_down)
    assert np.array_equal(dev.rows, host.rows)
    ids = [5, 2]
    hc = dev.host_cache(ids)
    kp = dev.k_pool.numpy().view(np.uint16)
    for j, b in enumerate(ids):
        L = int(dev.seq_lens[b])
        assert hc.seq_lens[j] == L
        for t in range(0, L, 7):
            src = kp[dev.page_table[b, t // 16], :, t % 16, :]
            assert np.array_equal(hc.k_pool[hc.page_table[j, t // 16], :, t % 16, :], src)
    # N(0, 1) values
    vals = wl.bf16_bits_to_f32(kp[:64].reshape(-1))
    assert abs(float(vals.mean())) < 0.05 and abs(float(vals.std()) - 1.0) < 0.05
