"""Pins of the fp64 oracle against facts fixed outside the oracle itself.

Each ``check_*`` function raises AssertionError when the oracle disagrees with
a hand-derived fixture (tests/golden), a closed form, an invariant, a special
case that reduces to something simpler, or an independent library routine.
``test_planted_mistakes_are_caught`` plants plausible mistakes in the oracle
(on the CPU) and asserts that at least one check fails for each of them.
"""
import dataclasses
import hashlib
import math

import numpy as np
import pytest

import oracle.sp_oracle as so
from conftest import read_golden
from paper_2608_28099_gb300 import workloads as wl


# --------------------------------------------------------------------------- #
# helpers (no method arithmetic: only build inputs)
# --------------------------------------------------------------------------- #
@dataclasses.dataclass
class W:
    w_q: np.ndarray
    w_k: np.ndarray
    w_v: np.ndarray
    w_o: np.ndarray
    w_gate: np.ndarray
    w_up: np.ndarray
    w_down: np.ndarray
    g_in: np.ndarray
    g_post: np.ndarray
    soft_prompt: np.ndarray
    head_w: np.ndarray
    head_b: np.ndarray = None
    g_final: np.ndarray = None  # final norm before an LM-head readout (optional)
    w_fc: np.ndarray = None    # input fusion (optional)
    g_h: np.ndarray = None
    g_e: np.ndarray = None


def f32(a):
    return np.asarray(a, dtype=np.float32)


def random_layer(seed, d=16, hq=4, hkv=2, dh=8, f=24, k=3, C=3, pool=wl.POOL_MEAN, eps=1e-6):
    rng = np.random.default_rng(seed)
    sh = wl.Shape(d, hq, hkv, dh, f, k, C, rope_theta=100.0, rms_eps=eps,
                  w_dtype=wl.F32, kv_dtype=wl.F32, pool=pool)
    n = lambda *s: f32(rng.standard_normal(s) * 0.4)
    w = W(n(hq * dh, d), n(hkv * dh, d), n(hkv * dh, d), n(d, hq * dh), n(f, d), n(f, d), n(d, f),
          f32(1 + 0.1 * rng.standard_normal(d)), f32(1 + 0.1 * rng.standard_normal(d)),
          n(k, d), n(C, d), f32(rng.standard_normal(C)))
    return sh, w


def hand_layer():
    sh = wl.Shape(2, 1, 1, 2, 1, 1, 2, rope_theta=10000.0, rms_eps=0.0,
                  w_dtype=wl.F32, kv_dtype=wl.F32, pool=wl.POOL_LAST)
    I2 = f32(np.eye(2))
    w = W(I2, I2, I2, I2, f32([[1, 0]]), f32([[0, 1]]), f32([[1], [0]]),
          f32([1, 1]), f32([1, 1]), f32([[1, 1]]), np.eye(2), None)
    return sh, w


# --------------------------------------------------------------------------- #
# checks
# --------------------------------------------------------------------------- #
def check_hand_example():
    g = read_golden("hand_example_L2_k1.txt")
    sh, w = hand_layer()
    layer = so.Layer(sh, w)
    kc = np.array([[[1.0, 0.0]], [[0.0, 1.0]]])
    vc = kc.copy()
    tr = {}
    h2 = layer.rows_with_cache(layer.soft_prompt, kc, vc, trace=tr)
    np.testing.assert_allclose(tr["q"].ravel(), g["q"], atol=1e-9)
    np.testing.assert_allclose(tr["k_new"].ravel(), g["q"], atol=1e-9)
    np.testing.assert_allclose(tr["p"].ravel(), g["p"], atol=1e-9)
    np.testing.assert_allclose(tr["o"].ravel(), g["o"], atol=1e-9)
    np.testing.assert_allclose(layer.readout(h2), g["logits"], atol=1e-9)


def check_rope_pairs():
    g = read_golden("rope_pairs_dh4.txt")
    x = np.eye(4)[:3].reshape(3, 1, 1, 4)            # three inputs, T=1, H=1
    y = np.stack([so.rope(x[i], np.array([1]), 1.0e4) for i in range(3)]).reshape(3, 4)
    np.testing.assert_allclose(y[0], g["e0"], atol=1e-12)
    np.testing.assert_allclose(y[1], g["e1"], atol=1e-12)
    np.testing.assert_allclose(y[2], g["e2"], atol=1e-12)


def check_rope_relative_and_norm():
    """Rotation keeps norms and the score depends on position differences only."""
    rng = np.random.default_rng(5)
    q = rng.standard_normal((1, 1, 8))
    k = rng.standard_normal((1, 1, 8))
    np.testing.assert_allclose(np.linalg.norm(so.rope(q, np.array([37]), 100.0)), np.linalg.norm(q),
                               rtol=1e-12)
    s1 = np.sum(so.rope(q, np.array([40]), 100.0) * so.rope(k, np.array([33]), 100.0))
    s2 = np.sum(so.rope(q, np.array([107]), 100.0) * so.rope(k, np.array([100]), 100.0))
    np.testing.assert_allclose(s1, s2, rtol=1e-10)


def check_rope_frequencies_follow_theta():
    """Pair i turns by p * theta^(-2i/dh): at theta = 100, p = 3, dh = 4 pair 0
    turns 3 rad and pair 1 turns 3 / 10 = 0.3 rad; at dh = 8 pair 3 turns
    3 * 100^(-3/4) rad (closed forms from the definition of the frequencies)."""
    e0, e1 = np.eye(4)[0].reshape(1, 1, 4), np.eye(4)[1].reshape(1, 1, 4)
    np.testing.assert_allclose(so.rope(e0, np.array([3]), 100.0).ravel(),
                               [math.cos(3.0), 0.0, math.sin(3.0), 0.0], atol=1e-12)
    np.testing.assert_allclose(so.rope(e1, np.array([3]), 100.0).ravel(),
                               [0.0, math.cos(0.3), 0.0, math.sin(0.3)], atol=1e-12)
    e3 = np.eye(8)[3].reshape(1, 1, 8)
    a = 3.0 * 100.0 ** -0.75
    np.testing.assert_allclose(so.rope(e3, np.array([3]), 100.0).ravel(),
                               [0, 0, 0, math.cos(a), 0, 0, 0, math.sin(a)], atol=1e-12)


def check_softmax_rows_sum_to_one():
    sh, w = random_layer(1)
    layer = so.Layer(sh, w)
    rng = np.random.default_rng(2)
    L = 11
    kc = rng.standard_normal((L, sh.n_kv_heads, sh.head_dim))
    tr = {}
    layer.rows_with_cache(layer.soft_prompt, kc, kc * 0.5, trace=tr)
    sums = tr["p"].sum(axis=-1)
    np.testing.assert_allclose(sums, 1.0, atol=1e-12)
    # scores far beyond exp's range: [1000, 999] -> [1, e^-1] / (1 + e^-1)
    e = math.exp(-1.0)
    np.testing.assert_allclose(so.softmax_rows(np.array([[1000.0, 999.0]])), [[1 / (1 + e), e / (1 + e)]],
                               rtol=1e-12)
    # row r sees exactly L + r + 1 keys
    for r in range(sh.k_rows):
        nz = np.count_nonzero(tr["p"][r], axis=-1)
        assert np.all(nz == L + r + 1), (r, nz)


def check_incremental_equals_full_recompute():
    """Cache path == full causal layer over [context ; soft rows] (Eq. 1-3)."""
    cases = [dict(L=0), dict(L=1), dict(L=7), dict(L=2, k=5), dict(L=9, hq=2, hkv=2),
             dict(L=6, hq=6, hkv=2, k=1), dict(L=5, dh=4)]
    for i, c in enumerate(cases):
        L = c.pop("L")
        sh, w = random_layer(10 + i, **c)
        layer = so.Layer(sh, w)
        rng = np.random.default_rng(100 + i)
        ctx = rng.standard_normal((L, sh.d_model))
        kc, vc = layer.build_cache(ctx)
        inc = layer.rows_with_cache(layer.soft_prompt, kc, vc)
        full = layer.full_causal(np.concatenate([ctx, layer.soft_prompt], axis=0))[L:]
        np.testing.assert_allclose(inc, full, rtol=1e-10, atol=1e-10)


def check_gqa_equals_mha_with_repeated_kv():
    sh, w = random_layer(3, hq=6, hkv=2)
    G = sh.group
    sh_mha = dataclasses.replace(sh, n_kv_heads=sh.n_q_heads)
    dh = sh.head_dim
    rep = lambda m: np.repeat(m.reshape(sh.n_kv_heads, dh, -1), G, axis=0).reshape(-1, m.shape[1])
    w_mha = dataclasses.replace(w, w_k=rep(w.w_k), w_v=rep(w.w_v))
    rng = np.random.default_rng(4)
    kc = rng.standard_normal((9, sh.n_kv_heads, dh))
    vc = rng.standard_normal((9, sh.n_kv_heads, dh))
    a = so.Layer(sh, w).rows_with_cache(so.to_f64(w.soft_prompt, wl.F32), kc, vc)
    b = so.Layer(sh_mha, w_mha).rows_with_cache(so.to_f64(w.soft_prompt, wl.F32),
                                                np.repeat(kc, G, axis=1), np.repeat(vc, G, axis=1))
    np.testing.assert_allclose(a, b, rtol=1e-12, atol=1e-12)


def check_attention_matches_torch_sdpa():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(6)
    R, Hq, Hkv, dh, L = 4, 6, 2, 16, 13
    q = rng.standard_normal((R, Hq, dh))
    keys = rng.standard_normal((L + R, Hkv, dh))
    vals = rng.standard_normal((L + R, Hkv, dh))
    visible = np.arange(L + R)[None, :] <= (L + np.arange(R))[:, None]
    o = so.attention(q, keys, vals, visible, Hq // Hkv)
    tq = torch.from_numpy(q).permute(1, 0, 2)[None]                       # [1, Hq, R, dh]
    tk = torch.from_numpy(keys).permute(1, 0, 2).repeat_interleave(Hq // Hkv, 0)[None]
    tv = torch.from_numpy(vals).permute(1, 0, 2).repeat_interleave(Hq // Hkv, 0)[None]
    ref = torch.nn.functional.scaled_dot_product_attention(tq, tk, tv,
                                                           attn_mask=torch.from_numpy(visible))
    np.testing.assert_allclose(o, ref[0].permute(1, 0, 2).numpy(), rtol=1e-12, atol=1e-12)


def check_uniform_keys_give_mean_of_values():
    rng = np.random.default_rng(7)
    R, Hq, Hkv, dh, L = 3, 4, 2, 8, 10
    q = rng.standard_normal((R, Hq, dh))
    keys = np.tile(rng.standard_normal((1, Hkv, dh)), (L + R, 1, 1))
    vals = rng.standard_normal((L + R, Hkv, dh))
    visible = np.arange(L + R)[None, :] <= (L + np.arange(R))[:, None]
    o = so.attention(q, keys, vals, visible, 2)
    for r in range(R):
        for h in range(Hq):
            np.testing.assert_allclose(o[r, h], vals[: L + r + 1, h // 2].mean(axis=0),
                                       rtol=1e-12, atol=1e-12)


def check_head_blocks_and_group_map():
    """Head layout of Eq. 1-3 with G = Hq / Hkv = 2, dh = 2, d = Hq * dh: rows
    h*dh..h*dh+dh-1 of W_q form query head h, which reads KV head h // G, and
    the attention output enters W_o head-major.  With W_k = W_v = 0 (new keys and
    values are zero), cache values constant per KV head (c_j) and W_q nonzero for
    head 0 only, every head but 0 scores all keys equal, so its output is
    L / (L + r + 1) * c_{h // G}; head 0's is a different multiple of c_0.  W_o = I
    and W_down = 0 put the outputs in h2 - x."""
    hq, hkv, dh, L = 4, 2, 2, 5
    d = hq * dh
    sh, w = random_layer(67, d=d, hq=hq, hkv=hkv, dh=dh, f=3, k=2)
    rng = np.random.default_rng(68)
    wq = np.zeros((hq * dh, d))
    wq[:dh] = rng.standard_normal((dh, d)) * 2.0
    w = dataclasses.replace(w, w_q=f32(wq), w_k=f32(np.zeros((hkv * dh, d))),
                            w_v=f32(np.zeros((hkv * dh, d))), w_o=f32(np.eye(d)),
                            w_down=f32(np.zeros((d, sh.d_ff))))
    layer = so.Layer(sh, w)
    c = np.array([[1.0, -2.0], [3.0, 0.5]])                  # value of KV head j
    kc = rng.standard_normal((L, hkv, dh)) * 2.0
    vc = np.repeat(c[None], L, axis=0)
    x = rng.standard_normal((sh.k_rows, d))
    o = (layer.rows_with_cache(x, kc, vc) - x).reshape(sh.k_rows, hq, dh)
    for r in range(sh.k_rows):
        for h in range(1, hq):
            np.testing.assert_allclose(o[r, h], L / (L + r + 1) * c[h // 2], rtol=1e-12, atol=1e-12)
        a = o[r, 0] / c[0]
        np.testing.assert_allclose(a[0], a[1], rtol=1e-12)
        assert 0.0 < a[0] < 1.0 and abs(a[0] - L / (L + r + 1)) > 1e-3


def check_hand_built_cache_matches_full_recompute():
    """A one-token cache built by hand in the [token][KV head][dh] layout: the
    context row has unit rms, the input gain is 1 and eps 0, so its normalised
    row is itself, and rotation at position 0 is the identity; its key and value
    are then W_k x and W_v x split head-major.  The cached pass of the soft rows
    must equal the full causal pass over [context; soft rows] (Eq. 1-3)."""
    sh, w = random_layer(69, d=16, hq=4, hkv=2, dh=4, k=3, eps=0.0)
    w = dataclasses.replace(w, g_in=f32(np.ones(16)))
    layer = so.Layer(sh, w)
    xc = np.random.default_rng(70).standard_normal(16)
    xc = xc / np.sqrt(np.mean(xc * xc))
    kc = (np.asarray(w.w_k, np.float64) @ xc).reshape(1, 2, 4)
    vc = (np.asarray(w.w_v, np.float64) @ xc).reshape(1, 2, 4)
    full = layer.full_causal(np.vstack([xc[None], layer.soft_prompt]))[1:]
    np.testing.assert_allclose(layer.rows_with_cache(layer.soft_prompt, kc, vc), full,
                               rtol=1e-10, atol=1e-12)


def check_rms_norm():
    rng = np.random.default_rng(8)
    x = rng.standard_normal((5, 32))
    y = so.rms_norm(x, np.ones(32), 0.0)
    np.testing.assert_allclose(np.sqrt(np.mean(y * y, axis=-1)), 1.0, rtol=1e-12)
    np.testing.assert_allclose(so.rms_norm(3.5 * x, np.ones(32), 0.0), y, rtol=1e-12)
    # eps enters inside the root: a constant row c gives c / sqrt(c^2 + eps)
    c = np.full((1, 4), 0.5)
    np.testing.assert_allclose(so.rms_norm(c, np.ones(4), 0.75), 0.5 / 1.0, rtol=1e-12)


def check_silu():
    np.testing.assert_allclose(so.silu(np.array([1.0])), [0.7310585786300049], rtol=1e-14)
    z = np.linspace(-6, 6, 25)
    np.testing.assert_allclose(so.silu(z) - so.silu(-z), z, atol=1e-12)
    assert so.silu(np.array([0.0]))[0] == 0.0


def check_swiglu_block_by_hand():
    """d=2, d_ff=1 layer with zero attention output: h2 = h1 + W_down a with
    a = silu(n_0) * n_1 computed by hand from n = h1 / rms(h1)."""
    sh, w = hand_layer()
    layer = so.Layer(sh, w)
    x = np.array([[3.0, -1.0]])
    h2 = layer.finish(x, np.zeros((1, 1, 2)))
    rms = np.sqrt((9 + 1) / 2)
    n0, n1 = 3 / rms, -1 / rms
    a = n0 / (1 + np.exp(-n0)) * n1
    np.testing.assert_allclose(h2, [[3.0 + a, -1.0]], rtol=1e-12)


def check_readout_pooling():
    sh, w = random_layer(9, pool=wl.POOL_MEAN)
    h2 = np.random.default_rng(1).standard_normal((sh.k_rows, sh.d_model))
    lm = so.Layer(sh, w).readout(h2)
    ll = so.Layer(dataclasses.replace(sh, pool=wl.POOL_LAST), w).readout(h2)
    hw = np.asarray(w.head_w, np.float64)
    np.testing.assert_allclose(lm, hw @ h2.mean(axis=0) + w.head_b, rtol=1e-12)
    np.testing.assert_allclose(ll, hw @ h2[-1] + w.head_b, rtol=1e-12)
    # zero head gives the bias
    w0 = dataclasses.replace(w, head_w=np.zeros_like(w.head_w))
    np.testing.assert_allclose(so.Layer(sh, w0).readout(h2), w.head_b, rtol=0, atol=0)


def check_k1_mean_equals_last():
    sh, w = random_layer(12, k=1)
    w = dataclasses.replace(w, soft_prompt=w.soft_prompt[:1])
    rng = np.random.default_rng(3)
    kc = rng.standard_normal((5, sh.n_kv_heads, sh.head_dim))
    a = so.Layer(sh, w)
    b = so.Layer(dataclasses.replace(sh, pool=wl.POOL_LAST), w)
    np.testing.assert_allclose(a.readout(a.rows_with_cache(a.soft_prompt, kc, kc)),
                               b.readout(b.rows_with_cache(b.soft_prompt, kc, kc)), rtol=1e-14)


def check_paged_gather_matches_contiguous():
    sh = wl.Shape(64, 4, 2, 16, 64, 2, 2, w_dtype=wl.BF16, kv_dtype=wl.BF16)
    w = wl.custom(sh, [0, 1, 15, 16, 17, 40, 65, 130], wl.LAYOUT_CONTIGUOUS, 21)
    for P in (16, 32, 64):  # every page size the classify path takes
        paged = wl.contiguous_to_paged(w.cache, P, 5 + P)
        for b in range(8):
            k1, v1 = so.sequence_kv(w.cache, b)
            k2, v2 = so.sequence_kv(paged, b)
            assert k1.shape == (int(w.cache.seq_lens[b]), 2, 16)
            assert np.array_equal(k1, k2) and np.array_equal(v1, v2)


def check_cache_untouched():
    sh = wl.Shape(64, 4, 2, 16, 64, 2, 2, w_dtype=wl.BF16, kv_dtype=wl.BF16)
    w = wl.custom(sh, [5, 33], wl.LAYOUT_PAGED, 22)
    before = hashlib.sha256(w.cache.k_pool.tobytes() + w.cache.v_pool.tobytes()).hexdigest()
    so.classify(so.Layer(sh, w.weights), w.cache, w.seq_ids)
    after = hashlib.sha256(w.cache.k_pool.tobytes() + w.cache.v_pool.tobytes()).hexdigest()
    assert before == after


def check_fusion_hand_example():
    g = read_golden("fusion_hand_d2.txt")
    sh = wl.Shape(2, 1, 1, 2, 1, 1, 2, rms_eps=0.0, w_dtype=wl.F32, kv_dtype=wl.F32)
    _, w = random_layer(30, d=2, hq=1, hkv=1, dh=2, f=1, k=1, C=2)
    w = dataclasses.replace(w, w_fc=f32(np.reshape(g["w_fc"], (2, 4))), g_h=f32(g["g_h"]),
                            g_e=f32(g["g_e"]))
    layer = so.Layer(sh, w)
    x = layer.fuse(np.array([g["h"]]), np.array([g["e"]]))
    np.testing.assert_allclose(x.ravel(), g["x"], atol=1e-9)


def check_fusion_eps_inside_the_root():
    # constant rows 0.5 with eps = 0.75 and unit gains normalise to
    # 0.5 / sqrt(0.25 + 0.75) = 0.5 each; W_fc = [I | I] adds the two halves
    sh = wl.Shape(2, 1, 1, 2, 1, 1, 2, rms_eps=0.75, w_dtype=wl.F32, kv_dtype=wl.F32)
    _, w = random_layer(31, d=2, hq=1, hkv=1, dh=2, f=1, k=1, C=2)
    w = dataclasses.replace(w, w_fc=f32(np.concatenate([np.eye(2), np.eye(2)], axis=1)),
                            g_h=f32([1.0, 1.0]), g_e=f32([1.0, 1.0]))
    x = so.Layer(sh, w).fuse(np.full((1, 2), 0.5), np.full((1, 2), 0.5))
    np.testing.assert_allclose(x, [[1.0, 1.0]], rtol=1e-12)


def fused_layer(seed, w_fc_kind, unit_rows=False):
    sh, w = random_layer(seed, k=3)
    d = sh.d_model
    rng = np.random.default_rng(seed + 100)
    if w_fc_kind == "embed_only":      # [0 | I]
        fc = np.concatenate([np.zeros((d, d)), np.eye(d)], axis=1)
    elif w_fc_kind == "hidden_only":   # [I | 0]
        fc = np.concatenate([np.eye(d), np.zeros((d, d))], axis=1)
    else:
        fc = 0.3 * rng.standard_normal((d, 2 * d))
    w.w_fc = f32(fc)
    w.g_h = f32(1 + 0.1 * rng.standard_normal(d))
    w.g_e = f32(np.ones(d)) if w_fc_kind == "embed_only" else f32(1 + 0.1 * rng.standard_normal(d))
    if unit_rows:
        e = rng.standard_normal(w.soft_prompt.shape)
        w.soft_prompt = f32(e / np.sqrt(np.mean(e * e, axis=1, keepdims=True)))
    return sh, w


def check_fusion_with_embedding_only_is_the_row_path():
    # W_fc = [0 | I], unit gain, eps 0, unit-RMS soft prompt: the fused rows are
    # the soft-prompt rows themselves, whatever the hidden state
    sh, w = fused_layer(31, "embed_only", unit_rows=True)
    sh = dataclasses.replace(sh, rms_eps=0.0)
    layer = so.Layer(sh, w)
    cw = wl.custom(sh, [6, 11], wl.LAYOUT_CONTIGUOUS, 32)
    hidden = f32(np.random.default_rng(33).standard_normal((2, sh.d_model)) * 3)
    fused = so.classify(layer, cw.cache, cw.seq_ids, hidden=hidden)
    plain = so.classify(layer, cw.cache, cw.seq_ids)
    np.testing.assert_allclose(fused, plain, rtol=1e-5, atol=1e-6)


def check_fusion_with_hidden_only_ignores_the_prompt():
    # W_fc = [I | 0]: the soft prompt no longer reaches the layer
    sh, w = fused_layer(34, "hidden_only")
    cw = wl.custom(sh, [4, 9], wl.LAYOUT_PAGED, 35)
    hidden = f32(np.random.default_rng(36).standard_normal((2, sh.d_model)))
    a = so.classify(so.Layer(sh, w), cw.cache, cw.seq_ids, hidden=hidden)
    w2 = dataclasses.replace(w, soft_prompt=f32(w.soft_prompt[::-1] * 2 + 1))
    b = so.classify(so.Layer(sh, w2), cw.cache, cw.seq_ids, hidden=hidden)
    np.testing.assert_allclose(a, b, rtol=0, atol=1e-12)
    # and it does depend on the hidden state
    c = so.classify(so.Layer(sh, w), cw.cache, cw.seq_ids, hidden=f32(hidden * -1 + 0.5))
    assert np.max(np.abs(a - c)) > 1e-6


def check_tasks_with_hidden_fuse_their_own_prompt():
    """Several tasks over MTP inputs: task t fuses the hidden state with its own
    prompt (task 0 equals the single-task fused path with its prompt and head;
    changing task 1's prompt changes task 1 only)."""
    sh, w = fused_layer(37, "mixed")
    layer = so.Layer(sh, w)
    cw = wl.custom(sh, [5, 12], wl.LAYOUT_PAGED, 38)
    hidden = f32(np.random.default_rng(39).standard_normal((2, sh.d_model)))
    prompts, heads, biases = _tasks(40, 2, sh)
    a = so.classify_tasks(layer, cw.cache, cw.seq_ids, prompts, heads, biases, hidden=hidden)
    t0 = so.Layer(sh, dataclasses.replace(w, soft_prompt=prompts[0], head_w=heads[0], head_b=biases[0]))
    np.testing.assert_array_equal(a[:, 0], so.classify(t0, cw.cache, cw.seq_ids, hidden=hidden))
    p2 = prompts.copy()
    p2[1] = p2[1][::-1] * 2
    b = so.classify_tasks(layer, cw.cache, cw.seq_ids, p2, heads, biases, hidden=hidden)
    np.testing.assert_array_equal(a[:, 0], b[:, 0])
    assert np.max(np.abs(a[:, 1] - b[:, 1])) > 1e-6


def check_recursive_k1_equals_parallel_fused():
    sh, w = fused_layer(40, "random")
    sh = dataclasses.replace(sh, k_rows=1)
    w = dataclasses.replace(w, soft_prompt=w.soft_prompt[:1])
    layer = so.Layer(sh, w)
    cw = wl.custom(sh, [0, 7, 12], wl.LAYOUT_CONTIGUOUS, 41)
    hidden = f32(np.random.default_rng(42).standard_normal((3, sh.d_model)))
    a = so.classify_recursive(layer, cw.cache, cw.seq_ids, hidden)
    b = so.classify(layer, cw.cache, cw.seq_ids, hidden=hidden)
    np.testing.assert_allclose(a, b, rtol=1e-12, atol=1e-12)


def check_recursive_equals_stepwise_reconstruction():
    # rebuild SP-k from pinned pieces, differently: at step i fuse the previous
    # output with prompt row i, then run the parallel causal path over ALL rows
    # so far and take its last output
    for pool in (wl.POOL_MEAN, wl.POOL_LAST):
        sh, w = fused_layer(43, "random")
        sh = dataclasses.replace(sh, pool=pool)
        layer = so.Layer(sh, w)
        cw = wl.custom(sh, [0, 6, 11], wl.LAYOUT_PAGED, 44)
        hidden = f32(np.random.default_rng(45).standard_normal((3, sh.d_model)))
        got = so.classify_recursive(layer, cw.cache, cw.seq_ids, hidden)
        for b in range(3):
            kc, vc = so.sequence_kv(cw.cache, b)
            prev = hidden[b].astype(np.float64)[None, :]
            rows, outs = [], []
            for i in range(sh.k_rows):
                rows.append(layer.fuse(prev, layer.soft_prompt[i:i + 1])[0])
                h2 = layer.rows_with_cache(np.array(rows), kc, vc)
                outs.append(h2[-1])
                prev = h2[-1:]
            np.testing.assert_allclose(got[b], layer.readout(np.array(outs)), rtol=1e-9, atol=1e-12)


def check_recursive_embedding_only_is_the_row_path():
    # W_fc = [0 | I] with unit gain, eps 0, unit-RMS rows: every step's input is
    # its prompt row, so the recursion is the causal pass over the prompt rows
    sh, w = fused_layer(46, "embed_only", unit_rows=True)
    sh = dataclasses.replace(sh, rms_eps=0.0)
    layer = so.Layer(sh, w)
    cw = wl.custom(sh, [3, 10], wl.LAYOUT_CONTIGUOUS, 47)
    hidden = f32(np.random.default_rng(48).standard_normal((2, sh.d_model)))
    a = so.classify_recursive(layer, cw.cache, cw.seq_ids, hidden)
    b = so.classify(layer, cw.cache, cw.seq_ids)
    np.testing.assert_allclose(a, b, rtol=1e-5, atol=1e-6)


def _tasks(seed, T, sh):
    rng = np.random.default_rng(seed)
    prompts = f32(rng.standard_normal((T, sh.k_rows, sh.d_model)) * 0.4)
    heads = f32(rng.standard_normal((T, sh.n_classes, sh.d_model)))
    biases = f32(rng.standard_normal((T, sh.n_classes)))
    return prompts, heads, biases


def check_one_task_is_the_single_task_path():
    sh, w = random_layer(50)
    layer = so.Layer(sh, w)
    cw = wl.custom(sh, [0, 9, 20], wl.LAYOUT_PAGED, 51)
    got = so.classify_tasks(layer, cw.cache, cw.seq_ids, f32(w.soft_prompt[None]), f32(w.head_w[None]),
                            f32(w.head_b[None]))
    np.testing.assert_array_equal(got[:, 0], so.classify(layer, cw.cache, cw.seq_ids))


def check_tasks_are_isolated_and_permutable():
    sh, w = random_layer(52)
    layer = so.Layer(sh, w)
    cw = wl.custom(sh, [4, 13], wl.LAYOUT_CONTIGUOUS, 53)
    prompts, heads, biases = _tasks(54, 3, sh)
    a = so.classify_tasks(layer, cw.cache, cw.seq_ids, prompts, heads, biases)
    # another task's prompt and head change nothing for task 0
    p2, h2, b2 = prompts.copy(), heads.copy(), biases.copy()
    p2[1] = p2[1][::-1] * 3
    h2[2] = -h2[2]
    b = so.classify_tasks(layer, cw.cache, cw.seq_ids, p2, h2, b2)
    np.testing.assert_array_equal(a[:, 0], b[:, 0])
    assert np.max(np.abs(a[:, 1] - b[:, 1])) > 1e-6
    # permuting the tasks permutes the logits
    perm = [2, 0, 1]
    c = so.classify_tasks(layer, cw.cache, cw.seq_ids, prompts[perm], heads[perm], biases[perm])
    np.testing.assert_array_equal(c, a[:, perm])


def check_task_rows_belong_to_their_task():
    """Per-sequence rows [B, T, k, d]: task t reads its own rows rows[:, t] and
    nothing else (task 0 is the single-task path on rows[:, 0]; changing task
    1's rows changes task 1 only)."""
    sh, w = random_layer(56)
    layer = so.Layer(sh, w)
    cw = wl.custom(sh, [3, 10], wl.LAYOUT_PAGED, 57)
    prompts, heads, biases = _tasks(58, 2, sh)
    rng = np.random.default_rng(59)
    rows = f32(rng.standard_normal((2, 2, sh.k_rows, sh.d_model)) * 0.4)
    a = so.classify_tasks(layer, cw.cache, cw.seq_ids, prompts, heads, biases, rows=rows)
    t0 = so.Layer(sh, dataclasses.replace(w, head_w=heads[0], head_b=biases[0]))
    np.testing.assert_array_equal(a[:, 0], so.classify(t0, cw.cache, cw.seq_ids, rows=rows[:, 0]))
    rows2 = rows.copy()
    rows2[:, 1] = rows2[:, 1, ::-1] * 2
    b = so.classify_tasks(layer, cw.cache, cw.seq_ids, prompts, heads, biases, rows=rows2)
    np.testing.assert_array_equal(a[:, 0], b[:, 0])
    assert np.max(np.abs(a[:, 1] - b[:, 1])) > 1e-6


def check_norm_gains_fold_into_the_next_projection():
    """An RMSNorm gain scales channels of the normalised rows that feed only the
    next projection: g_in * s with the columns of W_q, W_k, W_v divided by s,
    or g_post * s with the columns of W_gate, W_up divided by s, leaves every
    logit unchanged for any positive s; either gain scaled alone changes them."""
    sh, w = random_layer(60)
    cw = wl.custom(sh, [6, 17], wl.LAYOUT_CONTIGUOUS, 61)
    s = f32(np.random.default_rng(62).uniform(0.5, 2.0, sh.d_model))
    run = lambda ww: so.classify(so.Layer(sh, ww), cw.cache, cw.seq_ids)
    base = run(w)
    folded_in = dataclasses.replace(w, g_in=w.g_in * s, w_q=w.w_q / s, w_k=w.w_k / s, w_v=w.w_v / s)
    folded_post = dataclasses.replace(w, g_post=w.g_post * s, w_gate=w.w_gate / s, w_up=w.w_up / s)
    # the folded weights are rounded to fp32 like the originals: compare loosely
    np.testing.assert_allclose(run(folded_in), base, rtol=1e-5, atol=1e-6)
    np.testing.assert_allclose(run(folded_post), base, rtol=1e-5, atol=1e-6)
    for alone in (dataclasses.replace(w, g_in=w.g_in * s), dataclasses.replace(w, g_post=w.g_post * s)):
        assert np.max(np.abs(run(alone) - base)) > 1e-3


def check_classify_follows_the_sequence_ids():
    """Logits of a batch of ids are the per-sequence logits in the ids' order
    (sequences of different lengths, so any mix-up shows)."""
    sh, w = random_layer(64)
    layer = so.Layer(sh, w)
    cw = wl.custom(sh, [2, 9, 14], wl.LAYOUT_PAGED, 65)
    ref = so.classify(layer, cw.cache, np.arange(3))
    for ids in ([2, 0, 1], [1, 1]):
        ids = np.array(ids, dtype=np.int32)
        np.testing.assert_array_equal(so.classify(layer, cw.cache, ids), ref[ids])
    assert np.max(np.abs(ref[0] - ref[2])) > 1e-6


def check_lm_head_readout_eps_inside_the_root():
    # a constant pooled vector c with gain 1 and head I normalises to
    # c / sqrt(c^2 + eps): 0.5 / sqrt(0.25 + 0.75) = 0.5
    sh = wl.Shape(2, 1, 1, 2, 1, 2, 2, rms_eps=0.75, w_dtype=wl.F32, kv_dtype=wl.F32)
    _, w = random_layer(66, d=2, hq=1, hkv=1, dh=2, f=1, k=2, C=2)
    w = dataclasses.replace(w, head_w=np.eye(2), head_b=None, g_final=f32([1.0, 1.0]))
    z = so.Layer(sh, w).readout(np.full((2, 2), 0.5))
    np.testing.assert_allclose(z, [0.5, 0.5], rtol=1e-12)


def check_lm_head_readout_hand_example():
    g = read_golden("lm_head_readout_d2.txt")
    sh = wl.Shape(2, 1, 1, 2, 1, 2, 2, rms_eps=0.0, w_dtype=wl.F32, kv_dtype=wl.F32)
    _, w = random_layer(60, d=2, hq=1, hkv=1, dh=2, f=1, k=2, C=2)
    w = dataclasses.replace(w, head_w=np.eye(2), head_b=None, g_final=f32(g["g_final"]))
    layer = so.Layer(sh, w)
    z = layer.readout(np.reshape(g["h2"], (2, 2)))
    np.testing.assert_allclose(z, g["logits"], atol=1e-9)
    np.testing.assert_allclose(z[1] - z[0], g["yes_minus_no"][0], atol=1e-9)


def check_lm_head_readout_is_scale_invariant():
    # the final norm makes the logits blind to a positive scale of the outputs
    sh, w = random_layer(61, eps=0.0)
    w = dataclasses.replace(w, g_final=f32(1 + 0.1 * np.random.default_rng(62).standard_normal(16)))
    layer = so.Layer(sh, w)
    h2 = np.random.default_rng(63).standard_normal((sh.k_rows, sh.d_model))
    np.testing.assert_allclose(layer.readout(h2 * 7.5), layer.readout(h2), rtol=1e-12, atol=1e-12)
    plain = so.Layer(sh, dataclasses.replace(w, g_final=None))
    assert np.max(np.abs(plain.readout(h2 * 7.5) - plain.readout(h2))) > 1e-3


def check_bf16_decode_fixed_patterns():
    # bf16 is the upper half of an IEEE binary32: these bit patterns have fixed values
    bits = np.array([0x3F80, 0xC020, 0x0001, 0x7F80, 0x8000, 0x4049, 0x0080], dtype=np.uint16)
    v = so.to_f64(bits, so.BF16)
    assert v.dtype == np.float64
    assert v[0] == 1.0 and v[1] == -2.5
    assert v[2] == 2.0 ** -133                     # smallest bf16 subnormal
    assert np.isposinf(v[3])
    assert v[4] == 0.0 and np.signbit(v[4])        # negative zero keeps its sign
    assert v[5] == 3.140625                        # 0x4049: 1.5703125 * 2
    assert v[6] == 2.0 ** -126                     # smallest normal


def _attention_step_case(seed, lens, kr=3):
    sh = wl.Shape(16, 4, 2, 8, 24, kr, 3, rope_theta=100.0, w_dtype=wl.F32, kv_dtype=wl.F32)
    w = wl.custom(sh, lens, wl.LAYOUT_PAGED, seed)
    _, lw = random_layer(seed + 1, k=kr)
    layer = so.Layer(sh, lw)
    rng = np.random.default_rng(seed + 2)
    x = rng.standard_normal((len(lens), kr, 16)) * 0.5
    return sh, w, layer, x


def check_attention_step_matches_the_layer_trace():
    # the step-level checker must agree with the attention inside the layer
    # pass, whose mask and positions the full causal recompute pins
    sh, w, layer, x = _attention_step_case(70, [0, 1, 5, 16, 23])
    q, kn, vn, want = [], [], [], []
    for i, sid in enumerate(w.seq_ids):
        kc, vc = so.sequence_kv(w.cache, int(sid))
        tr = {}
        layer.rows_with_cache(x[i], kc, vc, trace=tr)
        q.append(tr["q"]); kn.append(tr["k_new"]); vn.append(tr["v_new"]); want.append(tr["o"])
    got = so.attention_step(sh, w.cache, w.seq_ids, np.array(q), np.array(kn), np.array(vn))
    np.testing.assert_allclose(got, np.array(want), rtol=1e-12, atol=1e-12)
    # batch slot i reads the cache of seq_ids[i]: a permuted batch permutes the outputs
    perm = np.array([3, 0, 4, 1, 2])
    got_p = so.attention_step(sh, w.cache, w.seq_ids[perm], np.array(q)[perm], np.array(kn)[perm],
                              np.array(vn)[perm])
    np.testing.assert_allclose(got_p, np.array(want)[perm], rtol=1e-12, atol=1e-12)


def check_attention_step_uniform_keys_closed_form():
    # equal keys everywhere: row r averages the values of the L + r + 1 tokens it sees
    sh, w, _, _ = _attention_step_case(71, [0, 3, 17])
    rng = np.random.default_rng(72)
    B, kr, hq, hkv, dh = 3, sh.k_rows, sh.n_q_heads, sh.n_kv_heads, sh.head_dim
    key = rng.standard_normal((hkv, dh)).astype(np.float32).astype(np.float64)  # exact in the cache
    cache = dataclasses.replace(w.cache, k_pool=np.broadcast_to(
        key[None, :, None, :].astype(np.float32), w.cache.k_pool.shape).copy())
    q = rng.standard_normal((B, kr, hq, dh))
    kn = np.broadcast_to(key, (B, kr, hkv, dh)).copy()
    vn = rng.standard_normal((B, kr, hkv, dh))
    o = so.attention_step(sh, cache, w.seq_ids, q, kn, vn)
    for i, sid in enumerate(w.seq_ids):
        _, vc = so.sequence_kv(cache, int(sid))
        vals = np.concatenate([vc, vn[i]], axis=0)
        L = vc.shape[0]
        for r in range(kr):
            for h in range(hq):
                np.testing.assert_allclose(o[i, r, h], vals[:L + r + 1, h // sh.group].mean(axis=0),
                                           rtol=1e-12, atol=1e-12)


ALL_CHECKS = [check_bf16_decode_fixed_patterns, check_attention_step_matches_the_layer_trace,
              check_attention_step_uniform_keys_closed_form,
              check_lm_head_readout_hand_example, check_lm_head_readout_is_scale_invariant,
              check_one_task_is_the_single_task_path, check_tasks_are_isolated_and_permutable,
              check_task_rows_belong_to_their_task, check_norm_gains_fold_into_the_next_projection,
              check_rope_frequencies_follow_theta, check_classify_follows_the_sequence_ids,
              check_lm_head_readout_eps_inside_the_root, check_fusion_eps_inside_the_root,
              check_head_blocks_and_group_map, check_hand_built_cache_matches_full_recompute,
              check_tasks_with_hidden_fuse_their_own_prompt,
              check_recursive_k1_equals_parallel_fused,
              check_recursive_equals_stepwise_reconstruction,
              check_recursive_embedding_only_is_the_row_path,
              check_fusion_hand_example, check_fusion_with_embedding_only_is_the_row_path,
              check_fusion_with_hidden_only_ignores_the_prompt,
              check_hand_example, check_rope_pairs, check_rope_relative_and_norm,
              check_softmax_rows_sum_to_one, check_incremental_equals_full_recompute,
              check_gqa_equals_mha_with_repeated_kv, check_attention_matches_torch_sdpa,
              check_uniform_keys_give_mean_of_values, check_rms_norm, check_silu,
              check_swiglu_block_by_hand, check_readout_pooling, check_k1_mean_equals_last,
              check_paged_gather_matches_contiguous, check_cache_untouched]


@pytest.mark.parametrize("check", ALL_CHECKS, ids=lambda f: f.__name__)
def test_pin(check):
    check()


# --------------------------------------------------------------------------- #
# planted mistakes: every one must trip at least one pin
# --------------------------------------------------------------------------- #
# Each factory takes the original function and returns a wrong variant of it.
def _rope_flipped(orig):
    return lambda x, positions, theta: orig(x, -np.asarray(positions), theta)


def _rope_interleaved(orig):
    def f(x, positions, theta):
        dh = x.shape[-1]
        perm = np.concatenate([np.arange(0, dh, 2), np.arange(1, dh, 2)])
        return orig(x[..., perm], positions, theta)[..., np.argsort(perm)]
    return f


def _scale_1_over_dh(orig):
    return lambda q, keys, visible, group: orig(q / np.sqrt(q.shape[-1]), keys, visible, group)


def _no_causal_mask(orig):
    return lambda q, keys, values, visible, group: orig(q, keys, values, np.ones_like(visible),
                                                         group)


def _gqa_modulo(orig):
    def f(q, keys, visible, group):
        # query head h reads KV head h % Hkv instead of h // group
        Hq, Hkv = q.shape[1], keys.shape[1]
        expanded = keys[:, [h % Hkv for h in range(Hq)]]
        return orig(q, expanded, visible, 1)
    return f


def _rms_sum(orig):
    return lambda x, gain, eps: x / np.sqrt(np.sum(x * x, axis=-1, keepdims=True) + eps) * gain


def _rms_eps_outside(orig):
    return lambda x, gain, eps: x / (np.sqrt(np.mean(x * x, axis=-1, keepdims=True)) + eps) * gain


def _silu_sigmoid(orig):
    return lambda z: 1.0 / (1.0 + np.exp(-z))


def _positions_from_zero(orig):
    def f(self, x, k_cache, v_cache, trace=None):
        saved = self.project_qkv
        L = k_cache.shape[0]
        self.project_qkv = lambda xx, pos: saved(xx, np.asarray(pos) - L)
        try:
            return orig(self, x, k_cache, v_cache, trace)
        finally:
            del self.project_qkv
    return f


def _residual_dropped(orig):
    def f(self, x, o):
        return orig(self, np.zeros_like(x), o) + 0.0 * x
    return f


def _gate_up_swapped(orig):
    def f(self, x, o):
        self.w_gate, self.w_up = self.w_up, self.w_gate
        try:
            return orig(self, x, o)
        finally:
            self.w_gate, self.w_up = self.w_up, self.w_gate
    return f


def _readout_first_row(orig):
    return lambda self, h2: self.head_w @ h2[0] + self.head_b


def _gather_reversed(orig):
    def f(cache, seq_id):
        k, v = orig(cache, seq_id)
        if cache.layout == so.LAYOUT_PAGED:
            k, v = k[::-1].copy(), v[::-1].copy()
        return k, v
    return f


def _fusion_order_swapped(orig):
    def f(self, hidden, embed):
        eps = self.shape.rms_eps
        z = np.concatenate([so.rms_norm(embed, self.g_e, eps), so.rms_norm(hidden, self.g_h, eps)],
                           axis=-1)
        return z @ self.w_fc.T
    return f


def _fusion_gains_swapped(orig):
    def f(self, hidden, embed):
        self.g_h, self.g_e = self.g_e, self.g_h
        try:
            return orig(self, hidden, embed)
        finally:
            self.g_h, self.g_e = self.g_e, self.g_h
    return f


def _fusion_hidden_unnormalised(orig):
    def f(self, hidden, embed):
        eps = self.shape.rms_eps
        z = np.concatenate([hidden * self.g_h, so.rms_norm(embed, self.g_e, eps)], axis=-1)
        return z @ self.w_fc.T
    return f


def _recursive_variant(feed_input=False, fixed_position=False, no_append=False, row_zero=False):
    """classify_recursive with one planted mistake (same loop otherwise)."""
    def f(layer, cache, seq_ids, hidden, traces=None):
        sh = layer.shape
        k = layer.soft_prompt.shape[0]
        out = []
        for i, sid in enumerate(np.asarray(seq_ids)):
            kc, vc = so.sequence_kv(cache, int(sid))
            L = kc.shape[0]
            prev = so.to_f64(hidden[i], sh.w_dtype)[None, :]
            keys, values, outs = kc, vc, []
            for step in range(k):
                e = layer.soft_prompt[0:1] if row_zero else layer.soft_prompt[step:step + 1]
                x = layer.fuse(prev, e)
                q, kn, vn = layer.project_qkv(x, np.array([L if fixed_position else L + step]))
                ks = np.concatenate([kc if no_append else keys, kn], axis=0)
                vs = np.concatenate([vc if no_append else values, vn], axis=0)
                keys, values = ks, vs
                o = so.attention(q, ks, vs, np.ones((1, ks.shape[0]), dtype=bool), sh.group)
                a = layer.finish(x, o)
                outs.append(a[0])
                prev = x if feed_input else a
            out.append(layer.readout(np.array(outs)))
        return np.array(out)
    return f


def _readout_norm_before_pool(orig):
    def f(self, h2):
        if self.g_final is None:
            return orig(self, h2)
        n = so.rms_norm(h2, self.g_final, self.shape.rms_eps)
        pooled = n.mean(axis=0) if self.shape.pool == so.POOL_MEAN else n[-1]
        return self.head_w @ pooled + self.head_b
    return f


def _readout_final_norm_ignored(orig):
    def f(self, h2):
        pooled = h2.mean(axis=0) if self.shape.pool == so.POOL_MEAN else h2[-1]
        return self.head_w @ pooled + self.head_b
    return f


def _bf16_low_half(orig):
    def f(arr, dtype_code):
        a = np.asarray(arr)
        if dtype_code == so.BF16:
            return a.astype(np.uint32).view(np.float32).astype(np.float64)
        return orig(arr, dtype_code)
    return f


def _post_norm_takes_input_gain(orig):
    def f(self, x, o):
        saved, self.g_post = self.g_post, self.g_in
        try:
            return orig(self, x, o)
        finally:
            self.g_post = saved
    return f


def _input_norm_takes_post_gain(orig):
    def f(self, x, positions):
        saved, self.g_in = self.g_in, self.g_post
        try:
            return orig(self, x, positions)
        finally:
            self.g_in = saved
    return f


def _task_rows_of_first_task(orig):
    def f(layer, cache, seq_ids, prompts, heads, biases=None, rows=None, hidden=None):
        r = None if rows is None else np.repeat(rows[:, :1], rows.shape[1], axis=1)
        return orig(layer, cache, seq_ids, prompts, heads, biases, r, hidden)
    return f


def _rope_theta_fixed(orig):
    return lambda x, positions, theta: orig(x, positions, 1.0e4)


def _softmax_without_shift(orig):
    def f(s):
        e = np.exp(s)
        return e / e.sum(axis=-1, keepdims=True)
    return f


def _sequence_ids_ignored(orig):
    def f(layer, cache, seq_ids, rows=None, traces=None, hidden=None):
        return orig(layer, cache, np.arange(len(seq_ids)), rows, traces, hidden)
    return f


def _readout_eps_dropped(orig):
    def f(self, h2):
        saved = self.shape
        self.shape = dataclasses.replace(saved, rms_eps=0.0)
        try:
            return orig(self, h2)
        finally:
            self.shape = saved
    return f


def _o_flattened_dim_major(orig):
    def f(self, x, o):
        return orig(self, x, np.ascontiguousarray(o.transpose(0, 2, 1)).reshape(o.shape))
    return f


def _query_heads_reversed(orig):
    def f(self, x, positions):
        q, k, v = orig(self, x, positions)
        return q[:, ::-1].copy(), k, v
    return f


def _kv_heads_reversed(orig):
    def f(self, x, positions):
        q, k, v = orig(self, x, positions)
        return q, k[:, ::-1].copy(), v[:, ::-1].copy()
    return f


def _fusion_eps_dropped(orig):
    def f(self, hidden, embed):
        saved = self.shape
        self.shape = dataclasses.replace(saved, rms_eps=0.0)
        try:
            return orig(self, hidden, embed)
        finally:
            self.shape = saved
    return f


def _page_size_fixed_at_16(orig):
    def f(cache, seq_id):
        if cache.layout != so.LAYOUT_PAGED or cache.page_size == 16:
            return orig(cache, seq_id)
        # the pool's slots read as if pages held 16 tokens
        L = int(cache.seq_lens[seq_id])
        n_pg = (L + 15) // 16
        pages = cache.page_table[seq_id, :n_pg]
        hkv, dh = cache.k_pool.shape[1], cache.k_pool.shape[3]
        kp = cache.k_pool[pages][:, :, :16].transpose(0, 2, 1, 3).reshape(n_pg * 16, hkv, dh)[:L]
        vp = cache.v_pool[pages][:, :, :16].transpose(0, 2, 1, 3).reshape(n_pg * 16, hkv, dh)[:L]
        return so.to_f64(kp, cache.dtype), so.to_f64(vp, cache.dtype)
    return f


def _tasks_fuse_the_layer_prompt(orig):
    def f(layer, cache, seq_ids, prompts, heads, biases=None, rows=None, hidden=None):
        if hidden is not None:  # every task fuses with the handle's own prompt
            prompts = np.repeat(layer.soft_prompt[None].astype(np.float32), len(prompts), axis=0)
        return orig(layer, cache, seq_ids, prompts, heads, biases, rows, hidden)
    return f


def _attention_step_ids_ignored(orig):
    def f(shape, cache, seq_ids, q, k_new, v_new):
        return orig(shape, cache, np.arange(len(seq_ids)), q, k_new, v_new)
    return f


def _attention_step_mask_off_by_one(orig):
    def f(shape, cache, seq_ids, q, k_new, v_new):
        kr = q.shape[1]
        out = np.zeros_like(q, dtype=np.float64)
        for i, sid in enumerate(np.asarray(seq_ids)):
            kc, vc = so.sequence_kv(cache, int(sid))
            L = kc.shape[0]
            keys = np.concatenate([kc, k_new[i]], axis=0)
            values = np.concatenate([vc, v_new[i]], axis=0)
            # row r also sees new token r + 1 (one position into its future)
            visible = np.arange(L + kr)[None, :] <= (L + np.arange(kr))[:, None] + 1
            out[i] = so.attention(q[i], keys, values, visible, shape.group)
        return out
    return f


MUTANTS = {
    "bf16_decoded_from_low_half": (so, "to_f64", _bf16_low_half),
    "attention_step_mask_off_by_one": (so, "attention_step", _attention_step_mask_off_by_one),
    "lm_readout_norm_before_pool": (so.Layer, "readout", _readout_norm_before_pool),
    "lm_readout_final_norm_ignored": (so.Layer, "readout", _readout_final_norm_ignored),
    "recursion_feeds_layer_input": (so, "classify_recursive",
                                    lambda orig: _recursive_variant(feed_input=True)),
    "recursion_fixed_position": (so, "classify_recursive",
                                 lambda orig: _recursive_variant(fixed_position=True)),
    "recursion_forgets_new_keys": (so, "classify_recursive",
                                   lambda orig: _recursive_variant(no_append=True)),
    "recursion_reuses_first_prompt_row": (so, "classify_recursive",
                                          lambda orig: _recursive_variant(row_zero=True)),
    "fusion_order_swapped": (so.Layer, "fuse", _fusion_order_swapped),
    "fusion_gains_swapped": (so.Layer, "fuse", _fusion_gains_swapped),
    "fusion_hidden_unnormalised": (so.Layer, "fuse", _fusion_hidden_unnormalised),
    "rope_direction_flipped": (so, "rope", _rope_flipped),
    "rope_interleaved_pairs": (so, "rope", _rope_interleaved),
    "softmax_scale_1_over_dh": (so, "attention_probs", _scale_1_over_dh),
    "no_causal_mask": (so, "attention", _no_causal_mask),
    "gqa_head_modulo": (so, "attention_probs", _gqa_modulo),
    "rms_sum_not_mean": (so, "rms_norm", _rms_sum),
    "rms_eps_outside_root": (so, "rms_norm", _rms_eps_outside),
    "silu_is_sigmoid": (so, "silu", _silu_sigmoid),
    "positions_from_zero": (so.Layer, "rows_with_cache", _positions_from_zero),
    "residual_dropped": (so.Layer, "finish", _residual_dropped),
    "gate_up_swapped": (so.Layer, "finish", _gate_up_swapped),
    "readout_first_row": (so.Layer, "readout", _readout_first_row),
    "paged_gather_reversed": (so, "sequence_kv", _gather_reversed),
    "post_norm_takes_input_gain": (so.Layer, "finish", _post_norm_takes_input_gain),
    "input_norm_takes_post_gain": (so.Layer, "project_qkv", _input_norm_takes_post_gain),
    "task_rows_of_first_task": (so, "classify_tasks", _task_rows_of_first_task),
    "rope_theta_fixed_at_1e4": (so, "rope", _rope_theta_fixed),
    "softmax_without_max_shift": (so, "softmax_rows", _softmax_without_shift),
    "sequence_ids_ignored": (so, "classify", _sequence_ids_ignored),
    "lm_readout_eps_dropped": (so.Layer, "readout", _readout_eps_dropped),
    "o_flattened_dim_major": (so.Layer, "finish", _o_flattened_dim_major),
    "query_heads_reversed": (so.Layer, "project_qkv", _query_heads_reversed),
    "kv_heads_reversed": (so.Layer, "project_qkv", _kv_heads_reversed),
    "fusion_eps_dropped": (so.Layer, "fuse", _fusion_eps_dropped),
    "page_size_fixed_at_16": (so, "sequence_kv", _page_size_fixed_at_16),
    "tasks_fuse_the_layer_prompt": (so, "classify_tasks", _tasks_fuse_the_layer_prompt),
    "attention_step_ids_ignored": (so, "attention_step", _attention_step_ids_ignored),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_planted_mistakes_are_caught(name, monkeypatch):
    owner, attr, factory = MUTANTS[name]
    monkeypatch.setattr(owner, attr, factory(getattr(owner, attr)))
    failed = []
    for check in ALL_CHECKS:
        try:
            check()
        except AssertionError:
            failed.append(check.__name__)
    assert failed, f"planted mistake {name!r} passed every pin"
