"""Seeded synthetic workloads for the Speculative Probing classify path.

This module only draws random numbers and lays them out in memory.  It holds
none of the method's arithmetic (no normalisation, rotation, attention or
projection), so both the CUDA path and the fp64 oracle may consume what it
produces without sharing any of the computation under test.

Recipe (the paper's datasets and trained weights are not available; these
shapes stand in for its four models and its sequence-length mix, Sec. 5.1 and
Sec. 6):

* numpy ``SeedSequence(seed)`` is split into four independent streams:
  structure (lengths, page permutation), weights (layer matrices, norm gains,
  soft prompt, head), cache (K then V), rows (per-sequence input rows).
* matrices, soft prompt and head: N(0, 0.02); RMSNorm gains: 1 + N(0, 0.02)
  (a unit gain with a N(0, 0.02) offset; literal N(0, 0.02) gains would shrink
  every activation towards zero and leave nothing to compare).
* cached K/V: N(0, 1), interpreted as already rotated at their own positions.
* bf16 tensors are drawn in fp32 and rounded once, round-to-nearest-even, here;
  every consumer sees the same bytes.
* ragged lengths: integers uniform in the stated inclusive range.
* paged caches: 16-token pages, physical pages = sum ceil(L_b/16), assigned by a
  seeded random permutation; page layout is [page][kv_head][slot][head_dim].
* contiguous caches: one buffer, sequence b at a token offset, token-major
  [token][kv_head][head_dim].
* input fusion (optional): a fifth stream draws W_fc [d][2d] N(0, 0.02), the
  two fusion norm gains 1 + N(0, 0.02) and base hidden states [B][d] N(0, 1).
* several tasks (optional): a sixth stream draws the soft prompts, heads (and
  rows) of tasks 1..T-1; task 0 keeps the single-task draws.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional

import numpy as np

F32, BF16 = 0, 1
LAYOUT_CONTIGUOUS, LAYOUT_PAGED = 0, 1
POOL_MEAN, POOL_LAST = 0, 1


# --------------------------------------------------------------------------- #
# storage formats
# --------------------------------------------------------------------------- #
def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round fp32 values to bf16 (round-to-nearest-even) and return the bits."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    rounded = (u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)
    return rounded.astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """Widen bf16 bits to fp32 (exact)."""
    return (np.ascontiguousarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


# --------------------------------------------------------------------------- #
# shapes
# --------------------------------------------------------------------------- #
@dataclasses.dataclass
class Shape:
    """Dimensions of one frozen decoder layer plus its probe."""
    d_model: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    d_ff: int
    k_rows: int
    n_classes: int
    rope_theta: float = 1.0e4
    rms_eps: float = 1.0e-6
    w_dtype: int = BF16
    kv_dtype: int = BF16
    pool: int = POOL_MEAN
    page_size: int = 16
    n_tasks: int = 1         # probes (soft prompt + head) sharing one pass over the cache

    @property
    def group(self) -> int:
        return self.n_q_heads // self.n_kv_heads


@dataclasses.dataclass
class WorkloadSpec:
    name: str
    shape: Shape
    batch: int
    len_lo: int
    len_hi: int
    layout: int
    seed: int
    rows_per_seq: bool = False   # draw per-sequence input rows [B][k][d]
    fused: bool = False          # draw fusion weights and per-sequence hidden states [B][d]
    head_bias: bool = False
    ragged_frac: Optional[float] = None  # sweep: L uniform in [(1-f)L, (1+f)L]


def _shape_4b(k, C):
    return Shape(2560, 32, 8, 128, 9728, k, C)


def _shape_8b(k, C):
    return Shape(4096, 32, 8, 128, 12288, k, C)


def _shape_27b(k, C):
    return Shape(5120, 40, 8, 128, 17408, k, C)


def named(name: str, **overrides) -> WorkloadSpec:
    """The named workloads: 'tiny', '4b', '8b_paged', '27b_long' and sweep
    points 'sweep_B{B}_L{L}_k{k}_C{C}' (d=4096 shape, +-25% ragged, paged)."""
    if name == "tiny":
        spec = WorkloadSpec("tiny", Shape(128, 4, 2, 32, 256, 4, 2, w_dtype=F32, kv_dtype=F32),
                            1, 64, 64, LAYOUT_CONTIGUOUS, 0)
    elif name == "4b":
        spec = WorkloadSpec("4b", _shape_4b(8, 2), 16, 256, 2048, LAYOUT_CONTIGUOUS, 1)
    elif name == "8b_paged":
        spec = WorkloadSpec("8b_paged", _shape_8b(16, 4), 64, 1024, 8192, LAYOUT_PAGED, 2)
    elif name == "27b_long":
        spec = WorkloadSpec("27b_long", _shape_27b(16, 2), 8, 32768, 32768, LAYOUT_PAGED, 3)
    elif name.startswith("sweep_"):
        parts = dict((p[0], int(p[1:])) for p in name[len("sweep_"):].split("_"))
        L = parts["L"]
        spec = WorkloadSpec(name, _shape_8b(parts["k"], parts["C"]), parts["B"],
                            int(math.floor(0.75 * L)), int(math.ceil(1.25 * L)), LAYOUT_PAGED, 4,
                            ragged_frac=0.25)
    else:
        raise KeyError(f"unknown workload {name!r}")
    shape_over = {k: v for k, v in overrides.items() if hasattr(spec.shape, k)}
    spec_over = {k: v for k, v in overrides.items() if not hasattr(spec.shape, k)}
    if shape_over:
        spec.shape = dataclasses.replace(spec.shape, **shape_over)
    if spec_over:
        spec = dataclasses.replace(spec, **spec_over)
    return spec


SWEEP_POINTS = [f"sweep_B{B}_L{L}_k{k}_C{C}"
                for B in (1, 8, 32, 128, 256)
                for L in (512, 2048, 8192, 16384)
                for k in (1, 4, 16, 32)
                for C in (2, 16)]


# --------------------------------------------------------------------------- #
# generated data
# --------------------------------------------------------------------------- #
@dataclasses.dataclass
class Weights:
    """Layer, prompt and head tensors.  bf16 tensors are uint16 bit arrays,
    fp32 tensors are float32 arrays.  Matrices are row-major [out][in]."""
    w_q: np.ndarray
    w_k: np.ndarray
    w_v: np.ndarray
    w_o: np.ndarray
    w_gate: np.ndarray
    w_up: np.ndarray
    w_down: np.ndarray
    g_in: np.ndarray       # float32 [d]
    g_post: np.ndarray     # float32 [d]
    soft_prompt: np.ndarray  # w_dtype [k][d]
    head_w: np.ndarray     # float32 [C][d]
    head_b: Optional[np.ndarray]  # float32 [C] or None
    # input fusion in front of the layer (MTP): w_dtype [d][2d] and its two
    # RMSNorm gains, float32 [d]; None when rows are given directly
    w_fc: Optional[np.ndarray] = None
    g_h: Optional[np.ndarray] = None
    g_e: Optional[np.ndarray] = None
    # LM-head readout: final RMSNorm gain float32 [d] applied before the head
    g_final: Optional[np.ndarray] = None


@dataclasses.dataclass
class KVCache:
    """Either layout; arrays hold bf16 bits (uint16) or float32."""
    layout: int
    dtype: int
    seq_lens: np.ndarray           # int32 [n_seqs]
    # contiguous
    k_flat: Optional[np.ndarray] = None   # [sum L][Hkv][dh]
    v_flat: Optional[np.ndarray] = None
    offsets: Optional[np.ndarray] = None  # int64 [n_seqs] token offsets
    # paged
    k_pool: Optional[np.ndarray] = None   # [n_pages][Hkv][P][dh]
    v_pool: Optional[np.ndarray] = None
    page_table: Optional[np.ndarray] = None  # int32 [n_seqs][max_pages]
    page_size: int = 16

    @property
    def n_seqs(self) -> int:
        return int(self.seq_lens.shape[0])

    @property
    def n_pages(self) -> int:
        return 0 if self.k_pool is None else int(self.k_pool.shape[0])

    @property
    def max_pages(self) -> int:
        return 0 if self.page_table is None else int(self.page_table.shape[1])


@dataclasses.dataclass
class Workload:
    spec: WorkloadSpec
    weights: Weights
    cache: KVCache
    seq_ids: np.ndarray             # int32 [B] (which cache sequences are classified)
    rows: Optional[np.ndarray]      # w_dtype [B][k][d] or None (shared soft prompt)
    hidden: Optional[np.ndarray] = None  # w_dtype [B][d]: base hidden states (fused input)

    @property
    def shape(self) -> Shape:
        return self.spec.shape


def _normal(rng, shape, std, dtype_code):
    x = rng.standard_normal(size=shape, dtype=np.float32)
    if std != 1.0:
        x *= np.float32(std)
    return f32_to_bf16_bits(x) if dtype_code == BF16 else x


def draw_lengths(spec: WorkloadSpec, rng) -> np.ndarray:
    if spec.len_lo == spec.len_hi:
        return np.full(spec.batch, spec.len_lo, dtype=np.int32)
    return rng.integers(spec.len_lo, spec.len_hi, size=spec.batch, endpoint=True).astype(np.int32)


def draw_weights(shape: Shape, rng, head_bias: bool) -> Weights:
    d, hq, hkv, dh, f, k, C = (shape.d_model, shape.n_q_heads, shape.n_kv_heads,
                               shape.head_dim, shape.d_ff, shape.k_rows, shape.n_classes)
    wd = shape.w_dtype
    w_q = _normal(rng, (hq * dh, d), 0.02, wd)
    w_k = _normal(rng, (hkv * dh, d), 0.02, wd)
    w_v = _normal(rng, (hkv * dh, d), 0.02, wd)
    w_o = _normal(rng, (d, hq * dh), 0.02, wd)
    w_gate = _normal(rng, (f, d), 0.02, wd)
    w_up = _normal(rng, (f, d), 0.02, wd)
    w_down = _normal(rng, (d, f), 0.02, wd)
    g_in = (1.0 + 0.02 * rng.standard_normal(d)).astype(np.float32)
    g_post = (1.0 + 0.02 * rng.standard_normal(d)).astype(np.float32)
    soft_prompt = _normal(rng, (k, d), 0.02, wd)
    head_w = (0.02 * rng.standard_normal((C, d))).astype(np.float32)
    head_b = (0.02 * rng.standard_normal(C)).astype(np.float32) if head_bias else None
    return Weights(w_q, w_k, w_v, w_o, w_gate, w_up, w_down, g_in, g_post,
                   soft_prompt, head_w, head_b)


def draw_fusion(shape: Shape, seed: int, batch: int):
    """Input-fusion weights and base hidden states from a fifth stream of the
    seed (the first four are untouched): W_fc [d][2d] N(0, 0.02), gains
    1 + N(0, 0.02), hidden states [B][d] N(0, 1)."""
    rng = np.random.default_rng(np.random.SeedSequence(seed).spawn(5)[4])
    d, wd = shape.d_model, shape.w_dtype
    w_fc = _normal(rng, (d, 2 * d), 0.02, wd)
    g_h = (1.0 + 0.02 * rng.standard_normal(d)).astype(np.float32)
    g_e = (1.0 + 0.02 * rng.standard_normal(d)).astype(np.float32)
    hidden = _normal(rng, (batch, d), 1.0, wd)
    return w_fc, g_h, g_e, hidden


def with_tasks(w: "Workload", T: int) -> "Workload":
    """The workload with T tasks: task 0 keeps the drawn soft prompt, head (and
    rows); tasks 1..T-1 draw theirs from a sixth stream of the seed.  Stacked as
    soft_prompt [T k][d], head_w [T C][d], head_b [T C], rows [B][T k][d]."""
    sh = w.spec.shape
    if T <= 1:
        return w
    rng = np.random.default_rng(np.random.SeedSequence(w.spec.seed).spawn(6)[5])
    k, d, C, wd = sh.k_rows, sh.d_model, sh.n_classes, sh.w_dtype
    prompts = [w.weights.soft_prompt] + [_normal(rng, (k, d), 0.02, wd) for _ in range(T - 1)]
    heads = [w.weights.head_w] + [(0.02 * rng.standard_normal((C, d))).astype(np.float32)
                                  for _ in range(T - 1)]
    biases = None
    if w.weights.head_b is not None:
        biases = [w.weights.head_b] + [(0.02 * rng.standard_normal(C)).astype(np.float32)
                                       for _ in range(T - 1)]
    weights = dataclasses.replace(w.weights, soft_prompt=np.concatenate(prompts, axis=0),
                                  head_w=np.concatenate(heads, axis=0),
                                  head_b=None if biases is None else np.concatenate(biases))
    rows = w.rows
    if rows is not None:
        B = rows.shape[0]
        extra = [_normal(rng, (B, k, d), 0.02, wd) for _ in range(T - 1)]
        rows = np.concatenate([rows] + extra, axis=1)
    spec = dataclasses.replace(w.spec, shape=dataclasses.replace(sh, n_tasks=T))
    return dataclasses.replace(w, spec=spec, weights=weights, rows=rows)


def task_views(w: "Workload"):
    """(prompts [T][k][d], heads [T][C][d], biases [T][C] or None, rows
    [B][T][k][d] or None) of a stacked T-task workload."""
    sh = w.spec.shape
    T, k, d, C = sh.n_tasks, sh.k_rows, sh.d_model, sh.n_classes
    wt = w.weights
    rows = None if w.rows is None else w.rows.reshape(w.rows.shape[0], T, k, d)
    return (wt.soft_prompt.reshape(T, k, d), wt.head_w.reshape(T, C, d),
            None if wt.head_b is None else wt.head_b.reshape(T, C), rows)


def with_lm_head(w: "Workload") -> "Workload":
    """The workload read out through a frozen LM head: a final-norm gain
    1 + N(0, 0.02) and head rows standing in for the label tokens' lm_head rows
    (N(0, 0.02) per task, no bias), from a seventh stream of the seed."""
    sh = w.spec.shape
    rng = np.random.default_rng(np.random.SeedSequence(w.spec.seed).spawn(7)[6])
    g_final = (1.0 + 0.02 * rng.standard_normal(sh.d_model)).astype(np.float32)
    head = (0.02 * rng.standard_normal(w.weights.head_w.shape)).astype(np.float32)
    weights = dataclasses.replace(w.weights, g_final=g_final, head_w=head, head_b=None)
    return dataclasses.replace(w, weights=weights)


def with_fusion(w: "Workload") -> "Workload":
    """The same workload with fusion weights and hidden states attached."""
    w_fc, g_h, g_e, hidden = draw_fusion(w.spec.shape, w.spec.seed, len(w.seq_ids))
    weights = dataclasses.replace(w.weights, w_fc=w_fc, g_h=g_h, g_e=g_e)
    return dataclasses.replace(w, weights=weights, hidden=hidden)


def draw_cache(shape: Shape, lens: np.ndarray, layout: int, rng_struct, rng_kv) -> KVCache:
    hkv, dh, P = shape.n_kv_heads, shape.head_dim, shape.page_size
    dt = shape.kv_dtype
    store = np.uint16 if dt == BF16 else np.float32
    total = int(lens.sum())
    # K for every sequence first, then V, token-major per sequence
    k_flat = np.empty((total, hkv, dh), dtype=store)
    v_flat = np.empty((total, hkv, dh), dtype=store)
    offsets = np.zeros(len(lens), dtype=np.int64)
    if len(lens) > 1:
        offsets[1:] = np.cumsum(lens[:-1])
    chunk = 1 << 15
    for buf in (k_flat, v_flat):
        for t0 in range(0, total, chunk):
            t1 = min(total, t0 + chunk)
            buf[t0:t1] = _normal(rng_kv, (t1 - t0, hkv, dh), 1.0, dt)
    if layout == LAYOUT_CONTIGUOUS:
        return KVCache(LAYOUT_CONTIGUOUS, dt, lens.astype(np.int32), k_flat=k_flat, v_flat=v_flat,
                       offsets=offsets, page_size=P)
    n_pages_seq = [(int(L) + P - 1) // P for L in lens]
    n_pages = int(sum(n_pages_seq))
    max_pages = max(1, max(n_pages_seq) if n_pages_seq else 1)
    perm = rng_struct.permutation(n_pages).astype(np.int32)
    page_table = np.full((len(lens), max_pages), -1, dtype=np.int32)
    k_pool = np.zeros((max(n_pages, 1), hkv, P, dh), dtype=store)
    v_pool = np.zeros((max(n_pages, 1), hkv, P, dh), dtype=store)
    base = 0
    for b, L in enumerate(lens):
        L = int(L)
        npg = n_pages_seq[b]
        page_table[b, :npg] = perm[base:base + npg]
        o = int(offsets[b])
        for j in range(npg):
            t0, t1 = j * P, min(L, (j + 1) * P)
            phys = page_table[b, j]
            # [tokens][hkv][dh] -> [hkv][slot][dh]
            k_pool[phys, :, : t1 - t0, :] = k_flat[o + t0:o + t1].transpose(1, 0, 2)
            v_pool[phys, :, : t1 - t0, :] = v_flat[o + t0:o + t1].transpose(1, 0, 2)
        base += npg
    return KVCache(LAYOUT_PAGED, dt, lens.astype(np.int32), k_pool=k_pool, v_pool=v_pool,
                   page_table=page_table, page_size=P)


def generate(spec: WorkloadSpec) -> Workload:
    """Draw every input of one workload from its seed (see module docstring)."""
    ss = np.random.SeedSequence(spec.seed)
    s_struct, s_w, s_kv, s_rows = ss.spawn(4)
    rng_struct = np.random.default_rng(s_struct)
    lens = draw_lengths(spec, rng_struct)
    weights = draw_weights(spec.shape, np.random.default_rng(s_w), spec.head_bias)
    cache = draw_cache(spec.shape, lens, spec.layout, rng_struct, np.random.default_rng(s_kv))
    rows = None
    if spec.rows_per_seq:
        sh = spec.shape
        rows = _normal(np.random.default_rng(s_rows), (spec.batch, sh.k_rows, sh.d_model), 0.02,
                       sh.w_dtype)
    seq_ids = np.arange(spec.batch, dtype=np.int32)
    w = Workload(spec, weights, cache, seq_ids, rows)
    if spec.shape.n_tasks > 1:
        w = with_tasks(dataclasses.replace(w, spec=dataclasses.replace(
            spec, shape=dataclasses.replace(spec.shape, n_tasks=1))), spec.shape.n_tasks)
    return with_fusion(w) if spec.fused else w


@dataclasses.dataclass
class DeviceWorkload:
    """A paged workload whose K/V pools live only on the device (see
    generate_on_device).  Host side: lengths, page table, weights, rows."""
    spec: WorkloadSpec
    weights: Weights
    seq_lens: np.ndarray      # int32 [B]
    page_table: np.ndarray    # int32 [B][max_pages]
    n_pages: int
    k_pool: object            # torch int16 (bf16 bits) [n_pages][Hkv][P][dh] on the device
    v_pool: object
    seq_ids: np.ndarray
    rows: Optional[np.ndarray]

    @property
    def shape(self) -> Shape:
        return self.spec.shape

    def host_cache(self, ids) -> KVCache:
        """The sequences `ids` copied back into a host paged cache (renumbered
        0..len(ids)-1, pages compacted) for a CPU consumer."""
        import torch
        ids = [int(i) for i in ids]
        P = self.shape.page_size
        lens = self.seq_lens[ids].astype(np.int32)
        n_seq_pages = [(int(L) + P - 1) // P for L in lens]
        max_pages = max(1, max(n_seq_pages) if n_seq_pages else 1)
        phys = [self.page_table[i, :n] for i, n in zip(ids, n_seq_pages)]
        flat = np.concatenate(phys) if phys else np.zeros(0, np.int32)
        sel = torch.as_tensor(flat.astype(np.int64), device=self.k_pool.device)
        k = self.k_pool.index_select(0, sel).cpu().numpy().view(np.uint16) if len(flat) else None
        v = self.v_pool.index_select(0, sel).cpu().numpy().view(np.uint16) if len(flat) else None
        hkv, dh = self.shape.n_kv_heads, self.shape.head_dim
        if k is None:
            k = np.zeros((1, hkv, P, dh), np.uint16)
            v = np.zeros_like(k)
        table = np.full((len(ids), max_pages), -1, dtype=np.int32)
        base = 0
        for j, n in enumerate(n_seq_pages):
            table[j, :n] = np.arange(base, base + n, dtype=np.int32)
            base += n
        return KVCache(LAYOUT_PAGED, BF16, lens, k_pool=k, v_pool=v, page_table=table, page_size=P)


def generate_on_device(spec: WorkloadSpec, device="cuda", weights: Optional[Weights] = None
                       ) -> DeviceWorkload:
    """A paged bf16 workload too large to draw on the host: lengths, page
    permutation, weights and rows come from the same numpy streams as
    generate(spec); the K/V values are N(0, 1) drawn on the device by a torch
    generator seeded from the cache stream (so they differ from generate()'s
    values but follow the same distribution)."""
    import torch
    assert spec.layout == LAYOUT_PAGED and spec.shape.kv_dtype == BF16
    ss = np.random.SeedSequence(spec.seed)
    s_struct, s_w, s_kv, s_rows = ss.spawn(4)
    rng_struct = np.random.default_rng(s_struct)
    lens = draw_lengths(spec, rng_struct)
    if weights is None:
        weights = draw_weights(spec.shape, np.random.default_rng(s_w), spec.head_bias)
    sh = spec.shape
    P = sh.page_size
    n_seq_pages = [(int(L) + P - 1) // P for L in lens]
    n_pages = int(sum(n_seq_pages))
    max_pages = max(1, max(n_seq_pages) if n_seq_pages else 1)
    perm = rng_struct.permutation(n_pages).astype(np.int32)
    table = np.full((len(lens), max_pages), -1, dtype=np.int32)
    base = 0
    for b, n in enumerate(n_seq_pages):
        table[b, :n] = perm[base:base + n]
        base += n
    gen = torch.Generator(device=device)
    gen.manual_seed(int(np.random.default_rng(s_kv).integers(0, 2**62)))
    shape4 = (max(n_pages, 1), sh.n_kv_heads, P, sh.head_dim)
    k_pool = torch.randn(shape4, generator=gen, device=device, dtype=torch.float32).to(torch.bfloat16)
    v_pool = torch.randn(shape4, generator=gen, device=device, dtype=torch.float32).to(torch.bfloat16)
    rows = None
    if spec.rows_per_seq:
        rows = _normal(np.random.default_rng(s_rows), (spec.batch, sh.k_rows, sh.d_model), 0.02,
                       sh.w_dtype)
    return DeviceWorkload(spec, weights, lens.astype(np.int32), table, n_pages,
                          k_pool.view(torch.int16), v_pool.view(torch.int16),
                          np.arange(spec.batch, dtype=np.int32), rows)


def contiguous_to_paged(cache: KVCache, page_size: int, seed: int) -> KVCache:
    """Re-lay a contiguous cache into shuffled pages holding the same values."""
    assert cache.layout == LAYOUT_CONTIGUOUS
    lens = cache.seq_lens
    P = page_size
    n_pages_seq = [(int(L) + P - 1) // P for L in lens]
    n_pages = int(sum(n_pages_seq))
    max_pages = max(1, max(n_pages_seq) if n_pages_seq else 1)
    perm = np.random.default_rng(seed).permutation(n_pages).astype(np.int32)
    hkv, dh = cache.k_flat.shape[1], cache.k_flat.shape[2]
    page_table = np.full((len(lens), max_pages), -1, dtype=np.int32)
    k_pool = np.zeros((max(n_pages, 1), hkv, P, dh), dtype=cache.k_flat.dtype)
    v_pool = np.zeros_like(k_pool)
    base = 0
    for b, L in enumerate(lens):
        L = int(L)
        npg = n_pages_seq[b]
        page_table[b, :npg] = perm[base:base + npg]
        o = int(cache.offsets[b])
        for j in range(npg):
            t0, t1 = j * P, min(L, (j + 1) * P)
            phys = page_table[b, j]
            k_pool[phys, :, : t1 - t0, :] = cache.k_flat[o + t0:o + t1].transpose(1, 0, 2)
            v_pool[phys, :, : t1 - t0, :] = cache.v_flat[o + t0:o + t1].transpose(1, 0, 2)
        base += npg
    return KVCache(LAYOUT_PAGED, cache.dtype, lens.copy(), k_pool=k_pool, v_pool=v_pool,
                   page_table=page_table, page_size=P)


def custom(shape: Shape, lens, layout: int, seed: int, rows_per_seq=False, head_bias=False,
           name="custom") -> Workload:
    """A workload with explicit per-sequence lengths (edge cases in tests)."""
    lens = np.asarray(lens, dtype=np.int32)
    spec = WorkloadSpec(name, shape, len(lens), int(lens.min(initial=0)), int(lens.max(initial=0)),
                        layout, seed, rows_per_seq=rows_per_seq, head_bias=head_bias)
    ss = np.random.SeedSequence(seed)
    s_struct, s_w, s_kv, s_rows = ss.spawn(4)
    rng_struct = np.random.default_rng(s_struct)
    weights = draw_weights(shape, np.random.default_rng(s_w), head_bias)
    cache = draw_cache(shape, lens, layout, rng_struct, np.random.default_rng(s_kv))
    rows = None
    if rows_per_seq:
        rows = _normal(np.random.default_rng(s_rows), (len(lens), shape.k_rows, shape.d_model),
                       0.02, shape.w_dtype)
    return Workload(spec, weights, cache, np.arange(len(lens), dtype=np.int32), rows)
