"""fp64 CPU oracle for the Speculative Probing classify path.

TEST INFRASTRUCTURE.  Only the tests, ``__graft_entry__.smoke()`` and the CPU
baseline leg of ``bench.py`` may import or run this module.  It shares no code
with the CUDA path: it decodes the stored bytes itself and evaluates every step
from its plain definition in float64, step by step, in the order the paper
gives.  Nothing here is blocked, fused or reordered.

What is computed (Sec. 3.1, Sec. 3.2, Sec. 3.3 Eq. 1-3):

* k soft-prompt rows are appended after a sequence whose n = L cached keys and
  values already sit in the draft head's cache (Sec. 3.3).
* each row passes once through the frozen single decoder layer of the draft head
  (Sec. 3.1): pre-norm RMSNorm, Q/K/V projections, rotary embedding at the
  row's position, grouped-query attention over [cached ; new] keys (Eq. 1-3),
  output projection and residual, post-norm RMSNorm, SwiGLU feed-forward and
  residual.
* the new keys/values live only in local arrays here (the scratch buffer of
  Sec. 3.3); the cache passed in is never modified.
* a linear head reads class logits from the pooled outputs (Sec. 3.2,
  "Classification head"; pooled state per Fig. 2 and App. B).

Readings where the paper is silent (each is listed in the design notes):

1. rows are evaluated in the parallel form: all k rows at positions L..L+k-1 in
   one layer pass, row r attending causally to the cache and to new rows 0..r.
2. pooling: MEAN over the k outputs by default, LAST (row k-1) optional.
3. RMSNorm: y = x / sqrt(mean(x^2) + eps) * gain, mean over the hidden dim.
4. rotary embedding: NeoX rotate-half pairing (i, i + dh/2), frequency
   theta^(-2i/dh), applied to queries and keys, never to values; cached keys
   are stored already rotated at their own positions.
5. softmax scale 1/sqrt(dh) (Eq. 1); query head h reads KV head floor(h / G).
6. SwiGLU: a = silu(W_gate n) * (W_up n), silu(z) = z / (1 + exp(-z)).
7. head: logits = W_head pooled + bias (bias zero when absent); raw logits, no
   sigmoid.
8. no final norm before the head; no projection biases.
9. input fusion (Sec. 3.1, MTP architecture): the layer input is
   x = W_fc [RMSNorm(h; g_h) ; RMSNorm(e; g_e)] with W_fc stored [d][2d], the
   normalised hidden state first and the normalised embedding second (the
   order the paper lists them in); for probing, e is soft-prompt row r and h the
   base model's last hidden state of the sequence (Sec. 3.2, single-step
   probing), the same h for all k rows in the parallel form.
10. recursive probing SP-k (Sec. 3.2, "Recursive probing"): step 1 fuses the
   base hidden state h with soft-prompt row 1; step i > 1 fuses the layer output
   of step i-1 with row i.  Step i is one layer pass of one row at position
   L + i - 1 whose attention sees the cache and the new keys/values of steps
   1..i (the KV caching of Fig. 2).  The head reads the pooled step outputs
   (reading 2: MEAN by default, LAST = the k-th step's output).
11. several tasks over one cache (Sec. 3.3: classifiers with different soft
   prompts and heads share the same draft-head KV cache): task t has its own k
   soft-prompt rows and head; its rows sit at positions L..L+k-1 and attend to
   the cache and to the task's own new rows only, so each task's logits are
   those of a single-task classify with that task's prompt and head.
12. LM-head readout (Sec. 5 ablation "Classification head": the frozen lm_head's
   yes/no token logits): the head rows are the label tokens' rows of the
   frozen LM head and the pooled state first passes the head's final RMSNorm
   (gain g_final, the layer's eps): logits = W_head RMSNorm(pool(h2); g_final)
   (+ bias).  The yes/no difference is logits[yes] - logits[no].
13. head layout (grouped-query attention with no storage order in the paper):
   rows h*dh..h*dh+dh-1 of W_q are query head h, rows j*dh.. of W_k and W_v
   are KV head j, cached tokens hold [KV head][dh] in that order, and the
   attention output reaches W_o concatenated head-major.
"""
from __future__ import annotations

import numpy as np

F32, BF16 = 0, 1
LAYOUT_CONTIGUOUS, LAYOUT_PAGED = 0, 1
POOL_MEAN, POOL_LAST = 0, 1


# --------------------------------------------------------------------------- #
# storage decode (the oracle's own; bf16 is the upper half of an IEEE fp32)
# --------------------------------------------------------------------------- #
def to_f64(arr, dtype_code: int) -> np.ndarray:
    """Decode stored values (bf16 bits as uint16, or float32) to float64."""
    a = np.asarray(arr)
    if dtype_code == BF16:
        assert a.dtype == np.uint16, a.dtype
        widened = a.astype(np.uint32) << np.uint32(16)
        return widened.view(np.float32).astype(np.float64)
    assert a.dtype == np.float32, a.dtype
    return a.astype(np.float64)


# --------------------------------------------------------------------------- #
# the layer's pieces, each from its definition
# --------------------------------------------------------------------------- #
def rms_norm(x: np.ndarray, gain: np.ndarray, eps: float) -> np.ndarray:
    """RMSNorm over the last axis (reading 3)."""
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return x / np.sqrt(ms + eps) * gain


def rope(x: np.ndarray, positions: np.ndarray, theta: float) -> np.ndarray:
    """Rotary embedding, rotate-half pairing (reading 4).

    x: [..., T, H, dh]; positions: [T] (absolute, 0-based).  For pair i < dh/2
    with angle phi = p * theta^(-2i/dh): (a, b) -> (a cos phi - b sin phi,
    b cos phi + a sin phi), where a = x[i] and b = x[i + dh/2].
    """
    dh = x.shape[-1]
    half = dh // 2
    i = np.arange(half, dtype=np.float64)
    freq = theta ** (-2.0 * i / dh)                           # [half]
    phi = np.asarray(positions, dtype=np.float64)[:, None] * freq[None, :]   # [T, half]
    cos = np.cos(phi)[:, None, :]                            # [T, 1, half]
    sin = np.sin(phi)[:, None, :]
    a = x[..., :half]
    b = x[..., half:]
    return np.concatenate([a * cos - b * sin, b * cos + a * sin], axis=-1)


def silu(z: np.ndarray) -> np.ndarray:
    return z / (1.0 + np.exp(-z))


def softmax_rows(s: np.ndarray) -> np.ndarray:
    """Softmax along the last axis; masked entries carry -inf."""
    m = np.max(s, axis=-1, keepdims=True)
    e = np.exp(s - m)
    return e / np.sum(e, axis=-1, keepdims=True)


def attention_probs(q: np.ndarray, keys: np.ndarray, visible: np.ndarray, group: int):
    """Eq. 1 softmax for every query row and head.

    q: [R, Hq, dh]; keys: [T, Hkv, dh]; visible: bool [R, T].
    Returns p: [R, Hq, T].
    """
    R, Hq, dh = q.shape
    T = keys.shape[0]
    p = np.zeros((R, Hq, T))
    for h in range(Hq):
        g = h // group                                          # reading 5
        s = (q[:, h, :] @ keys[:, g, :].T) / np.sqrt(dh)        # [R, T]
        s = np.where(visible, s, -np.inf)
        p[:, h, :] = softmax_rows(s)
    return p


def attention(q, keys, values, visible, group):
    """Eq. 1: O = softmax(Q K'^T / sqrt(dh)) V' per head.  Returns [R, Hq, dh]."""
    p = attention_probs(q, keys, visible, group)
    R, Hq, _ = q.shape
    o = np.zeros((R, Hq, values.shape[-1]))
    for h in range(Hq):
        o[:, h, :] = p[:, h, :] @ values[:, h // group, :]
    return o


# --------------------------------------------------------------------------- #
# model: weights decoded once to float64
# --------------------------------------------------------------------------- #
class Layer:
    """The frozen decoder layer and the probe (soft prompt + head) in fp64."""

    def __init__(self, shape, weights):
        self.shape = shape
        wd = shape.w_dtype
        self.w_q = to_f64(weights.w_q, wd)
        self.w_k = to_f64(weights.w_k, wd)
        self.w_v = to_f64(weights.w_v, wd)
        self.w_o = to_f64(weights.w_o, wd)
        self.w_gate = to_f64(weights.w_gate, wd)
        self.w_up = to_f64(weights.w_up, wd)
        self.w_down = to_f64(weights.w_down, wd)
        self.g_in = np.asarray(weights.g_in, dtype=np.float64)
        self.g_post = np.asarray(weights.g_post, dtype=np.float64)
        self.soft_prompt = to_f64(weights.soft_prompt, wd)
        self.head_w = np.asarray(weights.head_w, dtype=np.float64)
        self.head_b = (np.zeros(self.head_w.shape[0]) if weights.head_b is None
                       else np.asarray(weights.head_b, dtype=np.float64))
        gf = getattr(weights, "g_final", None)
        self.g_final = None if gf is None else np.asarray(gf, dtype=np.float64)
        fc = getattr(weights, "w_fc", None)
        self.w_fc = None if fc is None else to_f64(fc, wd)
        self.g_h = None if fc is None else np.asarray(weights.g_h, dtype=np.float64)
        self.g_e = None if fc is None else np.asarray(weights.g_e, dtype=np.float64)

    # -- input fusion (reading 9) ---------------------------------------------
    def fuse(self, hidden: np.ndarray, embed: np.ndarray) -> np.ndarray:
        """x = W_fc [RMSNorm(h; g_h) ; RMSNorm(e; g_e)] for matching rows of
        hidden [T, d] and embed [T, d].  Returns [T, d]."""
        eps = self.shape.rms_eps
        z = np.concatenate([rms_norm(hidden, self.g_h, eps), rms_norm(embed, self.g_e, eps)], axis=-1)
        return z @ self.w_fc.T

    # -- pieces of the layer -------------------------------------------------
    def project_qkv(self, x: np.ndarray, positions: np.ndarray):
        """Pre-norm, Q/K/V projection, rotation at `positions` (Sec. 3.3).

        x: [T, d] -> q [T, Hq, dh] (rotated), k [T, Hkv, dh] (rotated),
        v [T, Hkv, dh]."""
        sh = self.shape
        xn = rms_norm(x, self.g_in, sh.rms_eps)
        T = x.shape[0]
        q = (xn @ self.w_q.T).reshape(T, sh.n_q_heads, sh.head_dim)
        k = (xn @ self.w_k.T).reshape(T, sh.n_kv_heads, sh.head_dim)
        v = (xn @ self.w_v.T).reshape(T, sh.n_kv_heads, sh.head_dim)
        q = rope(q, positions, sh.rope_theta)
        k = rope(k, positions, sh.rope_theta)
        return q, k, v

    def finish(self, x: np.ndarray, o: np.ndarray) -> np.ndarray:
        """Output projection + residual, post-norm, SwiGLU + residual.

        x: [T, d] layer input rows; o: [T, Hq, dh] attention output."""
        sh = self.shape
        T = x.shape[0]
        h1 = x + o.reshape(T, sh.n_q_heads * sh.head_dim) @ self.w_o.T
        n = rms_norm(h1, self.g_post, sh.rms_eps)
        a = silu(n @ self.w_gate.T) * (n @ self.w_up.T)
        return h1 + a @ self.w_down.T

    def readout(self, h2: np.ndarray) -> np.ndarray:
        """Linear head on the pooled soft-prompt outputs (reading 2, 7), after
        the final norm when the head is an LM head's rows (reading 12)."""
        pooled = h2.mean(axis=0) if self.shape.pool == POOL_MEAN else h2[-1]
        if self.g_final is not None:
            pooled = rms_norm(pooled, self.g_final, self.shape.rms_eps)
        return self.head_w @ pooled + self.head_b

    # -- the classify path: k rows against a resident cache ------------------
    def rows_with_cache(self, x: np.ndarray, k_cache: np.ndarray, v_cache: np.ndarray,
                        trace: dict | None = None) -> np.ndarray:
        """One layer pass of k rows at positions L..L+k-1 over a cache of L
        tokens (Eq. 1-3).  x: [k, d]; k_cache, v_cache: [L, Hkv, dh] (float64).
        Returns h2: [k, d]."""
        sh = self.shape
        L = k_cache.shape[0]
        kr = x.shape[0]
        q, k_new, v_new = self.project_qkv(x, np.arange(L, L + kr))
        keys = np.concatenate([k_cache, k_new], axis=0)      # K' (Eq. 2)
        values = np.concatenate([v_cache, v_new], axis=0)    # V' (Eq. 3)
        t = np.arange(L + kr)[None, :]
        r = np.arange(kr)[:, None]
        visible = t <= (L + r)                                # reading 1
        o = attention(q, keys, values, visible, sh.group)
        h2 = self.finish(x, o)
        if trace is not None:
            trace.update(q=q, k_new=k_new, v_new=v_new, o=o, h2=h2,
                         p=attention_probs(q, keys, visible, sh.group))
        return h2

    # -- full causal recompute (used to pin the incremental path) ------------
    def full_causal(self, x_all: np.ndarray) -> np.ndarray:
        """The same layer run over all T rows at positions 0..T-1 with its own
        keys/values and a causal mask, no cache.  Returns h2: [T, d]."""
        T = x_all.shape[0]
        q, k, v = self.project_qkv(x_all, np.arange(T))
        visible = np.arange(T)[None, :] <= np.arange(T)[:, None]
        o = attention(q, k, v, visible, self.shape.group)
        return self.finish(x_all, o)

    def build_cache(self, x_ctx: np.ndarray):
        """Keys/values the layer itself would have cached for context rows
        x_ctx [L, d] at positions 0..L-1 (keys rotated, values not)."""
        _, k, v = self.project_qkv(x_ctx, np.arange(x_ctx.shape[0]))
        return k, v


# --------------------------------------------------------------------------- #
# cache access (the oracle's own gather from either layout)
# --------------------------------------------------------------------------- #
def sequence_kv(cache, seq_id: int):
    """Logical [L, Hkv, dh] float64 K and V of one cached sequence."""
    L = int(cache.seq_lens[seq_id])
    if cache.layout == LAYOUT_CONTIGUOUS:
        o = int(cache.offsets[seq_id])
        k = to_f64(cache.k_flat[o:o + L], cache.dtype)
        v = to_f64(cache.v_flat[o:o + L], cache.dtype)
        return k, v
    P = cache.page_size
    n_pg = (L + P - 1) // P
    pages = cache.page_table[seq_id, :n_pg]
    # pool [page][hkv][slot][dh] -> [page][slot][hkv][dh] -> [token][hkv][dh]
    hkv, dh = cache.k_pool.shape[1], cache.k_pool.shape[3]
    kp = cache.k_pool[pages].transpose(0, 2, 1, 3).reshape(n_pg * P, hkv, dh)[:L]
    vp = cache.v_pool[pages].transpose(0, 2, 1, 3).reshape(n_pg * P, hkv, dh)[:L]
    return to_f64(kp, cache.dtype), to_f64(vp, cache.dtype)


def classify(layer: Layer, cache, seq_ids, rows=None, traces: list | None = None,
             hidden=None) -> np.ndarray:
    """Logits [B, C] (float64) for the sequences `seq_ids` of `cache`.

    rows: None (every sequence uses the shared soft prompt) or stored
    per-sequence rows [B, k, d] in the layer's weight dtype.
    hidden: stored base hidden states [B, d] (weight dtype): the rows are then
    the fused inputs of the soft prompt (reading 9) and `rows` is ignored."""
    out = []
    k = layer.soft_prompt.shape[0]
    for i, sid in enumerate(np.asarray(seq_ids)):
        if hidden is not None:
            h = np.repeat(to_f64(hidden[i], layer.shape.w_dtype)[None, :], k, axis=0)
            x = layer.fuse(h, layer.soft_prompt)
        else:
            x = layer.soft_prompt if rows is None else to_f64(rows[i], layer.shape.w_dtype)
        kc, vc = sequence_kv(cache, int(sid))
        tr = {} if traces is not None else None
        h2 = layer.rows_with_cache(x, kc, vc, trace=tr)
        if traces is not None:
            traces.append(tr)
        out.append(layer.readout(h2))
    return np.array(out).reshape(len(out), layer.head_w.shape[0])


def classify_recursive(layer: Layer, cache, seq_ids, hidden, traces: list | None = None
                       ) -> np.ndarray:
    """Logits [B, C] of recursive probing (reading 10), one step at a time.

    hidden: stored base hidden states [B, d] (weight dtype)."""
    sh = layer.shape
    k = layer.soft_prompt.shape[0]
    out = []
    for i, sid in enumerate(np.asarray(seq_ids)):
        kc, vc = sequence_kv(cache, int(sid))
        L = kc.shape[0]
        prev = to_f64(hidden[i], sh.w_dtype)[None, :]          # [1, d]
        keys, values = kc, vc
        xs, outs = [], []
        for step in range(k):
            x = layer.fuse(prev, layer.soft_prompt[step:step + 1])        # [1, d]
            q, k_new, v_new = layer.project_qkv(x, np.array([L + step]))
            keys = np.concatenate([keys, k_new], axis=0)
            values = np.concatenate([values, v_new], axis=0)
            visible = np.ones((1, keys.shape[0]), dtype=bool)           # all earlier keys
            o = attention(q, keys, values, visible, sh.group)
            a = layer.finish(x, o)                                       # [1, d]
            xs.append(x[0])
            outs.append(a[0])
            prev = a
        h2 = np.array(outs)
        if traces is not None:
            traces.append({"x": np.array(xs), "h2": h2})
        out.append(layer.readout(h2))
    return np.array(out).reshape(len(out), layer.head_w.shape[0])


def classify_tasks(layer: Layer, cache, seq_ids, prompts, heads, biases=None, rows=None,
                   hidden=None) -> np.ndarray:
    """Logits [B, T, C] of T tasks (reading 11): one single-task classify per task.

    prompts: stored soft prompts [T, k, d] (weight dtype); heads [T, C, d]
    float; biases [T, C] or None; rows: per-sequence rows [B, T, k, d] or None;
    hidden: base hidden states [B, d] fused with each task's prompt (reading 9)."""
    T = len(prompts)
    out = []
    for t in range(T):
        task = Layer.__new__(Layer)
        task.__dict__.update(layer.__dict__)
        task.soft_prompt = to_f64(prompts[t], layer.shape.w_dtype)
        task.head_w = np.asarray(heads[t], dtype=np.float64)
        task.head_b = (np.zeros(task.head_w.shape[0]) if biases is None
                       else np.asarray(biases[t], dtype=np.float64))
        out.append(classify(task, cache, seq_ids, None if rows is None else rows[:, t],
                            hidden=hidden))
    return np.stack(out, axis=1)


def attention_step(shape, cache, seq_ids, q, k_new, v_new) -> np.ndarray:
    """The attention step alone (Eq. 1-3) for already rotated inputs.

    q: [B, k, Hq, dh]; k_new, v_new: [B, k, Hkv, dh] (float64).
    Returns o: [B, k, Hq, dh] float64."""
    B, kr = q.shape[0], q.shape[1]
    out = np.zeros_like(q, dtype=np.float64)
    for i, sid in enumerate(np.asarray(seq_ids)):
        kc, vc = sequence_kv(cache, int(sid))
        L = kc.shape[0]
        keys = np.concatenate([kc, k_new[i]], axis=0)
        values = np.concatenate([vc, v_new[i]], axis=0)
        visible = np.arange(L + kr)[None, :] <= (L + np.arange(kr))[:, None]
        out[i] = attention(q[i], keys, values, visible, shape.group)
    return out
