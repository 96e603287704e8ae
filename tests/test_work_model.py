"""The bench's algorithmic work model (the numerator of every roofline
fraction), checked on the CPU against closed forms for the named workloads."""
import os
import sys
from types import SimpleNamespace

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2608_28099_gb300 import workloads as wl  # noqa: E402


def light(name, lens):
    """The named workload's shape and lengths, without drawing its tensors."""
    spec = wl.named(name)
    lens = np.asarray(lens, dtype=np.int64)
    return SimpleNamespace(shape=spec.shape, seq_ids=np.arange(len(lens)),
                           cache=SimpleNamespace(seq_lens=lens))


def test_27b_long_bytes_and_flops():
    # B = 8 sequences of 32768 cached tokens, 8 KV heads of 128 dims, bf16 K and V
    w = light("27b_long", [32768] * 8)
    st, tot = bench.work_model(w, per_seq_rows=True)
    kv = 8 * 32768 * 8 * 128 * 2 * 2
    assert kv == 1 << 30
    assert tot["kv_bytes"] == kv
    # 128 query rows: rotated queries and new keys/values in (fp32), outputs out (fp32)
    assert st["attention"]["bytes"] == kv + 128 * (40 + 16) * 128 * 4 + 128 * 40 * 128 * 4
    # the seven layer matrices in bf16 (Q/K/V 7168 x 5120, O 5120 x 5120, gate,
    # up and down 17408 x 5120) and the fp32 head
    wq = (7168 * 5120 + 5120 * 5120 + 3 * 17408 * 5120) * 2
    assert tot["weight_bytes"] == wq + 2 * 5120 * 4
    assert abs(tot["weight_bytes"] / 1e6 - 660.6) < 0.1
    # attention flops: 4 dh Hq (k sum L + B k (k + 1) / 2) for QK^T and PV
    assert st["attention"]["flops"] == 4 * 128 * 40 * (16 * 8 * 32768 + 8 * 16 * 17 // 2)
    # every projection is 2 M N K with M = 128 rows
    assert st["gate_up"]["flops"] == 2 * 128 * 2 * 17408 * 5120
    assert st["qkv"]["flops"] == 2 * 128 * 7168 * 5120


def test_shared_prompt_reads_no_qkv_weights():
    # with the shared soft prompt the Q/K/V projection is precomputed at create
    w = light("4b", [256, 2048])
    st, tot = bench.work_model(w, per_seq_rows=False)
    assert "qkv" not in st
    st2, tot2 = bench.work_model(w, per_seq_rows=True)
    assert tot2["weight_bytes"] - tot["weight_bytes"] == (32 + 16) * 128 * 2560 * 2


def test_tasks_and_recursion_scale_as_stated():
    base = light("27b_long", [1000, 3000])
    _, t1 = bench.work_model(base, per_seq_rows=True)
    # recursive SP-k re-reads the cache and every weight once per step
    _, tr = bench.work_model(base, per_seq_rows=True, recursive=True)
    assert tr["kv_bytes"] == 16 * t1["kv_bytes"]
    assert tr["total_bytes"] == 16 * (t1["kv_bytes"] + t1["weight_bytes"])
    # T tasks share one pass over the cache
    multi = SimpleNamespace(shape=wl.named("27b_long", n_tasks=4).shape, seq_ids=base.seq_ids,
                            cache=base.cache)
    _, t4 = bench.work_model(multi, per_seq_rows=True)
    assert t4["kv_bytes"] == t1["kv_bytes"]
