#!/usr/bin/env python
"""Throughput of the Speculative Probing classify path on one GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload 4b] [--impl ours|reference]
    python bench.py --sweep [all|quick] [--steps K] [--warmup W]

One step = one sp_classify call over one batch of the named seeded workload
(every stage of the path: input norm, Q/K/V projection, rotation, split-KV
attention over the resident cache, merge, output projection, post-norm,
gate/up, SwiGLU, down projection, pooling and readout).  Inputs are resident
in HBM before timing; L2 is flushed (a 256 MiB write) between steps; each step
is timed with CUDA events on the launching stream.  Prints one JSON line.

Multi-GPU: the path shards by sequence with no exchange step, so N ranks run N
independent replicas (weak scaling) and `value` counts all ranks' sequences
over the slowest rank's time.

--sweep times the serving sweep at the d=4096 shape (batch x length x k x
classes, bf16 paged caches with +-25% ragged lengths drawn on the device) and
prints one JSON line per point with its stage times, the achieved HBM
fraction and the projections' weight GB/s and TFLOP/s, then a summary line
naming the rows (batch x k) where the projections turn tensor-bound.
"""
from __future__ import annotations

import argparse
import dataclasses
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

# The fp64 oracle's parallelism comes from a pool of worker processes, one per
# host core, each with single-threaded BLAS (fixed before numpy loads), so the
# reported core count is the number of workers that ran.
for _var in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
    os.environ.setdefault(_var, "1")

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "classified sequences/sec and µs/call at 1 GB300; achieved HBM GB/s vs 8 TB/s"
UNIT = "sequences/s"
FALLBACK_HBM_GBS, FALLBACK_BF16_TFLOPS = 6800.0, 1900.0
FLUSH_BYTES = 256 << 20

# DRAM read + write per launch of the dominant kernel, from one ncu capture of
# the current kernel on the same workload; a workload or kernel without such a
# capture reports null.
# The attention kernel's figure includes the output projection's weights that its
# CTAs prefetch into L2 as they finish (52.4 MB on 27b_long, 21 MB on 4b): the next kernel's
# bytes, issued early.
TRAFFIC_BYTES = {("27b_long", "attention"): 1132865280, ("4b", "attention"): 99155712}


def parse_args():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=20)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--workload", default="27b_long",
                   help="tiny, 4b, 8b_paged or 27b_long (default: the largest single-GPU "
                        "configuration, B=8 x L=32768, d=5120, paged)")
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--rows", default="per-seq", choices=["per-seq", "shared", "hidden"],
                   help="per-seq: per-sequence input rows (full layer per call); "
                        "shared: the soft prompt, whose Q/K/V projection is precomputed; "
                        "hidden: base hidden states through the MTP input fusion "
                        "(sp_classify_hidden)")
    p.add_argument("--head", default="linear", choices=["linear", "lm"],
                   help="linear: trained linear head; lm: frozen LM-head rows after the final norm")
    p.add_argument("--tasks", type=int, default=1,
                   help="probes (soft prompt + head) sharing each pass over the cache")
    p.add_argument("--recursive", action="store_true",
                   help="with --rows hidden: recursive probing SP-k (k single-row steps)")
    p.add_argument("--cpu-seconds", type=float, default=12.0)
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--sweep", nargs="?", const="all", default=None, choices=["all", "quick"],
                   help="time the serving-sweep points instead of one workload")
    return p.parse_args()


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            mp = json.load(f)
        return float(mp["hbm_gbs"]), float(mp["bf16_tflops"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, FALLBACK_BF16_TFLOPS, "fallback"


# --------------------------------------------------------------------------- #
# the algorithmic work model (bytes and flops every stage must move/do)
# --------------------------------------------------------------------------- #
def work_model(w, per_seq_rows: bool, fused: bool = False, recursive: bool = False):
    sh = w.shape
    # T tasks stack T k rows per sequence and read T heads
    B, k, d = len(w.seq_ids), sh.k_rows * sh.n_tasks, sh.d_model
    hq, hkv, dh, f, C = sh.n_q_heads, sh.n_kv_heads, sh.head_dim, sh.d_ff, sh.n_classes * sh.n_tasks
    es = 2 if sh.w_dtype == 1 else 4
    kes = 2 if sh.kv_dtype == 1 else 4
    M = B * k
    lens = w.cache.seq_lens[w.seq_ids].astype(np.int64)
    nqkv = (hq + 2 * hkv) * dh

    def gemm(N, K):
        return {"bytes": N * K * es + M * K * es + M * N * es, "flops": 2 * M * N * K}

    st = {}
    if fused:
        # RMSNorm of the B hidden states and their projection by W_fc's hidden half
        st["fusion"] = {"bytes": d * d * es + 2 * B * d * es + M * d * 4, "flops": 2 * B * d * d}
    if per_seq_rows or fused:
        st["qkv"] = gemm(nqkv, d)
    kv_bytes = int(lens.sum()) * hkv * dh * 2 * kes
    st["attention"] = {"bytes": kv_bytes + M * nqkv * 4 + M * hq * dh * 4,
                       "flops": int(4 * dh * hq * (k * lens.sum() + B * k * (k + 1) // 2))}
    st["o_proj"] = gemm(d, hq * dh)
    st["gate_up"] = gemm(2 * f, d)
    st["down"] = gemm(d, f)
    st["readout"] = {"bytes": C * d * 4 + M * d * 4, "flops": 2 * B * C * d}
    total_bytes = sum(v["bytes"] for v in st.values())
    weight_bytes = ((nqkv * d if (per_seq_rows or fused) else 0) + (d * d if fused else 0)
                    + d * hq * dh + 3 * f * d) * es + C * d * 4
    totals = {"kv_bytes": kv_bytes, "weight_bytes": weight_bytes, "total_bytes": total_bytes,
              "total_flops": sum(v["flops"] for v in st.values())}
    if recursive:
        # k steps of one row per sequence: every step reads all weights and the
        # cache again; the flops are those of the parallel form (B k rows in all)
        call = {"bytes": k * (kv_bytes + weight_bytes), "flops": totals["total_flops"]}
        return {"call": call}, {"kv_bytes": k * kv_bytes, "weight_bytes": k * weight_bytes,
                                "total_bytes": call["bytes"], "total_flops": call["flops"]}
    return st, totals


# --------------------------------------------------------------------------- #
# clocks
# --------------------------------------------------------------------------- #
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.out = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"], stdout=self.out,
                stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.3)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.out.close()
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    smax.append(float(parts[2]))
                except ValueError:
                    continue
                for n, v in zip(names, parts[5:9]):
                    if v.lower().startswith("active"):
                        reasons.add(n)
        os.unlink(self.path)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax),
                "reasons": sorted(reasons), "samples": len(sm)}


# --------------------------------------------------------------------------- #
# reference arm: the fp64 oracle on the host cores
# --------------------------------------------------------------------------- #
def cores():
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


# State the oracle workers inherit when the pool forks (set before any CUDA call).
_ORACLE = {}


def _oracle_one(i: int):
    """Classify sequence i % B of the workload with the oracle (one worker)."""
    import oracle.sp_oracle as so
    st = _ORACLE
    w, layer = st["w"], st["layer"]
    i %= len(w.seq_ids)
    rows = w.rows[i:i + 1] if (st["per_seq"] and w.rows is not None) else None
    hid = w.hidden[i:i + 1] if w.hidden is not None else None
    if st["recursive"]:
        so.classify_recursive(layer, w.cache, w.seq_ids[i:i + 1], hid)
    else:
        so.classify(layer, w.cache, w.seq_ids[i:i + 1], rows, hidden=hid)


def _oracle_worker(args):
    """Sequences first, first + stride, ... until `seconds` have passed (at
    least one); returns how many were classified."""
    first, stride, seconds = args
    n, t0 = 0, time.perf_counter()
    while True:
        _oracle_one(first + n * stride)
        n += 1
        if time.perf_counter() - t0 >= seconds:
            return n


def _mem_available() -> int | None:
    try:
        with open("/proc/meminfo") as f:
            for line in f:
                if line.startswith("MemAvailable:"):
                    return int(line.split()[1]) * 1024
    except OSError:
        pass
    return None


class OraclePool:
    """The oracle on the host cores: one single-threaded worker process per
    core (capped by free memory), forked before any CUDA call so that the
    workers share the decoded weights and the workload."""

    def __init__(self, w, per_seq_rows: bool, recursive: bool):
        import multiprocessing as mp

        import oracle.sp_oracle as so
        _ORACLE.update(w=w, layer=so.Layer(w.shape, w.weights), per_seq=per_seq_rows,
                       recursive=recursive)
        sh = w.shape
        # float64 temporaries of one sequence: its gathered K and V, the
        # attention probabilities and the layer's activations (x4 headroom)
        L = int(w.cache.seq_lens[w.seq_ids].max(initial=0)) + sh.k_rows
        per = 8 * (2 * L * sh.n_kv_heads * sh.head_dim + 2 * sh.k_rows * sh.n_q_heads * L
                   + 4 * sh.k_rows * (sh.d_model + sh.d_ff))
        n = cores()
        avail = _mem_available()
        if avail is not None:
            n = max(1, min(n, int(avail // (4 * per + (256 << 20)))))
        self.workers = n
        self.pool = mp.get_context("fork").Pool(n)

    def rate(self, seconds: float):
        """(sequences/s, sequences, seconds) with every worker busy for about
        `seconds` (each finishes the sequence it is on)."""
        t0 = time.perf_counter()
        counts = self.pool.map(_oracle_worker, [(j, self.workers, seconds)
                                                for j in range(self.workers)], chunksize=1)
        el = time.perf_counter() - t0
        return sum(counts) / el, sum(counts), el

    def step(self, first: int):
        """One sequence per worker (first, first + 1, ...): the wall time."""
        t0 = time.perf_counter()
        self.pool.map(_oracle_one, [first + j for j in range(self.workers)], chunksize=1)
        return time.perf_counter() - t0

    def close(self):
        self.pool.close()
        self.pool.join()


def run_reference(args, spec, w, rank, world):
    if rank != 0:
        return
    pool = OraclePool(w, args.rows == "per-seq", recursive_mode(args))
    B = len(w.seq_ids)
    times = []
    for step in range(args.warmup + args.steps):
        el = pool.step(step * pool.workers)
        if step >= args.warmup:
            times.append(el)
    pool.close()
    per_step = pool.workers
    value = per_step * len(times) / sum(times)
    sample = (f"{per_step} sequence(s) of workload {spec.name} (of its {B}) per step, one per "
              f"worker process, {per_step} single-threaded workers; {args.steps} steps after "
              f"{args.warmup} warm-up")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * sum(times) / len(times), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": workload_config(spec, w, args),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": per_step, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def recursive_mode(args) -> bool:
    return bool(args.recursive) and args.rows == "hidden"


def workload_config(spec, w, args):
    sh = w.shape
    lens = w.cache.seq_lens[w.seq_ids]
    return {"workload": spec.name, "batch": len(w.seq_ids),
            "seq_len": (f"{spec.len_lo}" if spec.len_lo == spec.len_hi
                        else f"U[{spec.len_lo},{spec.len_hi}] mean {float(lens.mean()):.0f}"),
            "d_model": sh.d_model, "heads": f"{sh.n_q_heads}q/{sh.n_kv_heads}kv",
            "head_dim": sh.head_dim, "d_ff": sh.d_ff, "k_rows": sh.k_rows,
            "n_classes": sh.n_classes,
            "kv_layout": "paged16" if w.cache.layout == 1 else "contiguous",
            "rows": args.rows, "seed": spec.seed,
            "form": "recursive SP-k" if recursive_mode(args) else "parallel k rows",
            "n_tasks": sh.n_tasks, "head": args.head,
            "l2": "flushed between steps (256 MiB write)",
            "timing": ("CUDA events per step around a CUDA-graph replay of one "
                       + ("sp_classify_hidden" if w.hidden is not None else "sp_classify"))}


# --------------------------------------------------------------------------- #
# ranks
# --------------------------------------------------------------------------- #
def rank_max(x: float, device) -> float:
    """Maximum of x over the ranks of the default process group (x itself when
    there is none): the slowest rank's time."""
    import torch
    import torch.distributed as dist
    if not dist.is_available() or not dist.is_initialized() or dist.get_world_size() == 1:
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def shard_spec(spec, rank: int):
    """Rank r classifies its own batch of the same configuration: an independent
    draw (seed + 1000 r) of the workload."""
    return spec if rank == 0 else dataclasses.replace(spec, seed=spec.seed + 1000 * rank)


# --------------------------------------------------------------------------- #
# our arm
# --------------------------------------------------------------------------- #
def run_ours(args, spec, w, rank, world, oracle_pool=None):
    import torch
    import torch.distributed as dist

    import paper_2608_28099_gb300 as sp
    from paper_2608_28099_gb300 import build_lib

    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    if rank == 0:
        build_lib.build()
    if world > 1:
        dist.barrier()
    sp.load_library()
    per_seq = args.rows == "per-seq"
    B = len(w.seq_ids)
    lens = w.cache.seq_lens
    model = sp.Model(w.shape, w.weights, B, int(lens.max(initial=0)))
    h = model.handle
    recursive = recursive_mode(args)
    if recursive:
        sp.sp_set_option(h, sp.SP_OPT_RECURSIVE, 1)
    cache = sp.DeviceCache(w.cache)
    ids = torch.from_numpy(np.ascontiguousarray(w.seq_ids, dtype=np.int32)).cuda()
    fused = w.hidden is not None
    rows = hidden = None
    if per_seq:
        r = np.ascontiguousarray(w.rows)
        rows = torch.from_numpy(r.view(np.int16) if r.dtype == np.uint16 else r).cuda()
    if fused:
        r = np.ascontiguousarray(w.hidden)
        hidden = torch.from_numpy(r.view(np.int16) if r.dtype == np.uint16 else r).cuda()
    T = w.shape.n_tasks
    logits = torch.empty((B, T, w.shape.n_classes), dtype=torch.float32, device="cuda")
    flush = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device="cuda")
    stream = torch.cuda.current_stream()

    def step():
        # the stream is looked up per call so that a graph capture sees its own
        if fused:
            sp.sp_classify_hidden(h, torch.cuda.current_stream(), B, ids, cache.seq_lens,
                                  cache.desc, hidden, logits)
        else:
            sp.sp_classify(h, torch.cuda.current_stream(), B, ids, cache.seq_lens, cache.desc,
                           rows, logits)

    for _ in range(args.warmup):
        flush.zero_()
        step()
    torch.cuda.synchronize()
    assert sp.sp_check_status(h) == 0, sp.sp_last_error()
    launches_per_step = sp.sp_last_launch_count(h)

    def capture():
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            step()
        torch.cuda.synchronize()
        return g

    def timed(run_once, n):
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(n)]
        for i in range(n):
            flush.zero_()
            ev[i][0].record(stream)
            run_once()
            ev[i][1].record(stream)
        torch.cuda.synchronize()
        return [a.elapsed_time(b) for a, b in ev]

    # one sp_classify call captured in a CUDA graph, replayed per step
    graph = capture()
    for _ in range(args.warmup):
        flush.zero_()
        graph.replay()
    clocks = ClockSampler(local)
    clocks.start()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    step_ms = timed(graph.replay, args.steps)
    if world > 1:
        dist.barrier()
    clk = clocks.stop()
    ms = rank_max(sum(step_ms) / len(step_ms), "cuda")
    assert sp.sp_check_status(h) == 0, sp.sp_last_error()
    eager_ms = sum(timed(step, args.steps)) / args.steps

    # per-stage device times: events the library records around each stage,
    # captured as event nodes of a second graph
    sp.sp_set_option(h, sp.SP_OPT_PROFILE, 1)
    pgraph = capture()
    acc = {}
    for i in range(args.steps):
        flush.zero_()
        pgraph.replay()
        for name, v in sp.sp_stage_times(h).items():
            acc.setdefault(name, []).append(v)
    sp.sp_set_option(h, sp.SP_OPT_PROFILE, 0)
    stage_ms = {k: sum(v) / len(v) for k, v in acc.items()}

    # end to end through the host entry point: pinned inputs up, logits down
    h_ids = torch.from_numpy(np.ascontiguousarray(w.seq_ids, dtype=np.int32)).pin_memory()
    h_lens = torch.from_numpy(np.ascontiguousarray(lens[w.seq_ids], dtype=np.int32)).pin_memory()
    h_rows = rows.cpu().pin_memory() if rows is not None else None
    h_hidden = hidden.cpu().pin_memory() if hidden is not None else None
    h_logits = torch.empty((B, T, w.shape.n_classes), dtype=torch.float32).pin_memory()
    e2e_s = []
    for i in range(args.warmup + args.steps):
        flush.zero_()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        if fused:
            sp.sp_classify_hidden_host(h, stream, B, h_ids, h_lens, cache.desc, h_hidden, h_logits)
        else:
            sp.sp_classify_host(h, stream, B, h_ids, h_lens, cache.desc, h_rows, h_logits)
        el = time.perf_counter() - t0
        if i >= args.warmup:
            e2e_s.append(el)
    e2e_mean = rank_max(sum(e2e_s) / len(e2e_s), "cuda")
    h2d = h_ids.numel() * 4 + h_lens.numel() * 4 + (h_rows.numel() * h_rows.element_size()
                                                     if h_rows is not None else 0)
    if h_hidden is not None:
        h2d += h_hidden.numel() * h_hidden.element_size()
    d2h = h_logits.numel() * 4

    if rank != 0:
        model.close()
        return
    hbm, tfl, peak_src = peaks()
    st_work, totals = work_model(w, per_seq, fused, recursive)
    # dominant kernel: the stage with the largest device time
    named = {"attention": "attention", "qkv": "qkv", "o_proj": "o_proj", "gate_up": "gate_up",
             "down": "down", "readout": "readout", "fusion": "fusion"}
    cand = {k: v for k, v in stage_ms.items() if k in named and k in st_work}
    if not cand:  # no per-stage markers (recursive form): the whole call
        stage_ms = dict(stage_ms, call=ms)
        cand = {"call": ms}
    dom = max(cand, key=cand.get)
    wk = st_work[dom]
    dur_s = stage_ms[dom] / 1e3
    intensity = wk["flops"] / wk["bytes"]
    ridge = tfl * 1e12 / (hbm * 1e9)
    if intensity > ridge:
        bound, ach, peak, unit = "tensor", wk["flops"] / dur_s / 1e12, tfl, "TFLOP/s"
    else:
        bound, ach, peak, unit = "hbm", wk["bytes"] / dur_s / 1e9, hbm, "GB/s"
    traffic = TRAFFIC_BYTES.get((spec.name, dom))
    roofline = {"bound": bound, "kernel": dom, "achieved": ach, "peak": peak, "unit": unit,
                "frac": ach / peak, "traffic": traffic,
                "peak_source": f"{peak_src} ({'hbm_gbs' if bound == 'hbm' else 'bf16_tflops'})",
                "algorithmic_bytes": wk["bytes"], "algorithmic_flops": wk["flops"],
                "ms": stage_ms[dom]}
    path_bytes = totals["total_bytes"]
    cpu = None
    if oracle_pool is not None:
        rate, n, el = oracle_pool.rate(args.cpu_seconds)
        cpu = {"value": rate, "unit": UNIT, "cores": oracle_pool.workers, "kind": "oracle",
               "sample": f"{n} sequences of workload {spec.name} over {el:.1f} s, one sequence "
                         f"at a time per worker process, {oracle_pool.workers} single-threaded "
                         f"workers"}
        oracle_pool.close()
    value = world * B / (ms / 1e3)
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "us_per_call": ms * 1e3,
            "eager_ms_per_step": eager_ms,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16"
            if w.shape.w_dtype == 1 else "f32", "data": "synthetic (seeded, random-init)",
            "config": workload_config(spec, w, args),
            "hbm": {"algorithmic_bytes_per_call": path_bytes,
                    "gbs": path_bytes / (ms / 1e3) / 1e9,
                    "frac_of_8tbs": path_bytes / (ms / 1e3) / 8e12,
                    "frac_of_measured": path_bytes / (ms / 1e3) / (hbm * 1e9),
                    "kv_bytes": totals["kv_bytes"], "weight_bytes": totals["weight_bytes"]},
            "roofline": roofline,
            "stages_ms": stage_ms,
            "cpu_baseline": cpu,
            "e2e": {"value": world * B / e2e_mean, "unit": UNIT, "h2d_bytes_per_step": h2d,
                    "d2h_bytes_per_step": d2h, "ms_per_step": e2e_mean * 1e3},
            "gpu_launches": launches_per_step * args.steps,
            "clocks": clk}
    print(json.dumps(line), flush=True)
    model.close()


# --------------------------------------------------------------------------- #
# serving sweep
# --------------------------------------------------------------------------- #
QUICK_SWEEP = [f"sweep_B{B}_L{L}_k{k}_C16" for B in (1, 32, 256) for L in (512, 8192)
               for k in (1, 16)]


def run_sweep(args):
    import torch

    import paper_2608_28099_gb300 as sp
    from paper_2608_28099_gb300 import build_lib
    from paper_2608_28099_gb300 import workloads as wl

    torch.cuda.set_device(0)
    build_lib.build()
    sp.load_library()
    hbm, tfl, peak_src = peaks()
    tfl_sus = tfl
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            tfl_sus = float(json.load(f).get("bf16_tflops_sustained", tfl))
    except Exception:
        pass
    names = wl.SWEEP_POINTS if args.sweep == "all" else QUICK_SWEEP
    specs = [wl.named(n, rows_per_seq=True) for n in names]
    flush = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device="cuda")
    max_len = max(s.len_hi for s in specs)
    max_b = max(s.batch for s in specs)
    models, base_w = {}, None
    by_bl = {}
    for s in specs:
        by_bl.setdefault((s.batch, s.len_lo, s.len_hi), []).append(s)
    results = []
    clocks = ClockSampler(0)
    clocks.start()
    for (B, lo, hi), group in by_bl.items():
        dev = None
        for s in group:
            k, C = s.shape.k_rows, s.shape.n_classes
            if (k, C) not in models:
                sw = wl.generate_on_device(s)  # weights for this (k, C); pools discarded
                del sw.k_pool, sw.v_pool
                models[(k, C)] = (sp.Model(s.shape, sw.weights, max_b, max_len), sw.weights)
            model, weights = models[(k, C)]
            dw = wl.generate_on_device(s, weights=weights)
            cache = sp.DevicePagedCache(dw)
            h = model.handle
            ids = torch.arange(B, dtype=torch.int32, device="cuda")
            r = np.ascontiguousarray(dw.rows)
            rows = torch.from_numpy(r.view(np.int16)).cuda()
            logits = torch.empty((B, C), dtype=torch.float32, device="cuda")

            def step():
                sp.sp_classify(h, torch.cuda.current_stream(), B, ids, cache.seq_lens, cache.desc,
                               rows, logits)

            for _ in range(args.warmup):
                step()
            torch.cuda.synchronize()
            assert sp.sp_check_status(h) == 0, sp.sp_last_error()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                step()
            torch.cuda.synchronize()
            times = []
            for _ in range(args.steps):
                flush.zero_()
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record()
                g.replay()
                e1.record()
                torch.cuda.synchronize()
                times.append(e0.elapsed_time(e1))
            ms = statistics.median(times)
            sp.sp_set_option(h, sp.SP_OPT_PROFILE, 1)
            pg = torch.cuda.CUDAGraph()
            with torch.cuda.graph(pg):
                step()
            acc = {}
            for _ in range(max(3, args.steps // 2)):
                flush.zero_()
                pg.replay()
                for nme, v in sp.sp_stage_times(h).items():
                    acc.setdefault(nme, []).append(v)
            sp.sp_set_option(h, sp.SP_OPT_PROFILE, 0)
            stage_us = {nme: 1e3 * statistics.median(v) for nme, v in acc.items()}
            assert sp.sp_check_status(h) == 0, sp.sp_last_error()
            fake = wl.Workload(s, weights, wl.KVCache(wl.LAYOUT_PAGED, wl.BF16, dw.seq_lens),
                               dw.seq_ids, dw.rows)
            st_work, totals = work_model(fake, True)
            proj = [n for n in ("qkv", "o_proj", "gate_up", "down") if n in st_work]
            p_bytes = sum(st_work[n]["bytes"] for n in proj)
            p_flops = sum(st_work[n]["flops"] for n in proj)
            p_us = sum(stage_us.get(n, 0.0) for n in proj)
            M = B * k
            hbm_floor = p_bytes / (hbm * 1e9) * 1e6
            # MMA work issued: Q/K/V and O always take hi + lo activations (two
            # passes); gate/up and down take plain bf16 when the mean pools >= 8 rows
            mlp_passes = 1 if k >= 8 else 2
            issued = sum(st_work[n]["flops"] * (mlp_passes if n in ("gate_up", "down") else 2)
                         for n in proj)
            tensor_floor = issued / (tfl_sus * 1e12) * 1e6
            line = {"sweep_point": s.name, "B": B, "L": f"U[{lo},{hi}]", "k": k, "C": C,
                    "rows": M, "us_per_call": ms * 1e3, "seq_per_s": B / (ms / 1e3),
                    "hbm_gbs": totals["total_bytes"] / (ms / 1e3) / 1e9,
                    "frac_of_8tbs": totals["total_bytes"] / (ms / 1e3) / 8e12,
                    "frac_of_measured": totals["total_bytes"] / (ms / 1e3) / (hbm * 1e9),
                    "attention": {"us": stage_us.get("attention"),
                                  "gbs": st_work["attention"]["bytes"] / (stage_us.get("attention", 1e9) * 1e3)},
                    "projections": {"us": p_us, "weight_gbs": p_bytes / (p_us * 1e3) if p_us else None,
                                    "tflops": p_flops / (p_us * 1e6) if p_us else None,
                                    "hbm_floor_us": hbm_floor, "tensor_floor_us": tensor_floor,
                                    "bound": "tensor" if tensor_floor > hbm_floor else "hbm"},
                    "stages_us": stage_us}
            results.append(line)
            print(json.dumps(line), flush=True)
            del g, pg, cache, dw
            torch.cuda.empty_cache()
    clk = clocks.stop()
    tensor_rows = sorted({r["rows"] for r in results if r["projections"]["bound"] == "tensor"})
    hbm_rows = sorted({r["rows"] for r in results if r["projections"]["bound"] == "hbm"})
    summary = {"sweep": args.sweep, "points": len(results),
               "projection_crossover": {"largest_hbm_bound_rows": max(hbm_rows) if hbm_rows else None,
                                        "smallest_tensor_bound_rows": min(tensor_rows) if tensor_rows else None,
                                        "note": "tensor floor counts two MMA passes for hi + lo "
                                                "activations (Q/K/V, O; the MLP when k < 8) and one "
                                                "for plain bf16; the same tcgen05 kernels serve both "
                                                "sides"},
               "peaks": {"hbm_gbs": hbm, "bf16_tflops_sustained": tfl_sus, "source": peak_src},
               "clocks": clk, "steps": args.steps, "warmup": args.warmup,
               "l2": "flushed between steps (256 MiB write)"}
    print(json.dumps(summary), flush=True)
    for m, _ in models.values():
        m.close()


def main():
    args = parse_args()
    if args.sweep:
        run_sweep(args)
        return
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        if args.impl == "reference":
            if rank != 0:
                return
        else:
            import torch
            torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", "0")))
            dist.init_process_group("nccl")
    from paper_2608_28099_gb300 import workloads as wl
    spec = shard_spec(wl.named(args.workload, rows_per_seq=(args.rows == "per-seq"),
                               fused=(args.rows == "hidden"), n_tasks=max(1, args.tasks)), rank)
    w = wl.generate(spec)
    if args.head == "lm":
        w = wl.with_lm_head(w)
    if args.impl == "reference":
        run_reference(args, spec, w, rank, world)
    else:
        # the oracle's worker pool forks here, before this process touches CUDA
        pool = None
        if world == 1 and not args.no_cpu_baseline:
            pool = OraclePool(w, args.rows == "per-seq", recursive_mode(args))
        run_ours(args, spec, w, rank, world, pool)
    if world > 1 and args.impl != "reference":
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
