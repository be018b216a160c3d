"""Benchmark of the evicted decode step on GB300.

Workload (default): Qwen2.5-Math-7B decode geometry (28 layers, 28 query /
4 KV heads, head_dim 128, bf16), a batch of 64 independent sequences with
prior context lengths drawn uniformly from [512, 16384], budget B=64 and
recent window W=8.  The prompts are loaded with zero scores; the first decode
step evicts each unit down to B+W (timed separately as `first_step_ms`); the
sequences then move into a steady-state cache of capacity B+W+1 (a dense
slab; `kvr_cache_copy_sequences`, timed as `move_to_steady_cache_ms`), and
every step after that is the steady state: append, attend over B+W+1 rows,
accumulate scores, evict one row per (sequence, layer, KV head).

One "step" = one decode token for all 64 sequences and all 28 layers, run as
one kvr_decode_step call over every layer.  `value` is steps/s with inputs
resident in HBM; `e2e` is the same metric with the step's q/k/v copied from
pinned host memory and its output copied back inside the timed region.

`python bench.py --impl reference` times the fp64 CPU oracle on the same
workload instead (a bounded sample: one of the 64 sequences per step,
extrapolated to the whole batch).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2608_15797_gb300 import cost_model, inputs  # noqa: E402

NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=4000)
    p.add_argument("--warmup", type=int, default=50)
    p.add_argument("--impl", default="kvr", choices=["kvr", "reference"])
    p.add_argument("--workload", default="7b_s64_b64")
    p.add_argument("--seed", type=int, default=0)
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--cpu-seconds", type=float, default=15.0)
    p.add_argument("--cpu-all-seconds", type=float, default=8.0,
                   help="oracle seconds per process for the all-cores rate")
    p.add_argument("--per-layer-steps", type=int, default=500,
                   help="steps timed as one launch per layer")
    p.add_argument("--latency-steps", type=int, default=1000,
                   help="steps of the single-sequence latency run")
    p.add_argument("--prior-min", type=int, default=inputs.PRIOR_LEN_RANGE[0],
                   help="shortest prior context (profiling uses a small case)")
    p.add_argument("--prior-max", type=int, default=inputs.PRIOR_LEN_RANGE[1])
    p.add_argument("--e2e-steps", type=int, default=1000)
    p.add_argument("--repeats", type=int, default=7,
                   help="the headline's K-step region is timed this many "
                        "times; value is the median")
    p.add_argument("--no-rows", action="store_true",
                   help="skip the other rows' sub-records of the default line")
    p.add_argument("--fused-groups", type=int, default=0,
                   help="units computed at once per SM by the fused kernel "
                        "(0: the library's choice)")
    p.add_argument("--mode", default="step",
                   choices=["step", "helper", "fork", "fork-copy", "rkv",
                            "crossover", "absorb", "entropy"],
                   help="step: the evicted decode step (the headline); "
                        "helper: full-context decode of the 1.5B helper at "
                        "16k context; fork: 72B best-of-8 candidate step")
    p.add_argument("--entropy-dtype", default="bf16", choices=["bf16", "f32"],
                   help="logit element type for --mode entropy")
    p.add_argument("--fork-kernel", type=int, default=0, choices=[0, 1, 2, 3, 4],
                   help="--mode fork candidate kernel (kvr_fork_set_kernel): "
                        "0 library's choice, 1 batched, 2 chunked, 3 one CTA "
                        "a unit, 4 generic")
    p.add_argument("--absorb-kernel", type=int, default=0, choices=[0, 1],
                   help="--mode absorb kernel: 0 tcgen05 (tensor memory), "
                        "1 mma.sync")
    p.add_argument("--entropy-kernel", type=int, default=0, choices=[0, 1, 2],
                   help="--mode entropy kernel: 0 library's choice, "
                        "1 persistent streaming, 2 one CTA per piece")
    p.add_argument("--seqs", type=int, default=0,
                   help="sequences for --mode helper/fork/absorb/rkv "
                        "(0: 16 / 4 / 64 / 64)")
    p.add_argument("--chunk-groups", type=int, default=0,
                   help="chunked kernel: consumer groups per SM (0 auto, -1 off)")
    p.add_argument("--chunk-stages", type=int, default=0,
                   help="chunked kernel: ring stages per group (0 auto)")
    p.add_argument("--fused-group-warps", type=int, default=0,
                   help="warps sharing one unit in the fused kernel "
                        "(0: the library's choice)")
    return p.parse_args()


def metric_name(w):
    return (f"evicted decode steps/s at 7B geometry, B={w.budget}, W={w.window}"
            f" ({w.n_seq} sequences x {w.n_layers} layers per step)")


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            return json.load(f), "measured"
    return {"hbm_gbs": FALLBACK_HBM_GBS}, "fallback"


# --------------------------------------------------------------------------
# CPU oracle timing (the reference arm and the cpu_baseline field)
# --------------------------------------------------------------------------

def oracle_rate(w, seed, max_seconds, max_steps=None):
    from oracle import oracle as orc
    L, H, G, d = w.n_layers, w.n_kv_heads, w.group, w.head_dim
    m = w.budget + w.window
    o = orc.OracleCache(1, L, H, G, d, cap=m + 1)
    k, v = inputs.prompt(w, seed, 0, m)
    o.load(0, k, v, first_pos=16384 - m)
    pre = [inputs.step_inputs(w, seed, i, 1) for i in range(8)]
    o.step(*pre[0], B=w.budget, W=w.window)
    spent, n = 0.0, 0
    while spent < max_seconds and (max_steps is None or n < max_steps):
        q, kn, vn = pre[(n + 1) % len(pre)]
        t = time.perf_counter()
        o.step(q, kn, vn, B=w.budget, W=w.window)
        spent += time.perf_counter() - t
        n += 1
    per_seq_step = spent / n
    # one step of the workload = n_seq sequences
    return 1.0 / (per_seq_step * w.n_seq), n, spent


def oracle_rate_batch(w, seed, steps, warmup, budget_s=120.0):
    """The reference arm: the fp64 oracle stepping the workload's whole
    batch (w.n_seq sequences, every layer and KV head) from the steady state
    (B + W rows a unit; the first eviction from the prior context is, as in
    the GPU arm, not part of the metric), `warmup` untimed steps then
    `steps` timed ones, on one core.  Where `steps` full-batch steps would
    not fit in budget_s, each step takes the first s < n_seq sequences and
    the rate is scaled to the batch (reported).  Returns (rate in batch
    steps/s, timed seconds, sequences a step)."""
    from oracle import oracle as orc
    L, H, G, d = w.n_layers, w.n_kv_heads, w.group, w.head_dim
    m = w.budget + w.window
    per_seq = 1.0 / (oracle_rate(w, seed, 0.5)[0] * w.n_seq)  # s a sequence-step
    S = int(max(1, min(w.n_seq, budget_s / max(1e-9, per_seq * (steps + warmup)))))
    o = orc.OracleCache(S, L, H, G, d, cap=m + 1)
    for sq in range(S):
        k, v = inputs.prompt(w, seed, sq, m)
        o.load(sq, k, v, first_pos=16384 - m)
    pre = [inputs.step_inputs(w, seed, i, S) for i in range(4)]
    o.step(*pre[0], B=w.budget, W=w.window)
    for i in range(warmup):
        o.step(*pre[(i + 1) % 4], B=w.budget, W=w.window)
    t0 = time.perf_counter()
    for i in range(steps):
        o.step(*pre[i % 4], B=w.budget, W=w.window)
    spent = time.perf_counter() - t0
    return steps * (S / w.n_seq) / spent, spent, S


def _oracle_worker(job):
    workload, seed, seconds = job
    w = inputs.WORKLOADS[workload]
    rate, n, spent = oracle_rate(w, seed, seconds)
    return rate, n, spent


def oracle_rate_all_cores(workload, seed, seconds, procs):
    """The same oracle sample on `procs` processes at once (one sequence
    each, started with spawn); returns the summed rate in steps/s."""
    import multiprocessing as mp
    with mp.get_context("spawn").Pool(procs) as pool:
        res = pool.map(_oracle_worker,
                       [(workload, seed + 101 * i, seconds) for i in range(procs)])
    return sum(r for r, _, _ in res), sum(n for _, n, _ in res)


# --------------------------------------------------------------------------
# clocks sampled during the timed region
# --------------------------------------------------------------------------

class ClockSampler:
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,"
             "clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
             "clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,"
             "clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.lines = []
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.QUERY,
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()
        t0 = time.time()
        while not self.lines and time.time() - t0 < 5:
            time.sleep(0.02)

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.time(), line.strip()))

    def mark(self):
        return time.time()

    def stop(self, t_begin, t_end):
        if self.proc is None:
            return None
        time.sleep(0.1)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        rows = [l for t, l in self.lines if t_begin <= t <= t_end + 0.05]
        if not rows:
            rows = [l for _, l in self.lines[-3:]]
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown",
                 "sw_power_cap"]
        for r in rows:
            f = [x.strip() for x in r.split(",")]
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except (ValueError, IndexError):
                continue
            for nm, val in zip(names, f[5:9]):
                if val.lower() == "active":
                    reasons.add(nm)
        if not sm:
            return None
        return {"sm_mhz": float(np.median(sm)), "sm_max_mhz": max(mx),
                "reasons": sorted(reasons), "samples": len(sm)}


# --------------------------------------------------------------------------
# the CUDA arm
# --------------------------------------------------------------------------

def kernel_source_hash(files):
    """sha256 (16 hex digits) of the named files under csrc/, in order."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2608_15797_gb300", "csrc")
    for fn in files:
        with open(os.path.join(csrc, fn), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def committed_traffic(name):
    """DRAM bytes per launch from the committed ncu summary profiles/<name>
    .json, if it was taken on the current sources of that kernel (the files
    it lists)."""
    path = os.path.join(ROOT, "profiles", f"{name}.json")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        d = json.load(f)
    files = d.get("kernel_sources")
    if not files or d.get("kernel_sources_sha") != kernel_source_hash(files):
        return None
    return d.get("dram_bytes_per_launch")


# --------------------------------------------------------------------------
# ranks: weak scaling, each rank its own sequences, no data-path collective
# --------------------------------------------------------------------------

def headline_config(args, w):
    """The config of the default line, the same on both arms."""
    launch_bytes = cost_model.step_unit_bytes(
        w.budget + w.window, w.head_dim, w.group, 2, 2, w.budget,
        w.window) * w.n_seq * w.n_layers * w.n_kv_heads
    return {"workload": args.workload, "n_seq": w.n_seq,
            "layers": w.n_layers, "kv_heads": w.n_kv_heads,
            "group": w.group, "head_dim": w.head_dim,
            "budget": w.budget, "window": w.window,
            "prior_len": f"U[{args.prior_min},{args.prior_max}]",
            "steady_capacity": w.budget + w.window + 1,
            "elem": "bf16",
            "l2": f"inputs larger than L2: {launch_bytes / 1e6:.0f} MB"
                  " touched per step, no flush",
            "per_rank_sequences": w.n_seq}


def rank_seeds(seed, rank):
    """Seeds of rank `rank`'s prior lengths and of its inputs: every rank
    decodes its own sequences (weak scaling)."""
    return seed + 7919 * rank, 1_000_003 * (seed + 1) + rank


def max_over_ranks(x, device=None):
    """The largest of every rank's x (the job ends with its slowest rank);
    x itself outside a process group of more than one rank."""
    import torch
    dist = torch.distributed
    if not (dist.is_available() and dist.is_initialized()) or \
            dist.get_world_size() == 1:
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(world, units_per_rank, max_ms):
    """Whole-job throughput: the units all ranks processed over the slowest
    rank's time."""
    return world * units_per_rank / (max_ms / 1e3)


def run_kvr(args, rank, world, local_rank):
    import torch
    from paper_2608_15797_gb300 import kvr

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    w = inputs.WORKLOADS[args.workload]
    S, L, H, G, d = w.n_seq, w.n_layers, w.n_kv_heads, w.group, w.head_dim
    B, W = w.budget, w.window
    len_seed, in_seed = rank_seeds(args.seed, rank)
    lens = inputs.prior_lengths(len_seed, S, args.prior_min, args.prior_max)
    cap = int(lens.max()) + 1
    cache = kvr.Cache(S, L, H, G, d, cap, kv_dtype="bf16", out_dtype="bf16",
                      device=dev)
    if args.fused_groups or args.fused_group_warps:
        kvr.kvr_cache_set_fused_tuning(cache.handle, args.fused_groups,
                                       args.fused_group_warps)
    if args.chunk_groups or args.chunk_stages:
        kvr.kvr_cache_set_chunk_tuning(cache.handle, args.chunk_groups,
                                       args.chunk_stages)
    gen = torch.Generator(device=dev)
    gen.manual_seed(in_seed)
    for s in range(S):
        n = int(lens[s])
        k = (torch.randn(L, H, n, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
        v = (torch.randn(L, H, n, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
        cache.load(s, k, v)
        del k, v
    torch.cuda.synchronize()

    n_pool = 16
    pool = []
    for _ in range(n_pool):
        q = (torch.randn(S, L, H * G, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
        kn = (torch.randn(S, L, H, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
        vn = (torch.randn(S, L, H, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
        pool.append((q, kn, vn))
    out = torch.empty(S, L, H * G, d, dtype=torch.bfloat16, device=dev)
    stream = torch.cuda.current_stream(dev)

    # First step: evicts every unit from its prior length down to B + W.
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    kvr.kvr_decode_step(cache.handle, 0, L, *pool[0], out, B, W, stream)
    ev1.record(stream)
    torch.cuda.synchronize()
    first_ms = ev0.elapsed_time(ev1)
    cache.sync_status()
    assert (cache.lengths() == B + W).all()
    # The prompt-sized cache (capacity max prior + 1, a 4 MB unit stride at
    # 16k) served only the first eviction: every sequence moves into a
    # steady-state cache of capacity B + W + 1, a dense slab, through the
    # library's sequence copy, and the timed steps run there.
    steady = kvr.Cache(S, L, H, G, d, B + W + 1, kv_dtype="bf16",
                       out_dtype="bf16", device=dev)
    if args.fused_groups or args.fused_group_warps:
        kvr.kvr_cache_set_fused_tuning(steady.handle, args.fused_groups,
                                       args.fused_group_warps)
    if args.chunk_groups or args.chunk_stages:
        kvr.kvr_cache_set_chunk_tuning(steady.handle, args.chunk_groups,
                                       args.chunk_stages)
    ev0.record(stream)
    steady.copy_from(cache, np.arange(S, dtype=np.int32),
                     np.arange(S, dtype=np.int32), stream)
    ev1.record(stream)
    torch.cuda.synchronize()
    move_ms = ev0.elapsed_time(ev1)
    del cache
    torch.cuda.empty_cache()
    cache = steady
    cache.sync_status()

    def step(i):
        q, kn, vn = pool[i % n_pool]
        kvr.kvr_decode_step(cache.handle, 0, L, q, kn, vn, out, B, W, stream)

    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize()

    K = args.steps
    # Two events bracket the K steps: an event between launches would stop
    # a launch from overlapping the tail of the one before it.  The K-step
    # region is timed `repeats` times (each bracketed by a barrier and a
    # synchronize on both sides); the value is the median region.
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    sampler = ClockSampler(local_rank) if rank == 0 else None
    if sampler:
        sampler.start()
    regions, launches = [], 0
    t_begin = time.time()
    for rep in range(max(1, args.repeats)):
        if world > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize()
        launches0 = cache.launch_count()
        t0.record(stream)
        for i in range(K):
            step(rep * K + i)
        t1.record(stream)
        torch.cuda.synchronize()
        launches = cache.launch_count() - launches0
        if world > 1:
            torch.distributed.barrier()
        regions.append(max_over_ranks(t0.elapsed_time(t1), dev))
    t_end = time.time()
    clocks = sampler.stop(t_begin, t_end) if sampler else None
    total_ms = float(np.median(regions))
    # One launch per steady-state step: the average launch duration is the
    # region's time over its launches (gaps between launches included).
    per_launch_ms = total_ms / max(1, launches)
    cache.sync_status()

    # The same steady-state steps as one launch per layer (L calls a step),
    # each layer's inputs and output contiguous.
    Kl = max(1, min(K, args.per_layer_steps))
    lpool = [[tuple(x[:, l:l + 1].contiguous() for x in pool[i])
              for l in range(L)] for i in range(4)]
    lout = [torch.empty(S, 1, H * G, d, dtype=torch.bfloat16, device=dev)
            for _ in range(L)]

    def layer_step(i):
        for l in range(L):
            q, kn, vn = lpool[i % 4][l]
            kvr.kvr_decode_step(cache.handle, l, l + 1, q, kn, vn, lout[l], B,
                                W, stream)

    for i in range(3):
        layer_step(i)
    torch.cuda.synchronize()
    t0.record(stream)
    for i in range(Kl):
        layer_step(i)
    t1.record(stream)
    torch.cuda.synchronize()
    per_layer_ms = t0.elapsed_time(t1) / Kl
    cache.sync_status()
    del lpool, lout

    # End to end through the public call with HOST buffers
    # (kvr_decode_step_host): every step's inputs copied in from pinned host
    # memory and its output copied back by the library, inside the timed
    # region.
    hpool = [tuple(x.cpu().pin_memory() for x in p) for p in pool[:4]]
    # Six staging sets: a stream's next copy-in queues behind its previous
    # step's copy-out, so a deeper rotation keeps the copy engines busy
    # (measured: 115.5 us a step at three, 111.5 at six; the copies alone
    # take 95.5 us a step over the host link).
    n_str = 6
    hout = [torch.empty(out.shape, dtype=out.dtype).pin_memory()
            for _ in range(n_str)]
    bi = sum(x.numel() * x.element_size() for x in hpool[0])
    bo = hout[0].numel() * hout[0].element_size()
    Ke = max(1, min(K, args.e2e_steps))
    stage = [tuple(torch.empty_like(x) for x in pool[0]) + (torch.empty_like(out),)
             for _ in range(n_str)]

    # Serial: copy in, decode, copy out, one stream.
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    e0.record(stream)
    for i in range(Ke):
        kvr.kvr_decode_step_host(cache.handle, 0, L, *hpool[i % len(hpool)],
                                 hout[0], *stage[0], B, W, stream)
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_serial_ms = max_over_ranks(e0.elapsed_time(e1), dev)

    # Pipelined (a serving loop): step i on stream i % 6 with staging set
    # i % 6; the library orders the steps, so step i + 1's copy in and step
    # i - 1's copy out overlap step i's compute.
    strs = [torch.cuda.Stream(dev) for _ in range(n_str)]
    torch.cuda.synchronize()
    e0.record(strs[0])
    for x in strs[1:]:
        x.wait_event(e0)
    for i in range(Ke):
        j = i % n_str
        kvr.kvr_decode_step_host(cache.handle, 0, L, *hpool[i % len(hpool)],
                                 hout[j], *stage[j], B, W, strs[j])
    for x in strs[1:]:
        ev = torch.cuda.Event()
        ev.record(x)
        strs[0].wait_event(ev)
    e1.record(strs[0])
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(e0.elapsed_time(e1), dev)
    cache.sync_status()

    unit_bytes = cost_model.step_unit_bytes(B + W, d, G, 2, 2, B, W)
    launch_bytes = unit_bytes * S * L * H
    return dict(total_ms=total_ms, per_launch_ms=per_launch_ms, K=K,
                regions=regions, per_layer_ms=per_layer_ms, Kl=Kl,
                first_ms=first_ms, move_ms=move_ms, clocks=clocks,
                e2e_ms=e2e_ms, Ke=Ke,
                e2e_serial_ms=e2e_serial_ms,
                bi=bi, bo=bo, launch_bytes=launch_bytes, lens=lens,
                launches=launches)


def run_latency_s1(args, local_rank):
    """Single-sequence 7B decode (prompt 512, B=64, W=8): steady-state
    step latency over all 28 layers, one launch per step.  The working set
    (4.8 MB) stays in L2, so this is a latency figure, not a bandwidth one."""
    import torch
    from paper_2608_15797_gb300 import kvr
    dev = torch.device("cuda", local_rank)
    w = inputs.WORKLOADS["7b_b64"]
    S, L, H, G, d = 1, w.n_layers, w.n_kv_heads, w.group, w.head_dim
    cache = kvr.Cache(S, L, H, G, d, w.prompt + 1, kv_dtype="bf16",
                      out_dtype="bf16", device=dev)
    k, v = inputs.prompt(w, args.seed, 0, w.prompt)
    bf = torch.bfloat16
    cache.load(0, torch.from_numpy(k).to(dev).to(bf),
               torch.from_numpy(v).to(dev).to(bf))
    pool = []
    for i in range(8):
        q, kn, vn = inputs.step_inputs(w, args.seed, i, 1)
        pool.append(tuple(torch.from_numpy(x).to(dev).to(bf) for x in (q, kn, vn)))
    out = torch.empty(S, L, H * G, d, dtype=torch.bfloat16, device=dev)
    stream = torch.cuda.current_stream(dev)
    for i in range(30):
        kvr.kvr_decode_step(cache.handle, 0, L, *pool[i % 8], out, w.budget,
                            w.window, stream)
    torch.cuda.synchronize()
    K = max(1, args.latency_steps)
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for i in range(K):
        kvr.kvr_decode_step(cache.handle, 0, L, *pool[i % 8], out, w.budget,
                            w.window, stream)
    t1.record(stream)
    torch.cuda.synchronize()
    cache.sync_status()
    return {"workload": "7b_b64 (1 sequence, prompt 512, B=64, W=8)",
            "us_per_step": t0.elapsed_time(t1) * 1e3 / K, "steps": K}


# --------------------------------------------------------------------------
# other rows of the path: full-context helper decode, candidate steps
# --------------------------------------------------------------------------

def _timed(fn, K, stream):
    import torch
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(K)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(K)]
    torch.cuda.synchronize()
    for i in range(K):
        starts[i].record(stream)
        fn(i)
        ends[i].record(stream)
    torch.cuda.synchronize()
    total = starts[0].elapsed_time(ends[-1])
    per = sum(a.elapsed_time(b) for a, b in zip(starts, ends)) / K
    return total, per


def run_helper(args):
    """1.5B helper geometry (28 layers, 12 q / 2 kv heads, d 128) at context
    16384: append + attention over every row, no scores, no eviction."""
    import torch
    from paper_2608_15797_gb300 import kvr
    w = inputs.WORKLOADS["1p5b_full16k"]
    S = args.seqs or 16
    L, H, G, d, ctx = w.n_layers, w.n_kv_heads, w.group, w.head_dim, w.prompt
    K, Wm = args.steps, args.warmup
    dev = torch.device("cuda", 0)
    cache = kvr.Cache(S, L, H, G, d, ctx + K + Wm + 1, "bf16", "bf16", device=dev)
    gen = torch.Generator(device=dev)
    gen.manual_seed(args.seed + 17)
    for s in range(S):
        k = (torch.randn(L, H, ctx, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
        v = (torch.randn(L, H, ctx, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
        cache.load(s, k, v)
        del k, v
    q = (torch.randn(S, L, H * G, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
    kn = (torch.randn(S, L, H, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
    vn = (torch.randn(S, L, H, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
    out = cache.new_out(L)
    need = kvr.kvr_decode_attend_workspace_bytes(cache.handle, 0, L, 0)
    ws = torch.empty(need, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)

    def step(i):
        kvr.kvr_decode_attend(cache.handle, 0, L, q, kn, vn, out, 0, ws,
                              ws.numel(), stream)

    for i in range(Wm):
        step(i)
    n0 = cache.launch_count()
    total, per = _timed(step, K, stream)
    launches = cache.launch_count() - n0
    cache.sync_status()
    m_mean = ctx + Wm + (K - 1) / 2.0  # rows before the append, mean over steps
    per_unit = cost_model.attend_full_unit_bytes(m_mean, d, G, 2, 2)
    launch_bytes = per_unit * S * L * H
    return dict(metric=f"full-context helper decode steps/s (1.5B geometry, "
                       f"context {ctx}, {S} sequences x {L} layers per step)",
                total_ms=total, per_ms=per, K=K, launches=launches,
                launch_bytes=launch_bytes,
                config={"workload": "1p5b_full16k", "n_seq": S, "layers": L,
                        "kv_heads": H, "group": G, "head_dim": d,
                        "context": ctx, "splits": "auto"},
                kernel="kvr_decode_attend (split partials + combine)")


def run_crossover(args):
    """The attention-side crossover of App. D (Eq. 14) measured on this GPU
    at 7B geometry: full-context decode attention (append + attention over
    every row, no scores; kvr_decode_attend) against the evicted step
    (append + attention + scores + selection + compaction over B' = B + W
    rows; kvr_decode_step), both over all 28 layers of S sequences.
    t_full(l) is measured at contexts from 64 to 16384 and fitted as
    a + b l; alpha = t_evict / t_full(B') - 1 and l* = (t_evict - a) / b,
    the context past which the evicted step is the cheaper one."""
    import torch
    from paper_2608_15797_gb300 import kvr
    w = inputs.WORKLOADS["7b_b64"]
    S = args.seqs or 16
    L, H, G, d = w.n_layers, w.n_kv_heads, w.group, w.head_dim
    dev = torch.device("cuda", 0)
    stream = torch.cuda.current_stream(dev)
    K, Wm = max(1, min(args.steps, 40)), max(3, args.warmup)
    gen = torch.Generator(device=dev)
    gen.manual_seed(args.seed + 31)

    def inputs_for(S):
        q = (torch.randn(S, L, H * G, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
        kn = (torch.randn(S, L, H, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
        vn = (torch.randn(S, L, H, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
        return q, kn, vn

    def loaded(rows, cap):
        cache = kvr.Cache(S, L, H, G, d, cap, "bf16", "bf16", device=dev)
        for s in range(S):
            k = (torch.randn(L, H, rows, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
            v = (torch.randn(L, H, rows, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
            cache.load(s, k, v)
            del k, v
        return cache

    def timed(fn):
        for i in range(Wm):
            fn()
        torch.cuda.synchronize()
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        t0.record(stream)
        for i in range(K):
            fn()
        t1.record(stream)
        torch.cuda.synchronize()
        return t0.elapsed_time(t1) * 1e3 / K  # us per call

    q, kn, vn = inputs_for(S)
    out = torch.empty(S, L, H * G, d, dtype=torch.bfloat16, device=dev)
    full = []
    drift = Wm + (K + 1) // 2  # each call appends a row: centre the mean
    for target in (72, 128, 256, 512, 640, 1024, 2048, 4096, 8192, 16384):
        ell = target - drift
        cache = loaded(ell, ell + Wm + K + 1)
        need = kvr.kvr_decode_attend_workspace_bytes(cache.handle, 0, L, 0)
        ws = torch.empty(max(need, 16), dtype=torch.uint8, device=dev)
        t = timed(lambda: kvr.kvr_decode_attend(cache.handle, 0, L, q, kn, vn,
                                                out, 0, ws, ws.numel(), stream))
        cache.sync_status()
        # mean rows attended over the timed calls
        full.append((ell + Wm + (K + 1) / 2.0, t))
        del cache, ws
    # Two evictors at each B' = B + W: the accumulated-attention step (one
    # fused kvr_decode_step) and the paper's R-KV eviction (App. C, lambda
    # 0.1, kvr_decode_step_rkv with its key-similarity pass: one launch at
    # B' = 72, attend+score then kvr_evict_compact_rkv at B' = 640), both
    # from a cache already at B + W rows.
    evict, evict_rkv = {}, {}
    for B, Wn in ((64, 8), (512, 128)):
        cache = loaded(B + Wn, B + Wn + 1)
        t = timed(lambda: kvr.kvr_decode_step(cache.handle, 0, L, q, kn, vn, out,
                                              B, Wn, stream))
        cache.sync_status()
        evict[B + Wn] = t
        del cache
        cache = loaded(B + Wn, B + Wn + 1)

        def rkv_step():
            kvr.kvr_decode_step_rkv(cache.handle, 0, L, q, kn, vn, out, B, Wn,
                                    0.1, stream)
        evict_rkv[B + Wn] = timed(rkv_step)
        cache.sync_status()
        del cache
    ls = np.array([x for x, _ in full])
    ts = np.array([y for _, y in full])
    fit = ls >= 512  # the bandwidth-bound part of the curve
    b, a = np.polyfit(ls[fit], ts[fit], 1)

    def crossover(ev):
        res = {}
        for bp, te in ev.items():
            t_bp = float(np.interp(bp, ls, ts))
            # first context at which full attention costs as much as the step
            above = np.nonzero(ts >= te)[0]
            if len(above) and above[0] > 0:
                i = above[0]
                lstar = float(ls[i - 1] + (te - ts[i - 1]) *
                              (ls[i] - ls[i - 1]) / (ts[i] - ts[i - 1]))
            elif len(above):
                lstar = float(ls[0])
            else:
                lstar = float((te - a) / b)
            res[bp] = {"t_evict_us": te, "t_full_at_Bphys_us": t_bp,
                       "alpha": te / t_bp - 1.0, "lstar_rows": lstar,
                       "lstar_over_Bphys": lstar / bp}
        return res
    return dict(full=[{"context": float(x), "us_per_step": float(y)} for x, y in full],
                fit={"a_us": float(a), "b_us_per_row": float(b)},
                res=crossover(evict), res_rkv=crossover(evict_rkv), S=S, K=K)


def run_absorb(args):
    """An accepted 64-token step absorbed by the evicted 7B base model in one
    call (kvr_absorb_chunk): 64 sequences x 28 layers, each unit at B+W = 72
    rows takes 64 new rows with causal attention and accumulated scores, then
    is cut back to 72.  One timed step = one call."""
    import torch
    from paper_2608_15797_gb300 import kvr
    w = inputs.WORKLOADS["7b_b64"]
    S = args.seqs or 64
    L, H, G, d, B, Wn, C = w.n_layers, w.n_kv_heads, w.group, w.head_dim, w.budget, w.window, 64
    dev = torch.device("cuda", 0)
    cache = kvr.Cache(S, L, H, G, d, B + Wn + C, "bf16", "bf16", device=dev)
    cache.set_absorb_kernel(args.absorb_kernel)
    gen = torch.Generator(device=dev)
    gen.manual_seed(args.seed + 37)
    for s in range(S):
        k = (torch.randn(L, H, B + Wn, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
        v = (torch.randn(L, H, B + Wn, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
        cache.load(s, k, v)
    pool = []
    for _ in range(4):
        q = (torch.randn(S, L, C, H * G, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
        kn = (torch.randn(S, L, C, H, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
        vn = (torch.randn(S, L, C, H, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
        pool.append((q, kn, vn))
    out = torch.empty(S, L, C, H * G, d, dtype=torch.bfloat16, device=dev)
    stream = torch.cuda.current_stream(dev)

    def step(i):
        q, kn, vn = pool[i % 4]
        kvr.kvr_absorb_chunk(cache.handle, 0, L, C, q, kn, vn, out, B, Wn, True,
                             stream)

    K, Wm = args.steps, max(3, args.warmup)
    for i in range(Wm):
        step(i)
    torch.cuda.synchronize()
    n0 = cache.launch_count()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for i in range(K):
        step(i)
    t1.record(stream)
    torch.cuda.synchronize()
    total = t0.elapsed_time(t1)
    launches = cache.launch_count() - n0
    cache.sync_status()
    ran = cache.last_absorb_kernel()
    units = S * L * H
    m = B + Wn
    # bytes: old K/V rows read, new k/v read, kept new rows written (at most
    # B + W of them, bounded by the chunk), q read, out written, scores and
    # positions read and written, state
    per_unit = (2 * m * d * 2 + 2 * C * d * 2 + 2 * min(C, m) * d * 2 +
                2 * C * G * d * 2 + 8 * m + 8 * m + 16)
    # flops over the causal triangle's mean width m + C/2: the mma.sync
    # kernel runs QK^T twice and PV with hi + lo terms; the tcgen05 kernel
    # runs QK^T once and PV with hi + lo (its column sums run on the CUDA
    # cores)
    if ran == 0:
        flops = C * G * (m + C / 2.0) * d * 2 * (1 + 2)
    else:
        flops = C * G * (m + C / 2.0) * d * 2 * (2 + 2)
    kernel = {0: "absorb_tc_kernel (tcgen05)", 1: "absorb_kernel (mma.sync)",
              2: "attend_score_kernel token by token"}.get(ran, "none")
    return dict(total_ms=total, per_ms=total / max(1, launches), K=K,
                launches=launches, launch_bytes=per_unit * units,
                launch_flops=flops * units, S=S, C=C, ran=ran, kernel=kernel)


def run_entropy(args):
    """The detector's entropy test on the candidates' next-token logits:
    64 problems x 8 candidates = 512 rows of 152,064 logits (Qwen2.5-Math's
    output width) per generated token, one kvr_entropy_step launch.  Rows
    have spreads in [3.6, 5.0] (entropy about 2.5-6.5 nats, below tau), so
    no row stops and every launch reads every row.  Three logit buffers
    rotate (each larger than L2)."""
    import torch
    from paper_2608_15797_gb300 import kvr
    rows, V = 512, inputs.VOCAB
    dt = args.entropy_dtype
    tdt = torch.bfloat16 if dt == "bf16" else torch.float32
    dev = torch.device("cuda", 0)
    det = kvr.EntropyDetector(rows, V, logits_dtype=dt, device=dev)
    det.set_kernel(args.entropy_kernel)
    gen = torch.Generator(device=dev)
    gen.manual_seed(args.seed + 41)
    sig = torch.linspace(3.6, 5.0, rows, device=dev).unsqueeze(1)
    bufs = [(torch.randn(rows, V, generator=gen, device=dev) * sig).to(tdt)
            for _ in range(3)]
    H = torch.empty(rows, dtype=torch.float32, device=dev)
    M = torch.empty_like(H)
    St = torch.empty(rows, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream(dev)

    def step(i, x=None):
        det.step(bufs[i % 3] if x is None else x, H, M, St, stream)

    K, Wm = args.steps, max(3, args.warmup)
    for i in range(Wm):
        step(i)
    torch.cuda.synchronize()
    n0 = det.launch_count()
    clocks = ClockSampler(0)
    clocks.start()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    tb = clocks.mark()
    t0.record(stream)
    for i in range(K):
        step(i)
    t1.record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop(tb, clocks.mark())
    total = t0.elapsed_time(t1)
    launches = det.launch_count() - n0
    det.sync_status()
    stopped = int((St != 0).sum().item())
    # end to end: logits from pinned host memory, stop flags back, per token
    host = [b.cpu().pin_memory() for b in bufs[:2]]
    flags = torch.empty(rows, dtype=torch.int32).pin_memory()
    xd = torch.empty_like(bufs[0])
    Ke = max(3, args.e2e_steps // 50)
    step(0, bufs[0])
    torch.cuda.synchronize()
    t0.record(stream)
    for i in range(Ke):
        xd.copy_(host[i % 2], non_blocking=True)
        step(i, xd)
        flags.copy_(St, non_blocking=True)
    t1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = t0.elapsed_time(t1)
    esz = 2 if dt == "bf16" else 4
    per_launch = rows * V * esz + rows * (4 * 12 + 16)
    return dict(total_ms=total, per_ms=total / max(1, launches), K=K,
                launches=launches, launch_bytes=per_launch, rows=rows, V=V,
                dtype=dt, stopped=stopped, clocks=clk, Ke=Ke, e2e_ms=e2e_ms,
                bi=rows * V * esz, bo=rows * 4)


def entropy_cpu_baseline(seconds):
    """The fp64 oracle's token_entropy on bounded samples of the same rows
    (8 rows of 152,064 logits per call), scaled to tokens/s."""
    import time
    from oracle import entropy as ent
    x = inputs.candidate_logits(0, 0, 8, inputs.VOCAB, 4.0)
    n, t0 = 0, time.perf_counter()
    while time.perf_counter() - t0 < seconds:
        ent.token_entropy(x)
        n += 8
    spent = time.perf_counter() - t0
    return n / spent, n, spent


def run_fork(args):
    """72B geometry (80 layers, 64 q / 8 kv heads, d 128), B=64, W=8: an
    evicted parent (B+W rows) forked to 8 candidates; one timed step is one
    candidate token for all 8 candidates, all layers, all sequences; the 64
    tokens of a reasoning step are followed by a commit (timed apart)."""
    import torch
    from paper_2608_15797_gb300 import kvr
    w = inputs.WORKLOADS["72b_bon8"]
    S = args.seqs or 4
    L, H, G, d, N = w.n_layers, w.n_kv_heads, w.group, w.head_dim, w.n_cand
    B, Wn, T = w.budget, w.window, w.cand_step
    dev = torch.device("cuda", 0)
    cache = kvr.Cache(S, L, H, G, d, B + Wn + T + 1, "bf16", "bf16", device=dev)
    if args.chunk_groups or args.chunk_stages:
        kvr.kvr_cache_set_chunk_tuning(cache.handle, args.chunk_groups,
                                       args.chunk_stages)
    gen = torch.Generator(device=dev)
    gen.manual_seed(args.seed + 29)
    for s in range(S):
        k = (torch.randn(L, H, B + Wn, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
        v = (torch.randn(L, H, B + Wn, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
        cache.load(s, k, v)
    q = (torch.randn(N, S, L, H * G, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
    kn = (torch.randn(N, S, L, H, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
    vn = (torch.randn(N, S, L, H, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
    out = torch.empty(N, S, L, H * G, d, dtype=torch.bfloat16, device=dev)
    stream = torch.cuda.current_stream(dev)
    chosen = np.zeros(S, np.int32)
    K = max(1, min(args.steps, 64 * 50))
    tok_ms, commit_ms, bytes_tok, launches = [], [], 0.0, 0
    n0 = cache.launch_count()
    done = 0
    warm = True
    while done < K:
        f = kvr.Fork(cache, N, T, kernel=args.fork_kernel)
        steps_here = T
        def step(i):
            kvr.kvr_fork_decode_attend_score(f.handle, 0, L, q, kn, vn, out, stream)
        tot, per = _timed(step, steps_here, stream)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        f.commit(chosen, B, Wn)
        e1.record(stream)
        torch.cuda.synchronize()
        if warm:
            warm = False
            n0 = cache.launch_count()
            continue
        tok_ms.append(per)
        commit_ms.append(e0.elapsed_time(e1))
        done += steps_here
    cache.sync_status()
    launches = cache.launch_count() - n0
    # algorithmic bytes of one candidate token (mean tail length T/2)
    np_rows, nt = B + Wn, (T - 1) / 2.0
    per_unit = (2 * np_rows * d * 2 + N * (2 * nt * d * 2 + 4 * d * 2 + 2 * G * d * 2
                                          + 8 * np_rows + 8 * (nt + 1) + 4))
    return dict(metric=f"72B best-of-{N} candidate tokens/s (B={B}, W={Wn}, "
                       f"{S} sequences x {L} layers x {N} candidates per token)",
                total_ms=float(np.mean(tok_ms)) * done, per_ms=float(np.mean(tok_ms)),
                K=done, launches=launches, launch_bytes=per_unit * S * L * H,
                commit_ms=float(np.mean(commit_ms)),
                config={"workload": "72b_bon8", "n_seq": S, "layers": L,
                        "kv_heads": H, "group": G, "head_dim": d, "n_cand": N,
                        "budget": B, "window": Wn, "cand_step": T},
                kernel="kvr_fork_decode_attend_score")


def run_rkv(args):
    """The evicted 7B step with the paper's R-KV eviction (App. C, lambda =
    0.1, in the library's reading): 64 sequences x 28 layers at B+W = 72
    rows; one timed step is kvr_decode_attend_score (append, attend,
    accumulate) and kvr_evict_compact_rkv (redundancy-aware TopB) over all
    layers, two launches.  The accumulated-attention step (one fused
    kvr_decode_step) is timed on the same state for comparison."""
    import torch
    from paper_2608_15797_gb300 import kvr
    w = inputs.WORKLOADS["7b_b64"]
    S = args.seqs or 64
    L, H, G, d, B, Wn = (w.n_layers, w.n_kv_heads, w.group, w.head_dim,
                         w.budget, w.window)
    lam = 0.1
    dev = torch.device("cuda", 0)
    cache = kvr.Cache(S, L, H, G, d, B + Wn + 1, "bf16", "bf16", device=dev)
    gen = torch.Generator(device=dev)
    gen.manual_seed(args.seed + 43)
    for s in range(S):
        k = (torch.randn(L, H, B + Wn, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
        v = (torch.randn(L, H, B + Wn, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
        cache.load(s, k, v)
    pool = []
    for _ in range(8):
        q = (torch.randn(S, L, H * G, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
        kn = (torch.randn(S, L, H, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
        vn = (torch.randn(S, L, H, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
        pool.append((q, kn, vn))
    out = torch.empty(S, L, H * G, d, dtype=torch.bfloat16, device=dev)
    stream = torch.cuda.current_stream(dev)

    def rkv_step(i):
        q, kn, vn = pool[i % 8]
        kvr.kvr_decode_step_rkv(cache.handle, 0, L, q, kn, vn, out, B, Wn,
                                lam, stream)

    def rkv_two_launches(i):
        q, kn, vn = pool[i % 8]
        kvr.kvr_decode_attend_score(cache.handle, 0, L, q, kn, vn, out, stream)
        kvr.kvr_evict_compact_rkv(cache.handle, 0, L, B, Wn, lam, stream)

    def score_step(i):
        q, kn, vn = pool[i % 8]
        kvr.kvr_decode_step(cache.handle, 0, L, q, kn, vn, out, B, Wn, stream)

    def timed(fn, K):
        for i in range(max(3, args.warmup)):
            fn(i)
        torch.cuda.synchronize()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for i in range(K):
            fn(i)
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1)

    K = args.steps
    n0 = cache.launch_count()
    rkv_ms = timed(rkv_step, K)
    launches = cache.launch_count() - n0 - max(3, args.warmup)
    score_ms = timed(score_step, K)
    two_ms = timed(rkv_two_launches, K)
    cache.sync_status()
    # One pass: the step's bytes (the key-similarity pass reads the keys
    # already staged for attention).
    attend = cost_model.step_unit_bytes(B + Wn, d, G, 2, 2, B, Wn)
    units = S * L * H
    return dict(total_ms=rkv_ms, per_ms=rkv_ms / K, K=K, launches=launches,
                launch_bytes=attend * units, profile="decode_step_rkv_7b_s64_b64",
                score_ms=score_ms / K, two_launch_ms=two_ms / K,
                metric=f"evicted decode steps/s with R-KV eviction at 7B "
                       f"geometry, B={B}, W={Wn}, lambda={lam} ({S} sequences"
                       f" x {L} layers per step)",
                config={"workload": "7b_s64_b64 R-KV", "n_seq": S, "layers": L,
                        "kv_heads": H, "group": G, "head_dim": d, "budget": B,
                        "window": Wn, "lambda": lam},
                kernel="kvr_decode_step_rkv (one launch: attention, scores "
                       "and the R-KV key-similarity pass over the staged "
                       "keys, selection, compaction)")


def run_fork_copy(args):
    """The paper's own candidate mode at 72B geometry (App. C): each
    reasoning step copies the evicted parent (B+W rows) into 8 candidate
    sequences, every candidate token is a kvr_decode_step over all of them
    with eviction back to B+W (64 tokens a step), and the chosen candidate is
    copied back.  One timed step is one candidate token for all 8 candidates,
    all layers, all sequences; the fork and commit copies are timed apart."""
    import torch
    from paper_2608_15797_gb300 import kvr
    w = inputs.WORKLOADS["72b_bon8"]
    S = args.seqs or 4
    L, H, G, d, N = w.n_layers, w.n_kv_heads, w.group, w.head_dim, w.n_cand
    B, Wn, T = w.budget, w.window, w.cand_step
    dev = torch.device("cuda", 0)
    cap = B + Wn + 1
    parent = kvr.Cache(S, L, H, G, d, cap, "bf16", "bf16", device=dev)
    kids = kvr.Cache(S * N, L, H, G, d, cap, "bf16", "bf16", device=dev)
    gen = torch.Generator(device=dev)
    gen.manual_seed(args.seed + 29)
    for s in range(S):
        k = (torch.randn(L, H, B + Wn, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
        v = (torch.randn(L, H, B + Wn, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
        parent.load(s, k, v)
    q = (torch.randn(S * N, L, H * G, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
    kn = (torch.randn(S * N, L, H, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
    vn = (torch.randn(S * N, L, H, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
    out = torch.empty(S * N, L, H * G, d, dtype=torch.bfloat16, device=dev)
    stream = torch.cuda.current_stream(dev)
    src = np.repeat(np.arange(S), N).astype(np.int32)
    dst = np.arange(S * N, dtype=np.int32)
    chosen = (np.arange(S) * N).astype(np.int32)
    K = max(1, min(args.steps, T * 50))
    tok_ms, fork_ms, commit_ms = [], [], []
    n0 = parent.launch_count() + kids.launch_count()
    done, warm = 0, True

    def copy_timed(fn):
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        fn()
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1)

    while done < K:
        fms = copy_timed(lambda: kids.copy_from(parent, src, dst, stream))

        def step(i):
            kvr.kvr_decode_step(kids.handle, 0, L, q, kn, vn, out, B, Wn,
                                stream)
        tot, per = _timed(step, T, stream)
        cms = copy_timed(lambda: parent.copy_from(kids, chosen, np.arange(
            S, dtype=np.int32), stream))
        if warm:
            warm = False
            n0 = parent.launch_count() + kids.launch_count()
            continue
        tok_ms.append(per)
        fork_ms.append(fms)
        commit_ms.append(cms)
        done += T
    parent.sync_status()
    kids.sync_status()
    launches = parent.launch_count() + kids.launch_count() - n0
    per_unit = cost_model.step_unit_bytes(B + Wn, d, G, 2, 2, B, Wn)
    copy_unit = 2 * (2 * (B + Wn) * d * 2 + 8 * (B + Wn) + 16)
    tms = float(np.mean(tok_ms))
    return dict(metric=f"72B best-of-{N} candidate tokens/s with eviction every "
                       f"token (B={B}, W={Wn}, {S} sequences x {L} layers x {N} "
                       f"candidates per token, candidates by copy)",
                total_ms=tms * done, per_ms=tms, K=done, launches=launches,
                launch_bytes=per_unit * S * N * L * H,
                fork_ms=float(np.mean(fork_ms)),
                commit_ms=float(np.mean(commit_ms)),
                fork_bytes=copy_unit * S * N * L * H,
                amortized_steps_per_s=T / ((tms * T + float(np.mean(fork_ms))
                                            + float(np.mean(commit_ms))) / 1e3),
                config={"workload": "72b_bon8", "n_seq": S, "layers": L,
                        "kv_heads": H, "group": G, "head_dim": d, "n_cand": N,
                        "budget": B, "window": Wn, "cand_step": T,
                        "candidates": "copies, eviction every token"},
                kernel="kvr_decode_step over the candidate sequences")


def run_sweep_row(args, B):
    """The throughput sweep at budget B (7B geometry, 64 sequences, W=8):
    the same measurement as the headline's value (one kvr_decode_step over
    all 28 layers a step, median of `repeats` K-step regions), without the
    end-to-end and per-layer legs."""
    import torch
    from paper_2608_15797_gb300 import kvr
    w = inputs.WORKLOADS[f"7b_s64_b{B}"]
    S, L, H, G, d, W = (w.n_seq, w.n_layers, w.n_kv_heads, w.group,
                        w.head_dim, w.window)
    dev = torch.device("cuda", 0)
    lo = max(args.prior_min, B + W + 1)
    lens = inputs.prior_lengths(args.seed + B, S, lo, max(lo, args.prior_max))
    cache = kvr.Cache(S, L, H, G, d, int(lens.max()) + 1, "bf16", "bf16",
                      device=dev)
    gen = torch.Generator(device=dev)
    gen.manual_seed(args.seed + 3 * B)
    for s in range(S):
        n = int(lens[s])
        k = (torch.randn(L, H, n, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
        v = (torch.randn(L, H, n, d, generator=gen, device=dev) * w.sigma).to(torch.bfloat16)
        cache.load(s, k, v)
        del k, v
    pool = [tuple((torch.randn(*shp, generator=gen, device=dev) * w.sigma)
                  .to(torch.bfloat16) for shp in ((S, L, H * G, d),
                                                  (S, L, H, d), (S, L, H, d)))
            for _ in range(8)]
    out = torch.empty(S, L, H * G, d, dtype=torch.bfloat16, device=dev)
    stream = torch.cuda.current_stream(dev)

    def step(i):
        kvr.kvr_decode_step(cache.handle, 0, L, *pool[i % 8], out, B, W,
                            stream)

    step(0)  # the first step evicts every unit to B + W
    torch.cuda.synchronize()
    assert (cache.lengths() == B + W).all()
    steady = kvr.Cache(S, L, H, G, d, B + W + 1, "bf16", "bf16", device=dev)
    steady.copy_from(cache, np.arange(S, dtype=np.int32),
                     np.arange(S, dtype=np.int32), stream)
    torch.cuda.synchronize()
    del cache
    torch.cuda.empty_cache()
    cache = steady
    # Warm up on the row's own steps for at least 50 ms of wall time: the
    # first tens of milliseconds after the set-up (a 60 GB prompt cache, a
    # first eviction over 16k-row units) run measurably slower.
    w0, i = time.time(), 0
    while i < max(3, args.warmup) or time.time() - w0 < 0.05:
        step(i)
        i += 1
        if i % 16 == 0:
            torch.cuda.synchronize()
    K = args.steps
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    regions, launches = [], 0
    for rep in range(max(1, args.repeats)):
        torch.cuda.synchronize()
        n0 = cache.launch_count()
        t0.record(stream)
        for i in range(K):
            step(rep * K + i)
        t1.record(stream)
        torch.cuda.synchronize()
        launches = cache.launch_count() - n0
        regions.append(t0.elapsed_time(t1))
    cache.sync_status()
    total = float(np.median(regions))
    unit_bytes = cost_model.step_unit_bytes(B + W, d, G, 2, 2, B, W)
    return dict(metric=metric_name(w), total_ms=total, per_ms=total / K, K=K,
                launches=launches, launch_bytes=unit_bytes * S * L * H,
                regions=regions, profile=f"decode_step_7b_s64_b{B}",
                config={"workload": f"7b_s64_b{B}", "budget": B, "window": W,
                        "prior_len": f"U[{lo},{max(lo, args.prior_max)}]",
                        "steady_capacity": B + W + 1},
                kernel="kvr_decode_step (one launch a step: the fused kernel "
                       "up to 160 rows a unit, the chunked one above)")


def row_record(r, unit, peak, peak_kind, value=None):
    """A compact sub-record of the default line for one row's result."""
    achieved = r["launch_bytes"] / (r["per_ms"] / 1e3) / 1e9
    rec = {"metric": r["metric"],
           "value": value if value is not None else r["K"] / (r["total_ms"] / 1e3),
           "unit": unit, "steps": r["K"],
           "ms_per_step": r["total_ms"] / r["K"], "config": r.get("config"),
           "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak,
                        "unit": "GB/s", "frac": achieved / peak,
                        "peak_kind": peak_kind,
                        "traffic": committed_traffic(r["profile"])
                        if "profile" in r else None,
                        "algorithmic_bytes_per_launch": r["launch_bytes"],
                        "launch_ms": r["per_ms"], "kernel": r.get("kernel")},
           "gpu_launches": r["launches"]}
    if "regions" in r:
        rec["regions_ms"] = [round(x, 5) for x in r["regions"]]
    for key in ("commit_ms", "fork_ms", "score_ms", "amortized_steps_per_s",
                "two_launch_ms"):
        if key in r:
            rec[key] = r[key]
    return rec


def sub_records(args):
    """The other rows, each a few milliseconds of timed region at its
    benchmarked size: the B = 128/256/512 sweep, the 72B candidate step and
    its commit, the paper's candidates-by-copy mode, chunk absorb, the R-KV
    step, the entropy test and the full-context helper."""
    import copy
    import torch
    peaks, peak_kind = measured_peaks()
    peak = float(peaks["hbm_gbs"])
    a = copy.copy(args)
    a.warmup = max(3, min(args.warmup, 10))
    a.steps = max(8, min(args.steps, 64))
    a.repeats = max(1, min(args.repeats, 5))
    a.seqs = 0
    out = {}
    torch.cuda.empty_cache()

    def run(name, fn, unit, **kw):
        try:
            out[name] = row_record(fn(), unit, peak, peak_kind, **kw)
        except Exception as e:  # reported, never silent
            out[name] = {"error": f"{type(e).__name__}: {e}"}
        torch.cuda.synchronize()
        torch.cuda.empty_cache()

    sampler = ClockSampler(0)
    sampler.start()
    t_begin = time.time()
    for B in (128, 256, 512):
        run(f"sweep_b{B}", lambda B=B: run_sweep_row(a, B), "steps/s")
    run("candidates_72b_bon8", lambda: run_fork(a), "candidate tokens/s")
    run("candidates_by_copy_72b_bon8", lambda: run_fork_copy(a),
        "candidate tokens/s")
    a_abs = copy.copy(a)
    a_abs.absorb_kernel = 0
    r_abs = {}

    def absorb():
        r = run_absorb(a_abs)
        r.update(metric="absorbed 64-token steps/s (7B, B=64, W=8, 64 "
                        "sequences x 28 layers a call)",
                 kernel=f"kvr_absorb_chunk ({r['kernel']})",
                 config={"workload": "7b absorb", "chunk": r["C"]})
        if r["ran"] == 0:  # the profile's kernel
            r["profile"] = "absorb_7b_s64_c64"
        r_abs.update(r)
        return r
    run("absorb_7b_c64", absorb, "calls/s")
    run("rkv_7b_b64", lambda: run_rkv(a), "steps/s")

    def entropy():
        r = run_entropy(a)
        r.update(metric=f"candidate rows screened/s by the entropy test "
                        f"({r['rows']} rows x {r['V']} {r['dtype']} logits a "
                        f"launch)",
                 kernel="kvr_entropy_step (entropy_stream_kernel)",
                 config={"rows": r["rows"], "vocab": r["V"]},
                 profile=f"entropy_stream_{r['rows']}x{r['V']}_{r['dtype']}")
        return r
    run("entropy_512x152064", entropy, "launches/s")
    run("helper_1p5b_16k", lambda: run_helper(a), "steps/s")
    out["clocks"] = sampler.stop(t_begin, time.time())
    return out


def print_row_line(args, r):
    peaks, peak_kind = measured_peaks()
    peak = float(peaks["hbm_gbs"])
    achieved = r["launch_bytes"] / (r["per_ms"] / 1e3) / 1e9
    line = {"metric": r["metric"], "value": r["K"] / (r["total_ms"] / 1e3),
            "unit": "steps/s", "n_gpus": 1, "steps": r["K"],
            "warmup": args.warmup, "ms_per_step": r["total_ms"] / r["K"],
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16", "data": "synthetic", "config": r["config"],
            "hbm_gbs": achieved,
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak,
                         "unit": "GB/s", "frac": achieved / peak,
                         "peak_kind": peak_kind,
                         "traffic": committed_traffic(r["profile"])
                         if "profile" in r else None,
                         "algorithmic_bytes_per_launch": r["launch_bytes"],
                         "launch_ms": r["per_ms"], "kernel": r["kernel"]},
            "gpu_launches": r["launches"]}
    for key in ("commit_ms", "fork_ms", "amortized_steps_per_s", "score_ms",
                "two_launch_ms"):
        if key in r:
            line[key] = r[key]
    if "fork_bytes" in r:
        line["fork_copy_gbs"] = r["fork_bytes"] / (r["fork_ms"] / 1e3) / 1e9
    print(json.dumps(line))


def main():
    args = parse()
    w = inputs.WORKLOADS[args.workload]
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        if rank != 0:
            return 0
        K = max(1, args.steps)
        rate, spent, S = oracle_rate_batch(w, args.seed, K, args.warmup)
        sample = (f"{K} steps of all {w.n_seq} sequences (every layer and KV "
                  f"head) from the steady state, {spent:.1f} s timed"
                  if S == w.n_seq else
                  f"{K} steps of {S} of the {w.n_seq} sequences from the "
                  f"steady state ({spent:.1f} s timed), scaled x{w.n_seq / S:.1f}")
        line = {
            "impl": "reference", "metric": metric_name(w), "value": rate,
            "unit": "steps/s", "n_gpus": args.gpus, "steps": K,
            "warmup": args.warmup, "ms_per_step": 1e3 / rate,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f64", "data": "synthetic",
            "config": headline_config(args, w),
            "cpu_baseline": {"value": rate, "unit": "steps/s", "cores": 1,
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": rate, "unit": "steps/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0},
        }
        print(json.dumps(line))
        return 0

    import torch
    if args.mode == "crossover":
        if rank == 0:
            r = run_crossover(args)
            r640, r72 = r["res"][640], r["res"][72]
            print(json.dumps({
                "metric": "attention-side crossover context l* at B'=640 "
                          "(7B geometry, Eq. 14; lower: eviction pays sooner)",
                "value": r640["lstar_rows"], "unit": "rows", "n_gpus": 1,
                "steps": r["K"], "warmup": args.warmup,
                "higher_is_better": False, "scaling": "weak",
                "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
                "config": {"workload": "7b crossover", "n_seq": r["S"],
                           "layers": 28, "kv_heads": 4, "group": 7,
                           "head_dim": 128},
                "alpha_640": r640["alpha"], "crossover_72": r72,
                "crossover_640": r640,
                "rkv": {"evictor": "R-KV, lambda 0.1 (kvr_decode_step_rkv)",
                        "alpha_640": r["res_rkv"][640]["alpha"],
                        "crossover_640": r["res_rkv"][640],
                        "crossover_72": r["res_rkv"][72]},
                "full_context": r["full"],
                "fit": r["fit"],
                "paper": {"lstar_rows": 2500, "alpha": 2.9, "B_phys": 640,
                          "note": "the paper's measurement on its own "
                                  "system, end to end; context only"}}))
        return 0
    if args.mode == "absorb":
        if rank == 0:
            r = run_absorb(args)
            peaks, peak_kind = measured_peaks()
            sec = r["per_ms"] / 1e3
            gbs = r["launch_bytes"] / sec / 1e9
            tfs = r["launch_flops"] / sec / 1e12
            print(json.dumps({
                "metric": f"absorbed 64-token steps/s (7B geometry, B=64, W=8, "
                          f"{r['S']} sequences x 28 layers per call)",
                "value": r["K"] / (r["total_ms"] / 1e3), "unit": "calls/s",
                "n_gpus": 1, "steps": r["K"], "warmup": args.warmup,
                "ms_per_step": r["total_ms"] / r["K"], "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
                "data": "synthetic",
                "config": {"workload": "7b absorb", "n_seq": r["S"], "layers": 28,
                           "kv_heads": 4, "group": 7, "head_dim": 128,
                           "chunk": r["C"], "budget": 64, "window": 8},
                "tokens_per_s": r["K"] * r["S"] * r["C"] / (r["total_ms"] / 1e3),
                "roofline": {"bound": "hbm", "achieved": gbs,
                             "peak": float(peaks["hbm_gbs"]), "unit": "GB/s",
                             "frac": gbs / float(peaks["hbm_gbs"]),
                             "peak_kind": peak_kind,
                             "traffic": committed_traffic("absorb_7b_s64_c64")
                             if r["S"] == 64 and r["ran"] == 0 else None,
                             "algorithmic_bytes_per_launch": r["launch_bytes"],
                             "launch_ms": r["per_ms"],
                             "kernel": r["kernel"]},
                "tensor": {"achieved_tflops": tfs,
                           "peak_tflops": float(peaks.get("bf16_tflops", 0)),
                           "frac": tfs / float(peaks.get("bf16_tflops", 1)),
                           "note": "issued tensor flops over the causal "
                                   "width, lo terms of P included"},
                "gpu_launches": r["launches"]}))
        return 0
    if args.mode == "entropy":
        if rank == 0:
            r = run_entropy(args)
            peaks, peak_kind = measured_peaks()
            sec = r["per_ms"] / 1e3
            gbs = r["launch_bytes"] / sec / 1e9
            line = {
                "metric": "candidate tokens screened/s by the entropy test "
                          f"({r['rows']} candidate rows x {r['V']} "
                          f"{r['dtype']} logits per launch)",
                "value": r["K"] * r["rows"] / (r["total_ms"] / 1e3),
                "unit": "tokens/s", "n_gpus": 1, "steps": r["K"],
                "warmup": args.warmup, "ms_per_step": r["total_ms"] / r["K"],
                "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": "f32", "data": "synthetic",
                "config": {"workload": "entropy detector, 64 problems x 8 "
                                       "candidates", "rows": r["rows"],
                           "vocab": r["V"], "logits": r["dtype"],
                           "window": 12, "guard": 24, "tau": 7.0,
                           "l2": "3 rotating logit buffers, each larger "
                                 "than L2"},
                "rows_stopped": r["stopped"],
                "roofline": {"bound": "hbm", "achieved": gbs,
                             "peak": float(peaks["hbm_gbs"]), "unit": "GB/s",
                             "frac": gbs / float(peaks["hbm_gbs"]),
                             "peak_kind": peak_kind,
                             "traffic": committed_traffic(
                                 f"entropy_stream_{r['rows']}x{r['V']}_"
                                 f"{r['dtype']}")
                             if args.entropy_kernel in (0, 1) else None,
                             "algorithmic_bytes_per_launch": r["launch_bytes"],
                             "launch_ms": r["per_ms"],
                             "kernel": "entropy_stream_kernel"
                             if args.entropy_kernel in (0, 1)
                             else "entropy_kernel"},
                "e2e": {"value": r["Ke"] * r["rows"] / (r["e2e_ms"] / 1e3),
                        "unit": "tokens/s", "h2d_bytes_per_step": r["bi"],
                        "d2h_bytes_per_step": r["bo"]},
                "gpu_launches": r["launches"],
                "clocks": r["clocks"],
            }
            if not args.no_cpu_baseline:
                rate, n, spent = entropy_cpu_baseline(min(args.cpu_seconds,
                                                          10.0))
                line["cpu_baseline"] = {
                    "value": rate, "unit": "tokens/s", "cores": 1,
                    "kind": "oracle",
                    "sample": f"{n} rows of {inputs.VOCAB} logits through the "
                              f"fp64 oracle in {spent:.1f} s"}
            print(json.dumps(line))
        return 0
    if args.mode != "step":
        if rank == 0:
            r = (run_helper(args) if args.mode == "helper" else
                 run_fork_copy(args) if args.mode == "fork-copy" else
                 run_rkv(args) if args.mode == "rkv" else
                 run_fork(args))
            print_row_line(args, r)
        return 0
    if world > 1:
        torch.distributed.init_process_group("nccl")
    r = run_kvr(args, rank, world, local_rank)
    if rank != 0:
        if world > 1:
            torch.distributed.destroy_process_group()
        return 0

    peaks, peak_kind = measured_peaks()
    peak = float(peaks["hbm_gbs"])
    steps_per_s = job_rate(world, r["K"], r["total_ms"])
    achieved = r["launch_bytes"] / (r["per_launch_ms"] / 1e3) / 1e9
    lat = run_latency_s1(args, local_rank) if world == 1 else None
    cpu = None
    if world == 1 and not args.no_cpu_baseline:
        rate, n, spent = oracle_rate(w, args.seed, args.cpu_seconds)
        cpu = {"value": rate, "unit": "steps/s", "cores": 1, "kind": "oracle",
               "sample": f"{n} steady-state steps of 1 of the {w.n_seq} "
                         f"sequences ({spent:.1f} s of fp64 oracle), scaled "
                         f"x{w.n_seq}"}
        procs = os.cpu_count() or 1
        if procs > 1 and args.cpu_all_seconds > 0:
            rate_all, n_all = oracle_rate_all_cores(
                args.workload, args.seed, args.cpu_all_seconds, procs)
            cpu["all_cores"] = {
                "value": rate_all, "cores": procs,
                "sample": f"{procs} processes, one sequence each, "
                          f"{args.cpu_all_seconds:.0f} s each ({n_all} "
                          f"sequence-steps), summed and scaled to "
                          f"{w.n_seq} sequences"}
    line = {
        "metric": metric_name(w), "value": steps_per_s, "unit": "steps/s",
        "n_gpus": world, "steps": r["K"], "warmup": args.warmup,
        "ms_per_step": r["total_ms"] / r["K"], "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic",
        "config": headline_config(args, w),
        "hbm_gbs": achieved,
        "hbm_frac_of_8tbs": achieved / NOMINAL_HBM_GBS,
        "first_step_ms": r["first_ms"],
        "move_to_steady_cache_ms": r["move_ms"],
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak,
                     "unit": "GB/s", "frac": achieved / peak,
                     "peak_kind": peak_kind,
                     "traffic": committed_traffic(
                         f"decode_step_{args.workload}"),
                     "algorithmic_bytes_per_launch": r["launch_bytes"],
                     "launch_ms": r["per_launch_ms"],
                     "launch_timing": "timed region / launches in it",
                     "kernel": "kvr_decode_step (all layers, one call)"},
        "e2e": {"value": job_rate(world, r["Ke"], r["e2e_ms"]),
                "unit": "steps/s", "h2d_bytes_per_step": r["bi"],
                "d2h_bytes_per_step": r["bo"],
                "call": "kvr_decode_step_host (host q/k/v in, host output "
                        "out; the library copies)",
                "copies": "every step's q/k/v in and output out inside the "
                          "timed region; steps rotate over 6 streams with "
                          "their own staging buffers, so copies overlap the "
                          "neighbouring steps' decode"},
        "e2e_serial": {"value": job_rate(world, r["Ke"], r["e2e_serial_ms"]),
                       "unit": "steps/s",
                       "note": "kvr_decode_step_host on one stream: copy in, "
                               "decode, copy out"},
        "gpu_launches": r["launches"],
        "per_layer_launches": {
            "launches_per_step": w.n_layers,
            "ms_per_step": r["per_layer_ms"],
            "steps_per_s": 1e3 / r["per_layer_ms"], "steps": r["Kl"]},
        "latency_1seq": lat,
        "clocks": r["clocks"],
        "cpu_baseline": cpu,
        "timing": {"regions_ms": [round(x, 5) for x in r["regions"]],
                   "value_from": "median of the K-step regions",
                   "spread": (max(r["regions"]) - min(r["regions"])) /
                             float(np.median(r["regions"]))},
    }
    if world == 1 and not args.no_rows:
        line["rows"] = sub_records(args)
    print(json.dumps(line))
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
