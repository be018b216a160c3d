"""The multi-rank path of bench.py on CPU: two gloo ranks.

Sequences shard across ranks with no data-path collective (weak scaling);
the only collectives are the timing barrier and the max over ranks of the
timed region.  These tests run the same host logic bench.py runs under
torchrun, with the gloo backend: every rank gets its own seeds and prior
lengths, the max over ranks reaches every rank, and the whole-job rate is
the units of all ranks over the slowest rank's time.
"""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench
from oracle import oracle as orc
from paper_2608_15797_gb300 import inputs


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        len_seed, in_seed = bench.rank_seeds(3, rank)
        lens = inputs.prior_lengths(len_seed, 4, 20, 40)
        # a replica's own work: one oracle step over its own sequences
        w = inputs.WORKLOADS["tiny"]
        o = orc.OracleCache(2, w.n_layers, w.n_kv_heads, w.group, w.head_dim,
                            cap=64)
        for s in range(2):
            k, v = inputs.prompt(w, len_seed, s, int(lens[s]))
            o.load(s, k, v)
        out = o.step(*inputs.step_inputs(w, in_seed % (1 << 31), 0, 2),
                     B=w.budget, W=w.window)
        dist.barrier()
        slowest = bench.max_over_ranks(10.0 + 5.0 * rank)
        q.put((rank, slowest, (len_seed, in_seed), lens.tolist(),
               float(np.abs(out).sum())))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks():
    port = _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in range(2))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, m0, s0, l0, o0), (r1, m1, s1, l1, o1) = res
    assert (r0, r1) == (0, 1)
    assert m0 == m1 == 15.0                  # every rank sees the slowest
    assert s0 != s1 and l0 != l1 and o0 != o1  # each rank its own sequences
    assert s0 == bench.rank_seeds(3, 0)      # and deterministic
    assert l0 == inputs.prior_lengths(s0[0], 4, 20, 40).tolist()


def test_job_rate_and_single_process_max():
    assert bench.job_rate(2, 100, 50.0) == pytest.approx(4000.0)
    assert bench.job_rate(1, 100, 50.0) == pytest.approx(2000.0)
    assert bench.max_over_ranks(7.5) == 7.5  # no process group: itself
