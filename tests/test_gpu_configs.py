"""The full-length runs of the workloads the parity target names, on the
default (fastest) kernels, in lock-step with the fp64 oracle:

- 7B decode geometry, prompt 512, 4096 decode steps, B=64, W=8 (every step
  checked: outputs, scores, retained sets);
- 7B stepwise best-of-4: prompt 512 (5% heavy keys), 2048 prior decode
  steps at B=128, W=8, then a 64-token candidate step shared by 4
  candidates, the re-eviction and commit, then more decoding;
- 72B decode geometry, prompt 1024, B=64, W=8: the first (evicting) step,
  then all 2048 decode tokens as 32 candidate steps of 8 candidates, each
  committed (the oracle in spawned worker processes).

The shorter cases of test_gpu_parity.py / test_gpu_fork.py cover the edges;
these cover the lengths (score drift over thousands of steps, tails that
fill their capacity).
"""
import numpy as np
import pytest
import torch

from oracle import parity
from paper_2608_15797_gb300 import inputs, kvr
from tests import harness, oracle_pool

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    torch.cuda.set_device(0)


def test_7b_4096_steps():
    w = inputs.WORKLOADS["7b_b64"]
    c, o = harness.make_pair(w, 40, 1, cap=w.prompt + 1)
    st = harness.lockstep(c, o, w, 40, w.steps, w.budget, w.window)
    assert st.steps == 4096
    assert (c.lengths() == w.budget + w.window).all()


def test_7b_best_of_4_after_2048_steps():
    w = inputs.WORKLOADS["7b_bon4"]
    c, o = harness.make_pair(w, 41, 1, cap=w.prompt + 1)
    harness.lockstep(c, o, w, 41, w.steps, w.budget, w.window)
    o = o.resized(w.budget + w.window + w.cand_step)
    o2, chosen, st = harness.fork_lockstep(c, o, w, 41, w.n_cand, w.cand_step,
                                           w.budget, w.window)
    assert st.steps == w.cand_step + 1  # the tokens, then the commit
    assert (c.lengths() == w.budget + w.window).all()
    harness.lockstep(c, o2.resized(w.budget + w.window + 1), w, 41, 16,
                     w.budget, w.window, step0=50_000)


def test_72b_best_of_8_full_length():
    """72B geometry, prompt 1024, B = 64, W = 8, N = 8: the prompt is cut to
    B + W by the first decode step, then all 2048 decode tokens run as 32
    candidate steps of 64 tokens, each forked from the committed parent
    (shared prefix), checked after every token (every candidate's outputs
    and the scores of all its rows), committed to a seeded pick and checked
    again.  The fp64 oracle runs in spawned worker processes, one per
    candidate and layer range (tests/oracle_pool.py)."""
    w = inputs.WORKLOADS["72b_bon8"]
    B, W, N, T = w.budget, w.window, w.n_cand, w.cand_step
    m = B + W
    n_steps = w.steps // T
    pool = oracle_pool.CandidateOraclePool(w, N, m, T, seed=42)
    try:
        c0, o = harness.make_pair(w, 42, 1, cap=w.prompt + 1)
        harness.lockstep(c0, o, w, 42, 1, B, W)
        # The compressed parent moves into a cache of the bench's capacity
        # (B + W + one candidate step + 1) through export / import.
        c = kvr.Cache(1, w.n_layers, w.n_kv_heads, w.group, w.head_dim,
                      m + T + 1, kv_dtype=w.dtype, out_dtype="f32")
        ex = c0.export(0)
        c.import_state(0, {x: (ex[x][:, :, :m + T + 1] if ex[x].ndim >= 3
                               else ex[x]) for x in ex})
        del c0
        pool.set_parent(o)
        a = pool.a
        total = parity.Stats()
        for j in range(n_steps):
            ex = c.export(0, kv=False)
            a["gpos"][...] = ex["pos"][..., :m]
            a["glen"][...] = ex["len"]
            f = kvr.Fork(c, N, T)
            pool.fork()
            for t in range(T):
                pool.token_inputs(10_000 + j * T + t)
                out = f.attend_score(*(harness.dev(a[x][:, None], w.dtype)
                                       for x in ("q", "kn", "vn")))
                a["out"][...] = out[:, 0].float().cpu().numpy()
                for k in range(N):
                    e = f.export(k, 0)
                    a["pscore"][k] = e["prefix_score"][..., :m]
                    a["tscore"][k] = e["tail_score"]
                    a["tpos"][k] = e["tail_pos"]
                    a["tlen"][k] = e["tail_len"]
                total.merge(pool.check(t))
            chosen = inputs.candidate_pick(42, j, 1, N)
            f.commit(chosen, B, W)
            del f
            ex = c.export(0, kv=False)
            a["gpos"][...] = ex["pos"][..., :m]
            a["gscore"][...] = ex["score"][..., :m]
            a["glen"][...] = ex["len"]
            st = pool.commit(chosen[0], B, W)
            assert st.units == w.n_layers * w.n_kv_heads
            total.merge(st)
        c.sync_status()
    finally:
        pool.close()
    assert total.steps == n_steps * (T + 1)
    assert (c.lengths() == m).all()
    print(f"72B best-of-8: {n_steps} candidate steps, {n_steps * T} tokens; "
          f"{total.adoptions} near-tie adoptions, max out excess "
          f"{total.max_out_excess:.3f}, max score rel "
          f"{total.max_score_rel:.2e}")
