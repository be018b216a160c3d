"""Candidates by copy with eviction every token (App. C best-of-(N+N), the
paper's own mode) against the oracle.

Forking copies the accepted sequence's live state into N candidate
sequences (kvr_cache_copy_sequences); the candidates then decode like any
sequence, each evicting to B + W after every token (kvr_decode_step), and
the chosen candidate is copied back as the persistent sequence.  The oracle
does the same with OracleCache.copy_sequences; every candidate's outputs,
scores and retained set are checked after every token.
"""
import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2608_15797_gb300 import inputs, kvr
from tests import harness

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    torch.cuda.set_device(0)


def _same_state(a, sa, b, sb, rows_only=False):
    """Sequence sa of cache a and sb of cache b hold the same live rows."""
    ea, eb = a.export(sa), b.export(sb)
    assert np.array_equal(ea["len"], eb["len"])
    assert np.array_equal(ea["next_pos"], eb["next_pos"])
    for l in range(a.L):
        for h in range(a.H):
            n = ea["len"][l, h]
            for key in ("pos", "score"):
                assert np.array_equal(ea[key][l, h, :n], eb[key][l, h, :n])
            for key in ("K", "V"):
                assert np.array_equal(ea[key][l, h, :n], eb[key][l, h, :n])


def _candidates(w, seed, S, N, cap, kid_cap, warm, cand_steps, commit_steps,
                fused=True, prompt_lens=None):
    c, o = harness.make_pair(w, seed, S, cap=cap, prompt_lens=prompt_lens)
    harness.lockstep(c, o, w, seed, warm, w.budget, w.window, fused=fused)
    kids = kvr.Cache(S * N, w.n_layers, w.n_kv_heads, w.group, w.head_dim,
                     kid_cap, kv_dtype=w.dtype, out_dtype="f32")
    kids.set_fused(fused)
    okids = orc.OracleCache(S * N, w.n_layers, w.n_kv_heads, w.group,
                            w.head_dim, kid_cap)
    src = np.repeat(np.arange(S), N)
    dst = np.arange(S * N)
    kids.copy_from(c, src, dst)
    okids.copy_sequences(o, src, dst)
    for i in range(S * N):
        _same_state(kids, i, c, src[i])
    st = harness.lockstep(kids, okids, w, seed + 1, cand_steps, w.budget,
                          w.window, fused=fused, step0=1000)
    pick = inputs.candidate_pick(seed, 0, S, N)
    chosen = np.arange(S) * N + pick
    c.copy_from(kids, chosen, np.arange(S))
    o.copy_sequences(okids, chosen, np.arange(S))
    for s in range(S):
        _same_state(c, s, kids, chosen[s])
    harness.lockstep(c, o, w, seed + 2, commit_steps, w.budget, w.window,
                     fused=fused, step0=2000)
    return st


@pytest.mark.parametrize("fused", [True, False])
def test_small_candidates_by_copy(fused):
    w = inputs.Workload("f", 2, 2, 3, 128, "bf16", 12, 4, 30, 0, sigma=1.0)
    _candidates(w, 31, 2, 3, cap=40, kid_cap=17, warm=3, cand_steps=9,
                commit_steps=3, fused=fused)


def test_7b_best_of_4_by_copy():
    """Config 3's shape: 7B, B = 128, W = 8, N = 4, with eviction every
    candidate token (the paper's mode), 24 candidate tokens."""
    w = inputs.WORKLOADS["7b_bon4"]
    st = _candidates(w, 32, 1, 4, cap=w.prompt + 1, kid_cap=w.budget + w.window + 1,
                     warm=2, cand_steps=24, commit_steps=2)
    assert st.units > 0


def test_72b_best_of_8_by_copy():
    """Config 4's shape: 72B, B = 64, W = 8, N = 8, eviction every token."""
    w = inputs.WORKLOADS["72b_bon8"]
    _candidates(w, 33, 1, 8, cap=151, kid_cap=w.budget + w.window + 1, warm=2,
                cand_steps=6, commit_steps=2, prompt_lens=[150])


def test_copy_within_one_cache_and_capacity():
    w = inputs.Workload("f", 1, 2, 2, 64, "f32", 6, 2, 10, 0, sigma=1.0)
    c, o = harness.make_pair(w, 34, 4, cap=12, prompt_lens=[10, 3, 0, 7])
    c.copy_from(c, [0, 1], [2, 3])
    o.copy_sequences(o, [0, 1], [2, 3])
    _same_state(c, 2, c, 0)
    _same_state(c, 3, c, 1)
    harness.lockstep(c, o, w, 34, 5, w.budget, w.window)
    # a smaller cache takes the rows once they fit
    small = kvr.Cache(2, 1, 2, 2, 64, 8, kv_dtype="f32", out_dtype="f32")
    small.copy_from(c, [0, 3], [1, 0])
    _same_state(small, 1, c, 0)
    _same_state(small, 0, c, 3)


def test_copy_errors():
    w = inputs.Workload("f", 1, 2, 2, 64, "f32", 6, 2, 10, 0, sigma=1.0)
    c, _ = harness.make_pair(w, 35, 3, cap=12)
    tiny = kvr.Cache(2, 1, 2, 2, 64, 4, kv_dtype="f32", out_dtype="f32")
    other = kvr.Cache(2, 1, 2, 2, 128, 12, kv_dtype="f32", out_dtype="f32")

    def expect(status, fn):
        with pytest.raises(kvr.KvrError) as e:
            fn()
        assert e.value.status == status

    expect(kvr.KVR_ECAPACITY, lambda: tiny.copy_from(c, [0], [0]))
    expect(kvr.KVR_EINVAL, lambda: other.copy_from(c, [0], [0]))
    expect(kvr.KVR_EINVAL, lambda: c.copy_from(c, [0, 1], [2, 2]))
    expect(kvr.KVR_EINVAL, lambda: c.copy_from(c, [0, 1], [1, 2]))
    expect(kvr.KVR_EINVAL, lambda: c.copy_from(c, [0], [3]))
    expect(kvr.KVR_EINVAL, lambda: c.copy_from(c, [-1], [2]))
    f = kvr.Fork(c, 2, 4)
    kids = kvr.Cache(2, 1, 2, 2, 64, 12, kv_dtype="f32", out_dtype="f32")
    expect(kvr.KVR_ESTATE, lambda: kids.copy_from(c, [0], [0]))
    del f
    kids.copy_from(c, [], [])
    c.sync_status()
