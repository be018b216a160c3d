"""Candidates (Sec. 2.2 Eq. 2, App. C best-of-(N+N)) against the oracle.

The oracle forks by physical copy (what the paper's engine does): each
candidate is a full copy of the parent that decodes its tokens without
eviction and is cut to B + W at commit.  The CUDA path shares the parent's
rows as a read-only prefix; both must agree on every candidate's outputs and
scores after every token, and on the committed parent.
"""
import numpy as np
import pytest
import torch

from oracle import parity
from paper_2608_15797_gb300 import inputs, kvr
from tests import harness

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    torch.cuda.set_device(0)


# The candidate kernels (kvr_fork_set_kernel): candidate-batched on
# 5th-generation tensor cores, candidate-batched on mma.sync (the default),
# chunked, one CTA per unit, generic.
PATHS = {"tc": 5, "batch": 1, "chunked": 2, "mma": 3, "generic": 4}


def _evicted_pair(w, seed, S, cap, prompt_lens, warm_steps):
    """Load prompts and run evicting steps so the parent sits at B + W rows."""
    c, o = harness.make_pair(w, seed, S, cap=cap, prompt_lens=prompt_lens)
    harness.lockstep(c, o, w, seed, warm_steps, w.budget, w.window)
    return c, o


@pytest.mark.parametrize("path", list(PATHS))
@pytest.mark.parametrize("n_cand", [1, 3, 8])
def test_small_fork_commit_then_continue(n_cand, path):
    """Tail lengths cross the 16-row tile and 32-row chunk boundaries (7
    tokens from a ragged parent, 37 for N = 8)."""
    w = inputs.Workload("f", 2, 2, 3, 128, "bf16", 12, 4, 30, 0, sigma=1.0)
    c, o = _evicted_pair(w, 21, 2, cap=60, prompt_lens=[30, 9], warm_steps=3)
    o2, chosen, st = harness.fork_lockstep(c, o, w, 21, n_cand,
                                           37 if n_cand == 8 else 7, w.budget,
                                           w.window, kernel=PATHS[path])
    assert (c.lengths() == np.minimum(o2.len.max(axis=2), 16)).all()
    # the committed parent keeps decoding in lock-step
    harness.lockstep(c, o2, w, 21, 4, w.budget, w.window, step0=100)


def test_fork_parent_is_read_only_while_alive():
    w = inputs.Workload("f", 1, 1, 2, 64, "f32", 4, 2, 8, 0, sigma=1.0)
    c, _ = harness.make_pair(w, 22, 1, cap=16)
    f = kvr.Fork(c, 2, 4)
    q, kn, vn = (harness.dev(a, "f32") for a in inputs.step_inputs(w, 22, 0, 1))
    with pytest.raises(kvr.KvrError) as e:
        c.step(q, kn, vn, 4, 2)
    assert e.value.status == kvr.KVR_ESTATE
    with pytest.raises(kvr.KvrError) as e:
        f.commit(np.array([2], np.int32), 4, 2)
    assert e.value.status == kvr.KVR_EINVAL
    f.commit(np.array([1], np.int32), 4, 2)
    with pytest.raises(kvr.KvrError) as e:
        f.commit(np.array([1], np.int32), 4, 2)
    assert e.value.status == kvr.KVR_ESTATE
    c.step(q, kn, vn, 4, 2)  # the parent is writable again


def test_fork_tail_capacity():
    w = inputs.Workload("f", 1, 1, 2, 128, "bf16", 4, 2, 8, 0, sigma=1.0)
    c, _ = harness.make_pair(w, 23, 1, cap=16)
    f = kvr.Fork(c, 2, 2)
    per = [inputs.step_inputs(w, 23, 0, 1, cand=k + 1) for k in range(2)]
    Q, K, V = (harness.dev(np.stack([p[i] for p in per]), "bf16") for i in range(3))
    f.attend_score(Q, K, V)
    f.attend_score(Q, K, V)
    with pytest.raises(kvr.KvrError) as e:
        f.attend_score(Q, K, V)
    assert e.value.status == kvr.KVR_ECAPACITY


def test_single_candidate_equals_plain_deferred_eviction():
    """With N = 1, fork + T tokens + commit equals the plain cache driven
    through the same T tokens with eviction held back, then one eviction."""
    w = inputs.Workload("f", 2, 2, 4, 128, "bf16", 10, 3, 40, 0, sigma=1.0)
    c1, o1 = _evicted_pair(w, 24, 2, cap=41, prompt_lens=[40, 22], warm_steps=2)
    c2, _ = _evicted_pair(w, 24, 2, cap=41, prompt_lens=[40, 22], warm_steps=2)
    T = 6
    f = kvr.Fork(c1, 1, T)
    for t in range(T):
        q, kn, vn = inputs.step_inputs(w, 24, 10_000 + t, 2, cand=1)
        f.attend_score(*(harness.dev(a[None], "bf16") for a in (q, kn, vn)))
        c2.attend_score(*(harness.dev(a, "bf16") for a in (q, kn, vn)))
    f.commit(np.zeros(2, np.int32), w.budget, w.window)
    c2.evict(w.budget, w.window)
    for s in range(2):
        a, b = c1.export(s, kv=False), c2.export(s, kv=False)
        assert (a["len"] == b["len"]).all()
        for l in range(2):
            for h in range(2):
                n = a["len"][l, h]
                ma = dict(zip(a["pos"][l, h, :n].tolist(), a["score"][l, h, :n].tolist()))
                mb = dict(zip(b["pos"][l, h, :n].tolist(), b["score"][l, h, :n].tolist()))
                assert ma.keys() == mb.keys()
                for p in ma:
                    assert abs(ma[p] - mb[p]) <= 1e-4 * max(abs(mb[p]), 1e-6)


@pytest.mark.parametrize("path", ["tc", "batch", "chunked", "mma"])
def test_7b_best_of_4(path):
    """7B geometry stepwise best-of-4: an evicted cache (prompt 512, B=128,
    W=8; heavy keys), forked to 4 candidates that decode a 16-token step
    sharing the prefix, then re-evicted and committed."""
    w = inputs.WORKLOADS["7b_bon4"]
    c, o = _evicted_pair(w, 25, 1, cap=w.prompt + 1, prompt_lens=[w.prompt],
                         warm_steps=2)
    o2, chosen, st = harness.fork_lockstep(c, o, w, 25, w.n_cand, 16, w.budget,
                                           w.window, kernel=PATHS[path])
    assert (c.lengths() == w.budget + w.window).all()


@pytest.mark.parametrize("path", ["tc", "batch", "chunked"])
def test_72b_best_of_8(path):
    """72B geometry (80 layers, 8 KV heads, G=8), B=64, N=8 candidates, an
    8-token step (reduced from 64 to keep the oracle fast)."""
    w = inputs.Workload("72b_small", 80, 8, 8, 128, "bf16", 64, 8, 200, 0,
                        sigma=1.0 / np.sqrt(128.0))
    c, o = _evicted_pair(w, 26, 1, cap=w.prompt + 1, prompt_lens=[w.prompt],
                         warm_steps=1)
    _, _, st = harness.fork_lockstep(c, o, w, 26, 8, 8, w.budget, w.window,
                                     kernel=PATHS[path])
    assert (c.lengths() == w.budget + w.window).all()
    assert st.kernels == [PATHS[path]] * 8


@pytest.mark.parametrize("path", ["tc", "batch", "chunked"])
def test_fork_empty_prefix_and_block_edges(path):
    """A parent with no live rows (an empty prefix) and one whose prefix is
    an exact multiple of the 32-row chunk, with 2 and 3 candidates (tail
    blocks of 64 and 32 rows per candidate), decoded so the tails cross 32
    and 64 rows, then committed."""
    w = inputs.Workload("fe", 1, 2, 2, 128, "bf16", 24, 8, 0, 0, sigma=1.0)
    for n_cand in (2, 3):
        c, o = harness.make_pair(w, 27, 2, cap=110, prompt_lens=[0, 32])
        harness.fork_lockstep(c, o, w, 27, n_cand, 70, w.budget, w.window,
                              kernel=PATHS[path])


def test_fork_prefix_longer_than_a_block():
    """A prefix of 200 rows (a full 128-row prefix block and a partial one in
    the candidate-batched kernel) with 4 candidates."""
    w = inputs.Workload("fl", 1, 1, 3, 128, "bf16", 1 << 20, 0, 0, 0, sigma=1.0)
    c, o = harness.make_pair(w, 28, 1, cap=240, prompt_lens=[200])
    harness.fork_lockstep(c, o, w, 28, 4, 12, w.budget, w.window,
                          kernel=PATHS["batch"])


@pytest.mark.parametrize("n_cand,G,lens,steps,out", [
    (8, 8, [72, 72], 64, "bf16"),   # the benchmarked shape: tails up to 64 rows
    (3, 3, [16, 5], 20, "f32"),     # ragged prefixes, G < 8 (padding rows)
    (1, 7, [128, 1], 17, "f32"),    # the longest prefix, and a 1-row one
    (5, 8, [0, 33], 5, "bf16"),     # an empty prefix
    (8, 1, [100, 64], 33, "f32"),   # G = 1
    (2, 5, [47, 80], 49, "bf16"),   # odd prefix and tail lengths
])
def test_tc_fork_shapes(n_cand, G, lens, steps, out):
    """The tensor-memory candidate kernel across candidate counts, group
    sizes, prefix lengths (0 to its 128-row limit; partial 16-row boxes) and
    tail lengths (partial and whole 16-row pieces, up to its 64-row limit),
    with both output types; every token must run on it."""
    w = inputs.Workload("ft", 2, 2, G, 128, "bf16", 12, 4, 0, 0, sigma=1.0)
    # the oracle's candidates are copies that keep every row until the commit
    c, o = harness.make_pair(w, 30, 2, cap=max(lens) + steps + 1,
                             prompt_lens=lens, out_dtype=out)
    _, _, st = harness.fork_lockstep(c, o, w, 30, n_cand, steps, w.budget,
                                     w.window, kernel=5)
    assert st.kernels == [5] * steps


def test_tc_fork_many_units_per_cta():
    """384 units (3 sequences x 16 layers x 8 KV heads) with ragged
    prefixes, so every persistent CTA takes several units through both of
    its unit slots and its ring and head buffers wrap many times."""
    w = inputs.Workload("ftm", 16, 8, 4, 128, "bf16", 12, 4, 0, 0, sigma=1.0)
    c, o = harness.make_pair(w, 31, 3, cap=128 + 18 + 1,
                             prompt_lens=[72, 30, 128], out_dtype="bf16")
    _, _, st = harness.fork_lockstep(c, o, w, 31, 4, 18, w.budget, w.window,
                                     kernel=5)
    assert st.kernels == [5] * 18


def test_tc_fork_falls_back_past_its_limits():
    """A prefix of 129 rows or a tail past 64 rows is outside the tensor-
    memory kernel: those steps run another kernel, with the same results."""
    w = inputs.Workload("ftl", 1, 2, 4, 128, "bf16", 12, 4, 0, 0, sigma=1.0)
    c, o = harness.make_pair(w, 32, 1, cap=133, prompt_lens=[129])
    _, _, st = harness.fork_lockstep(c, o, w, 32, 2, 3, w.budget, w.window,
                                     kernel=5)
    assert 5 not in st.kernels
    c, o = harness.make_pair(w, 33, 1, cap=108, prompt_lens=[40])
    _, _, st = harness.fork_lockstep(c, o, w, 33, 2, 67, w.budget, w.window,
                                     kernel=5)
    assert st.kernels[:65] == [5] * 65 and 5 not in st.kernels[65:]
