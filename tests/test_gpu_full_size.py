"""Parity at the benchmarked sizes, in the launch configuration bench.py
times, on sampled sequences.

Sequences are independent, so an oracle that holds a few of them (the
first, one in the middle and the last, which land on CTAs at both ends of
the persistent grids' unit order) checks those units of the full-size
launch exactly as a full oracle would; the other sequences run alongside
with device-drawn inputs that no check reads.

- decode step (Eq. 1 + TopB eviction, Sec. 2.1): 7B geometry, 64 sequences x
  28 layers x 4 KV heads = 7,168 units a launch, B = 64, 128, 256 and 512,
  W = 8, bf16 in and out.  The first step evicts every unit from its prior
  context (B + W + 16 to B + W + 600 rows here: the bench's longer prior
  contexts change only that untimed first step); the sequences then move
  into a steady-state cache of capacity B + W + 1, as in bench.py, where
  the steady-state steps run the fused kernel on 73 and 137-row units
  (B = 64, 128) or the chunked kernel on 265 and 521-row units.
- R-KV step (App. C, lambda = 0.1): the same 64 x 28 x 4 units at B + W = 72
  rows, attend+score then the R-KV eviction, then the one-launch R-KV step
  (kvr_decode_step_rkv) that bench.py --mode rkv times.
- chunk absorb (Algorithm 1's single forward pass over an accepted step): 64
  sequences x 28 layers at B + W = 72 rows taking 64-token chunks, as
  bench.py --mode absorb.
- candidate step (Sec. 2.2 Eq. 2): 72B geometry, the bench's 4 sequences x
  80 layers x 8 KV heads with 8 candidates and a 64-row tail capacity, every
  sequence checked (the bench's full size), a few candidate tokens, then
  the commit.
"""
import numpy as np
import pytest
import torch

from paper_2608_15797_gb300 import inputs
from tests import harness
from tests.test_gpu_absorb import absorb_lockstep
from tests.test_gpu_rkv import rkv_lockstep

pytestmark = pytest.mark.gpu

SAMPLE = [0, 37, 63]


@pytest.fixture(autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    torch.cuda.set_device(0)


@pytest.mark.parametrize("B", [64, 128, 256, 512])
def test_decode_step_7b_s64_sampled(B):
    """The throughput sweep's launches: B = 64 and 128 run the fused kernel
    on 73 and 137-row units (five and nine row tiles), B = 256 / 512 the
    chunked kernel on 265 / 521-row units; either way 7,168 units a launch
    over persistent CTAs, so every CTA works through many units and reuses
    its ring stages."""
    w = inputs.WORKLOADS[f"7b_s64_b{B}"]
    S, m = w.n_seq, B + w.window
    lens = inputs.prior_lengths(61 + B, S, m + 16, m + 600)
    c, o = harness.make_pair(w, 61 + B, S, cap=int(lens.max()) + 1,
                             prompt_lens=lens, out_dtype="bf16", sample=SAMPLE)
    launches = c.launch_count()
    harness.lockstep(c, o, w, 61 + B, 1, w.budget, w.window, sample=SAMPLE)
    # the first step evicts hundreds of rows (attend+score, then eviction)
    assert c.launch_count() - launches == 2
    # As bench.py does: the sequences move into a steady-state cache of
    # capacity B + W + 1 (a dense slab) and the timed steps run there.
    d = harness.guarded_cache(S, w.n_layers, w.n_kv_heads, w.group,
                              w.head_dim, m + 1, kv_dtype=w.dtype,
                              out_dtype="bf16")
    d.copy_from(c, np.arange(S, dtype=np.int32), np.arange(S, dtype=np.int32))
    del c
    launches = d.launch_count()
    st = harness.lockstep(d, o, w, 61 + B, 6, w.budget, w.window, step0=1,
                          sample=SAMPLE)
    assert st.units == 6 * len(SAMPLE) * w.n_layers * w.n_kv_heads
    assert (d.lengths() == m).all()
    assert d.launch_count() - launches == 6   # one launch a steady step


def test_rkv_step_7b_s64_b64_sampled():
    w = inputs.WORKLOADS["7b_b64"]
    S, m = 64, w.budget + w.window
    c, o = harness.make_pair(w, 62, S, cap=m + 1, prompt_lens=[m] * S,
                             out_dtype="bf16", sample=SAMPLE)
    st = rkv_lockstep(c, o, w, 62, 3, w.budget, w.window, 0.1, sample=SAMPLE)
    n0 = c.launch_count()
    st2 = rkv_lockstep(c, o, w, 62, 3, w.budget, w.window, 0.1, step0=3,
                       sample=SAMPLE, fused=True)
    assert c.launch_count() - n0 == 3   # the one-launch step bench.py times
    assert st.units + st2.units == 6 * len(SAMPLE) * w.n_layers * w.n_kv_heads
    assert (c.lengths() == m).all()


def test_absorb_7b_s64_c64_sampled():
    w = inputs.WORKLOADS["7b_b64"]
    S, m, C = 64, w.budget + w.window, 64
    c, o = harness.make_pair(w, 63, S, cap=m + C, prompt_lens=[m] * S,
                             out_dtype="bf16", sample=SAMPLE)
    for k in range(2):
        absorb_lockstep(c, o, w, 63, C, w.budget, w.window,
                        step0=20_000 + 100 * k, sample=SAMPLE)
    assert (c.lengths() == m).all()


def test_candidate_step_72b_bon8_full():
    w = inputs.WORKLOADS["72b_bon8"]
    S, m = 4, w.budget + w.window
    c, o = harness.make_pair(w, 64, S, cap=m + w.cand_step + 1,
                             prompt_lens=[m] * S, out_dtype="bf16")
    o = o.resized(m + w.cand_step)
    o2, chosen, st = harness.fork_lockstep(c, o, w, 64, w.n_cand, 4, w.budget,
                                           w.window, tail_cap=w.cand_step)
    assert st.steps == 5  # the tokens, then the commit
    assert (c.lengths() == m).all()
