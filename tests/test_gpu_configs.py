"""The full-length runs of the workloads the parity target names, on the
default (fastest) kernels, in lock-step with the fp64 oracle:

- 7B decode geometry, prompt 512, 4096 decode steps, B=64, W=8 (every step
  checked: outputs, scores, retained sets);
- 7B stepwise best-of-4: prompt 512 (5% heavy keys), 2048 prior decode
  steps at B=128, W=8, then a 64-token candidate step shared by 4
  candidates, the re-eviction and commit, then more decoding;
- 72B decode geometry, prompt 1024, B=64, W=8: the first (evicting) step,
  then a 64-token candidate step of 8 candidates and its commit.

The shorter cases of test_gpu_parity.py / test_gpu_fork.py cover the edges;
these cover the lengths (score drift over thousands of steps, tails that
fill their capacity).
"""
import numpy as np
import pytest
import torch

from paper_2608_15797_gb300 import inputs
from tests import harness

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


def test_72b_best_of_8_prompt_1024():
    w = inputs.WORKLOADS["72b_bon8"]
    c, o = harness.make_pair(w, 42, 1, cap=w.prompt + 1)
    harness.lockstep(c, o, w, 42, 1, w.budget, w.window)
    o = o.resized(w.budget + w.window + w.cand_step)
    o2, chosen, st = harness.fork_lockstep(c, o, w, 42, w.n_cand, w.cand_step,
                                           w.budget, w.window)
    assert st.steps == w.cand_step + 1  # the tokens, then the commit
    assert (c.lengths() == w.budget + w.window).all()
