"""Failure detection on the decode path, in forms that fault no GPU.

* A non-finite input (a NaN in q or in the appended key) leaves a softmax
  normaliser non-finite; every step kernel then sets the device error word
  and the next kvr_sync_status reports KVR_EDEVICE and clears the word.
* Every wait of the step kernels on an asynchronous copy is bounded.  A
  testing hook holds back the copies of one unit (nothing is issued, so
  nothing is left in flight) and the cache's wait limit is lowered to 1 ms:
  the launch must come back with the timeout bit set, without hanging.
* Either way the cache's state is then restored from a snapshot taken
  before the step (kvr_cache_export / kvr_cache_import, the resume path),
  and decoding continues in lock-step with the fp64 oracle.
* Every parity run's caller buffers sit between canary regions
  (tests/harness.py), checked after each run; a direct check here.
"""
import time

import numpy as np
import pytest
import torch

from paper_2608_15797_gb300 import inputs, kvr
from tests import harness

pytestmark = pytest.mark.gpu

W = 8
# kernel -> (budget B, use the one-launch kernels): the fused step takes
# units of at most 160 rows, the chunked one 161-1024, the streaming one
# 1025-2048; fused=False runs the generic pair.
KERNELS = {"fused": (64, True), "chunked": (200, True), "stream": (1100, True),
           "generic": (64, False)}


@pytest.fixture(autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    torch.cuda.set_device(0)


def _pair(kernel, seed):
    B, fused = KERNELS[kernel]
    w = inputs.Workload("fail", 2, 4, 7, 128, "bf16", B, W, B + W, 0,
                        sigma=1.0)
    c, o = harness.make_pair(w, seed, 2, cap=B + W + 2, fused=fused)
    harness.lockstep(c, o, w, seed, 2, B, W, fused=fused)
    return w, c, o


def _step(c, w, q, kn, vn, fused):
    qd, kd, vd = (harness.dev(a, w.dtype) for a in (q, kn, vn))
    if fused:
        c.step(qd, kd, vd, w.budget, W)
    else:
        c.attend_score(qd, kd, vd)
        c.evict(w.budget, W)


def _restore_and_continue(c, o, w, seed, snapshot, fused):
    for s, st in enumerate(snapshot):
        c.import_state(s, st)
    st = harness.lockstep(c, o, w, seed, 3, w.budget, W, fused=fused, step0=2)
    assert st.steps == 3


@pytest.mark.parametrize("kernel", list(KERNELS))
@pytest.mark.parametrize("where", ["q", "k_new"])
def test_nonfinite_input_sets_the_error_word(kernel, where):
    seed = 90 + list(KERNELS).index(kernel)
    w, c, o = _pair(kernel, seed)
    fused = KERNELS[kernel][1]
    snapshot = [c.export(s) for s in range(c.S)]
    q, kn, vn = inputs.step_inputs(w, seed, 2, c.S)
    if where == "q":
        q[1, 1, 5, 17] = np.nan        # one head of one unit
    else:
        kn[0, 0, 2, 3] = np.nan        # the new key of one unit
    _step(c, w, q, kn, vn, fused)
    with pytest.raises(kvr.KvrError) as e:
        c.sync_status()
    assert e.value.status == kvr.KVR_EDEVICE
    assert "non-finite" in str(e.value)
    c.sync_status()                    # the word was cleared
    _restore_and_continue(c, o, w, seed, snapshot, fused)


@pytest.mark.parametrize("kernel", ["fused", "chunked"])
def test_bounded_wait_runs_out_and_the_cache_recovers(kernel):
    seed = 95 + (kernel == "chunked")
    w, c, o = _pair(kernel, seed)
    snapshot = [c.export(s) for s in range(c.S)]
    launches = c.launch_count()
    c.set_wait_limit(1_000_000)        # 1 ms
    c.set_hold_first_unit(True)
    q, kn, vn = inputs.step_inputs(w, seed, 2, c.S)
    t0 = time.perf_counter()
    _step(c, w, q, kn, vn, True)
    with pytest.raises(kvr.KvrError) as e:
        c.sync_status()
    elapsed = time.perf_counter() - t0
    assert e.value.status == kvr.KVR_EDEVICE
    assert "timeout" in str(e.value)
    assert c.launch_count() == launches + 1   # one launch, and it returned
    assert elapsed < 1.5, elapsed     # the 1 ms bound, not the 2 s default
    c.set_hold_first_unit(False)
    c.set_wait_limit(0)
    c.sync_status()
    _restore_and_continue(c, o, w, seed, snapshot, True)


def test_wait_limit_arguments():
    w, c, o = _pair("fused", 97)
    with pytest.raises(kvr.KvrError) as e:
        c.set_wait_limit(3_000_000_000)
    assert e.value.status == kvr.KVR_EINVAL
    c.set_wait_limit(2_000_000_000)
    c.set_wait_limit(0)


def test_canaries_detect_a_write_past_the_buffer():
    """The guard check itself: a cache in a guarded buffer stays intact
    through steps, and a byte written just past the buffer is reported."""
    w, c, o = _pair("fused", 98)
    harness.check_guards(c)
    g = c._guards[0]
    g.raw[harness.GUARD + g.buf.numel()] = 0
    with pytest.raises(AssertionError, match="canary"):
        harness.check_guards(c)
