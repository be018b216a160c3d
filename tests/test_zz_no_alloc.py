"""kvr_decode_attend_score_noalloc against kvr_decode_attend_score.

The no-allocation entry point serves callers that cannot allocate device
memory for a call (a plug-in whose host program owns every allocation, a
service that fixes its footprint at start-up): it keeps its logit scratch in
a static device array inside the library.  It must give the same results as
the regular entry point, on consecutive calls (the shared array keeps the
previous call's contents), and reject calls larger than its array.

This file is collected last on purpose, so that a run stopping at the first
failure has already run every other test.
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


def _unit_rows(ex, l, h):
    n = ex["len"][l, h]
    return dict(zip(ex["pos"][l, h, :n].tolist(), ex["score"][l, h, :n].tolist()))


def test_noalloc_matches_regular_entry_point_on_two_calls():
    w = inputs.Workload("na", 2, 3, 7, 128, "bf16", 1 << 20, 0, 0, 2, sigma=1.0)
    lens = [300, 57]
    regular, _ = harness.make_pair(w, 31, 2, cap=310, prompt_lens=lens)
    noalloc, _ = harness.make_pair(w, 31, 2, cap=310, prompt_lens=lens)
    for t in range(2):  # two calls in a row through the shared array
        q, kn, vn = (harness.dev(a, "bf16") for a in inputs.step_inputs(w, 31, t, 2))
        ref = regular.attend_score(q, kn, vn)
        out = torch.full_like(ref, float("nan"))
        kvr.kvr_decode_attend_score_noalloc(noalloc.handle, 0, w.n_layers, q, kn,
                                            vn, out)
        torch.cuda.synchronize()
        parity.check_out(out.cpu().numpy(), ref.cpu().numpy(),
                         what=f"noalloc out, call {t}")
        for s in range(2):
            ea, eb = regular.export(s, kv=False), noalloc.export(s, kv=False)
            assert (ea["len"] == eb["len"]).all()
            for l in range(w.n_layers):
                for h in range(w.n_kv_heads):
                    a, b = _unit_rows(ea, l, h), _unit_rows(eb, l, h)
                    assert a.keys() == b.keys()
                    sa = np.array([a[p] for p in sorted(a)])
                    sb = np.array([b[p] for p in sorted(a)])
                    assert (np.abs(sb - sa) <= parity.SCORE_RTOL *
                            np.maximum(np.abs(sa), parity.SCORE_FLOOR)).all()
    noalloc.sync_status()
    regular.sync_status()


def test_noalloc_rejects_calls_beyond_its_array():
    # 8 KV heads x G=8 x 16385 rows x 4 B = 4.0001 MiB > the 4 MiB array
    w = inputs.Workload("big", 1, 8, 8, 128, "bf16", 1 << 20, 0, 0, 1, sigma=1.0)
    c, _ = harness.make_pair(w, 32, 1, cap=16385, prompt_lens=[16384])
    q, kn, vn = (harness.dev(a, "bf16") for a in inputs.step_inputs(w, 32, 0, 1))
    out = c.new_out(1)
    with pytest.raises(kvr.KvrError) as e:
        kvr.kvr_decode_attend_score_noalloc(c.handle, 0, 1, q, kn, vn, out)
    assert e.value.status == kvr.KVR_EINVAL
    assert "static scratch" in str(e.value)
    assert c.lengths().tolist() == [[16384]]  # nothing was enqueued
