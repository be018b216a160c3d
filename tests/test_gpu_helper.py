"""Full-context decode (the helper's cache: no scores, no eviction) against
the oracle's attention over every row (Eq. 1 with B >= length)."""
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


def _run(w, seed, lens, cap, steps, n_splits, out_dtype="f32"):
    c, o = harness.make_pair(w, seed, len(lens), cap=cap, prompt_lens=lens,
                             out_dtype=out_dtype)
    for t in range(steps):
        q, kn, vn = inputs.step_inputs(w, seed, t, len(lens))
        out = kvr.attend_full(c, *(harness.dev(a, "bf16") for a in (q, kn, vn)),
                              n_splits=n_splits)
        ref = o.step(q, kn, vn, evict=False)
        torch.cuda.synchronize()
        parity.check_out(out.float().cpu().numpy(), ref, what=f"out at {t}")
        for s in range(len(lens)):
            ex = c.export(s)
            assert (ex["len"] == lens[s] + t + 1).all()
            assert (ex["next_pos"] == lens[s] + t + 1).all()
            n = lens[s] + t
            np.testing.assert_array_equal(ex["K"][:, :, n], kn[s])
            np.testing.assert_array_equal(ex["V"][:, :, n], vn[s])
            assert (ex["pos"][:, :, n] == n).all()
    c.sync_status()
    return c


@pytest.mark.parametrize("n_splits", [0, 1, 3, 7])
def test_ragged_lengths_and_splits(n_splits):
    """Ragged lengths (a single row, a partial 64-row stage, several stages),
    G = 6 as in the 1.5B helper, unscaled inputs."""
    w = inputs.Workload("h", 2, 2, 6, 128, "bf16", 1 << 20, 0, 0, 3, sigma=1.0)
    _run(w, 41, [0, 37, 640, 1000], cap=1010, steps=3, n_splits=n_splits)


@pytest.mark.parametrize("G", [1, 8])
def test_group_sizes(G):
    w = inputs.Workload("h", 1, 3, G, 128, "bf16", 1 << 20, 0, 0, 2, sigma=1.0)
    _run(w, 42, [129, 300], cap=310, steps=2, n_splits=2, out_dtype="bf16")


def test_helper_geometry_16k_context():
    """Qwen2.5-Math-1.5B head geometry (12 q / 2 kv heads, d 128) at context
    16384 (4 of its 28 layers), N(0,1)/sqrt(128) inputs, library-chosen
    splits."""
    w = inputs.Workload("h16k", 4, 2, 6, 128, "bf16", 1 << 20, 0, 0, 2,
                        sigma=1.0 / np.sqrt(128.0))
    _run(w, 43, [16384], cap=16386, steps=2, n_splits=0)


def test_workspace_and_shape_errors():
    w = inputs.Workload("h", 1, 1, 2, 128, "bf16", 1 << 20, 0, 0, 1, sigma=1.0)
    c, _ = harness.make_pair(w, 44, 1, cap=300, prompt_lens=[200])
    q, kn, vn = (harness.dev(a, "bf16") for a in inputs.step_inputs(w, 44, 0, 1))
    need = kvr.kvr_decode_attend_workspace_bytes(c.handle, 0, 1, 4)
    ws = torch.empty(need - 16, dtype=torch.uint8, device="cuda")
    with pytest.raises(kvr.KvrError) as e:
        kvr.kvr_decode_attend(c.handle, 0, 1, q, kn, vn, c.new_out(1), 4, ws,
                              ws.numel())
    assert e.value.status == kvr.KVR_ENOMEM
    w32 = inputs.Workload("h", 1, 1, 2, 64, "f32", 1 << 20, 0, 0, 1, sigma=1.0)
    c32, _ = harness.make_pair(w32, 45, 1, cap=8, prompt_lens=[4])
    q, kn, vn = (harness.dev(a, "f32") for a in inputs.step_inputs(w32, 45, 0, 1))
    with pytest.raises(kvr.KvrError) as e:
        kvr.attend_full(c32, q, kn, vn)
    assert e.value.status == kvr.KVR_EINVAL


def test_helper_full_size_sampled():
    """bench.py --mode helper's launch: 16 sequences x all 28 layers of the
    1.5B geometry at context 16384, library-chosen splits, bf16 out.  The
    oracle holds sequences 0 and 15 (sequences are independent; the others
    run alongside on device-drawn prompts) and checks their outputs at every
    step, and the appended rows' lengths and positions."""
    w = inputs.WORKLOADS["1p5b_full16k"]
    S, samp, ctx = 16, [0, 15], w.prompt
    c, o = harness.make_pair(w, 46, S, cap=ctx + 3, prompt_lens=[ctx] * S,
                             out_dtype="bf16", sample=samp)
    n0 = c.launch_count()
    for t in range(2):
        q, kn, vn = inputs.step_inputs(w, 46, t, S)
        out = kvr.attend_full(c, *(harness.dev(a, "bf16") for a in (q, kn, vn)))
        ref = o.step(q[samp], kn[samp], vn[samp], evict=False)
        torch.cuda.synchronize()
        parity.check_out(out[samp].float().cpu().numpy(), ref,
                         what=f"out at {t}")
        assert (c.lengths() == ctx + t + 1).all()
        for i, s in enumerate(samp):
            ex = c.export(s, kv=False)
            assert (ex["pos"][:, :, ctx + t] == ctx + t).all()
    assert c.launch_count() - n0 == 2 * 2   # split partials + combine a step
    c.sync_status()
    harness.check_guards(c)
