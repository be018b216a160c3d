"""Parity of the CUDA decode step (through the C ABI) with the fp64 oracle.

Tolerances (oracle/parity.py): outputs |d| <= 2e-3 + 1e-2 |ref|; scores of
retained rows 1e-4 relative; retained sets exact up to swaps of oracle
near-ties (1e-4 relative), ties to the lower position.
"""
import numpy as np
import pytest
import torch

from oracle import oracle as orc
from oracle import parity
from paper_2608_15797_gb300 import inputs, kvr
from tests import harness

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    torch.cuda.set_device(0)


def test_tiny_workload_full_run():
    """Tiny: 1 layer, 4 q / 2 kv heads, d=64, fp32, prompt 128 (5% heavy
    keys) then 256 steps at B=16, W=8; the first step evicts 105 rows."""
    w = inputs.WORKLOADS["tiny"]
    c, o = harness.make_pair(w, 0, 1, cap=w.prompt + 1)
    st = harness.lockstep(c, o, w, 0, w.steps, w.budget, w.window)
    assert st.steps == 256
    assert (c.lengths() == w.budget + w.window).all()


@pytest.mark.parametrize("fused", [True, False])
def test_7b_geometry_lockstep(fused):
    """Qwen2.5-Math-7B decode geometry (28 layers, G=7, d=128, bf16,
    N(0,1)/sqrt(128)), prompt 512, B=64, W=8: 48 steps in lock-step.  The
    first step (513 rows) runs the generic kernels; the steady state runs the
    fused kernel unless it is disabled."""
    w = inputs.WORKLOADS["7b_b64"]
    c, o = harness.make_pair(w, 2, 1, cap=w.prompt + 1, fused=fused)
    st = harness.lockstep(c, o, w, 2, 48, w.budget, w.window)
    assert st.units == 48 * 28 * 4


@pytest.mark.parametrize("fused", [True, False])
def test_7b_unscaled_selection_exercised(fused):
    """Unscaled N(0,1) q/k: attention is peaked, so TopB decisions are far
    from ties and must match the oracle exactly."""
    w = inputs.WORKLOADS["7b_unscaled"]
    c, o = harness.make_pair(w, 3, 2, cap=w.prompt + 1, prompt_lens=[512, 301],
                             fused=fused)
    st = harness.lockstep(c, o, w, 3, 24, w.budget, w.window)
    assert st.adoptions == 0


@pytest.mark.parametrize("G,d,dtype", [(1, 128, "bf16"), (8, 128, "bf16"),
                                       (3, 64, "bf16"), (5, 64, "f32"),
                                       (7, 128, "f32")])
def test_group_sizes_and_dims(G, d, dtype):
    w = inputs.Workload("g", 2, 3, G, d, dtype, 9, 3, 33, 10, sigma=1.0)
    c, o = harness.make_pair(w, 4, 2, cap=40, prompt_lens=[33, 5])
    harness.lockstep(c, o, w, 4, 10, w.budget, w.window)


@pytest.mark.parametrize("fused", [True, False])
@pytest.mark.parametrize("B,W", [(1, 0), (0, 2), (5, 0), (1, 1), (30, 8)])
def test_budget_window_edges(B, W, fused):
    w = inputs.Workload("e", 1, 2, 2, 128, "bf16", B, W, 20, 8, sigma=1.0)
    c, o = harness.make_pair(w, 5, 2, cap=40, prompt_lens=[20, 1], fused=fused)
    harness.lockstep(c, o, w, 5, 8, B, W)


@pytest.mark.parametrize("G", [1, 4, 7, 8])
@pytest.mark.parametrize("B,W", [(64, 8), (100, 19), (3, 5), (128, 8),
                                 (140, 19)])
def test_fused_steady_state_shapes(G, B, W):
    """The fused kernel across group sizes and staged-row counts (the last
    16-row tile ragged or full), bf16 output, starting at B+W rows."""
    w = inputs.Workload("s", 2, 2, G, 128, "bf16", B, W, B + W, 6, sigma=1.0)
    c, o = harness.make_pair(w, 12, 3, cap=B + W + 1,
                             prompt_lens=[B + W, B + W, max(1, B + W - 9)],
                             out_dtype="bf16")
    n0 = c.launch_count()
    harness.lockstep(c, o, w, 12, 6, B, W)
    assert c.launch_count() - n0 == 6  # one fused launch per step


def test_empty_prompt_and_single_row():
    """Decoding from an empty cache: the first step attends to its own row
    only (out = v_new)."""
    w = inputs.Workload("z", 1, 2, 3, 128, "bf16", 2, 1, 0, 6, sigma=1.0)
    c, o = harness.make_pair(w, 6, 1, cap=8, prompt_lens=[0])
    q, kn, vn = inputs.step_inputs(w, 6, 0, 1)
    out = c.step(*(harness.dev(a, "bf16") for a in (q, kn, vn)), 2, 1)
    np.testing.assert_allclose(out.float().cpu().numpy()[0, 0],
                               np.repeat(vn[0, 0], 3, axis=0), rtol=0, atol=0)
    o.step(q, kn, vn, B=2, W=1)
    harness.lockstep(c, o, w, 6, 5, 2, 1, step0=1)


def test_no_eviction_is_full_attention():
    """B >= length: nothing is evicted and the output is full attention."""
    w = inputs.Workload("f", 3, 2, 4, 128, "bf16", 1000, 8, 70, 20, sigma=1.0)
    c, o = harness.make_pair(w, 7, 2, cap=100, prompt_lens=[70, 45])
    harness.lockstep(c, o, w, 7, 20, w.budget, w.window)
    assert c.lengths().tolist() == [[90] * 3, [65] * 3]


def test_long_first_eviction():
    """Prompts of ~[512, 16384] rows (the throughput workload's prior
    lengths), first step evicting thousands of rows per unit; the longest
    unit's logits exceed on-chip memory and go through the scratch area."""
    w = inputs.Workload("long", 2, 2, 7, 128, "bf16", 64, 8, 0, 3, sigma=1.0)
    lens = [9001, 600, 16384]
    c, o = harness.make_pair(w, 8, 3, cap=16385, prompt_lens=lens)
    st = harness.lockstep(c, o, w, 8, 3, 64, 8)
    assert (c.lengths() == 72).all()


def test_fused_equals_unfused_bitwise():
    w = inputs.Workload("u", 3, 2, 7, 128, "bf16", 16, 4, 50, 6, sigma=1.0)
    c1, _ = harness.make_pair(w, 9, 2, cap=60, prompt_lens=[50, 31])
    c2, _ = harness.make_pair(w, 9, 2, cap=60, prompt_lens=[50, 31])
    for t in range(6):
        q, kn, vn = (harness.dev(a, "bf16") for a in inputs.step_inputs(w, 9, t, 2))
        o1 = c1.step(q, kn, vn, 16, 4)
        o2 = c2.attend_score(q, kn, vn)
        c2.evict(16, 4)
        assert torch.equal(o1, o2)
        for s in range(2):
            e1, e2 = c1.export(s), c2.export(s)
            for l in range(3):
                for h in range(2):
                    n = e1["len"][l, h]
                    a = dict(zip(e1["pos"][l, h, :n], e1["score"][l, h, :n]))
                    b = dict(zip(e2["pos"][l, h, :n], e2["score"][l, h, :n]))
                    assert a == b


def test_selection_exact_on_kernel_scores():
    """Given the kernel's own fp32 scores, TopB must be exactly the oracle's
    selection on those same scores (no tolerance)."""
    w = inputs.Workload("x", 2, 4, 7, 128, "bf16", 20, 5, 90, 5, sigma=1.0)
    c, _ = harness.make_pair(w, 10, 2, cap=96, prompt_lens=[90, 60])
    for t in range(5):
        q, kn, vn = (harness.dev(a, "bf16") for a in inputs.step_inputs(w, 10, t, 2))
        c.attend_score(q, kn, vn)
        pre = [c.export(s, kv=False) for s in range(2)]
        c.evict(20, 5)
        post = [c.export(s, kv=False) for s in range(2)]
        for s in range(2):
            for l in range(2):
                for h in range(4):
                    n = pre[s]["len"][l, h]
                    pos = pre[s]["pos"][l, h, :n]
                    keep = orc.select_unit(pre[s]["score"][l, h, :n].astype(np.float64),
                                           pos, 20, 5)
                    m = post[s]["len"][l, h]
                    assert set(post[s]["pos"][l, h, :m].tolist()) == set(pos[keep].tolist())


def test_capacity_and_argument_errors():
    w = inputs.Workload("c", 1, 1, 2, 64, "bf16", 4, 1, 3, 2)
    c, _ = harness.make_pair(w, 11, 1, cap=4)
    q, kn, vn = (harness.dev(a, "bf16") for a in inputs.step_inputs(w, 11, 0, 1))
    c.attend_score(q, kn, vn)  # 4 rows: full
    with pytest.raises(kvr.KvrError) as e:
        c.attend_score(q, kn, vn)
    assert e.value.status == kvr.KVR_ECAPACITY
    with pytest.raises(kvr.KvrError) as e:
        c.evict(0, 0)
    assert e.value.status == kvr.KVR_EINVAL
    with pytest.raises(kvr.KvrError) as e:
        c.attend_score(q, kn, vn, layers=(0, 2))
    assert e.value.status == kvr.KVR_EINVAL
    c.evict(2, 1)
    assert c.lengths().tolist() == [[3]]
    c.sync_status()


@pytest.mark.parametrize("chunk", [(0, 0), (-1, 0)], ids=["chunked", "stream"])
@pytest.mark.parametrize("B,G,out", [(160, 7, "bf16"), (256, 7, "f32"),
                                     (512, 8, "bf16"), (170, 1, "f32")])
def test_long_unit_fused_step(B, G, out, chunk):
    """Budgets above the staged kernel's 160 rows (the throughput sweep's
    B = 256 / 512, W = 8, and two in between): the chunked kernel (and the
    older one-CTA-per-unit streaming kernel), one launch per step, in
    lock-step with the oracle from B + W rows on."""
    W = 8
    w = inputs.Workload("long_b", 2, 2, G, 128, "bf16", B, W, B + W, 5, sigma=1.0)
    c, o = harness.make_pair(w, 13, 2, cap=B + W + 1,
                             prompt_lens=[B + W, B + W - 37], out_dtype=out,
                             chunk=chunk)
    n0 = c.launch_count()
    harness.lockstep(c, o, w, 13, 5, B, W)
    assert c.launch_count() - n0 == 5


@pytest.mark.parametrize("rows", [128, 144, 160, 161, 1024, 1025, 2048, 2049])
def test_kernel_row_limits(rows):
    """Units at each one-launch kernel's row limit and one row past it (rows
    counted with the appended one): staged fused <= 160 (8, 9 and 10 row
    tiles at 128, 144 and 160), chunked <= 1024,
    streaming <= 2048, then the generic attend + evict pair.  Steady state,
    one eviction a step, ragged units, in lock-step with the oracle."""
    W = 8
    B = rows - 1 - W
    w = inputs.Workload("lim", 2, 2, 7, 128, "bf16", B, W, B + W, 4, sigma=1.0)
    c, o = harness.make_pair(w, 16, 2, cap=rows, prompt_lens=[B + W, B + W - 37],
                             out_dtype="bf16")
    n0 = c.launch_count()
    harness.lockstep(c, o, w, 16, 4, B, W)
    launches = c.launch_count() - n0
    assert launches == 4 if rows <= 2048 else launches == 8


@pytest.mark.parametrize("chunk", [(0, 0), (-1, 0)], ids=["chunked", "stream"])
def test_long_unit_growth_without_eviction(chunk):
    """Units growing from 100 to 300 rows with no eviction: the staged kernel
    while they fit, then the chunked (or streaming) kernel."""
    w = inputs.Workload("grow", 1, 2, 4, 128, "bf16", 1 << 20, 0, 0, 40, sigma=1.0)
    c, o = harness.make_pair(w, 14, 2, cap=400, prompt_lens=[100, 290],
                             chunk=chunk)
    harness.lockstep(c, o, w, 14, 40, w.budget, w.window)


def test_chunked_ring_configurations_agree_bitwise():
    """The chunked kernel's group count and ring depth change only the
    schedule: every (groups, stages) gives bit-identical outputs, scores and
    retained rows, on ragged units of 1..300 rows that cross chunk ends."""
    W, B = 8, 200
    w = inputs.Workload("cfg", 3, 2, 5, 128, "bf16", B, W, 0, 4, sigma=1.0)
    lens = [0, 31, 32, 33, 129, 300]
    res = []
    # every configuration here fits shared memory at 301 rows (the first
    # step's attend); one that did not would fall back to another kernel,
    # with other rounding
    for chunk in [(1, 2), (1, 3), (2, 2), (2, 3), (3, 2)]:
        c, _ = harness.make_pair(w, 15, len(lens), cap=310, prompt_lens=lens,
                                 chunk=chunk)
        outs = []
        for t in range(3):
            q, kn, vn = (harness.dev(a, "bf16")
                         for a in inputs.step_inputs(w, 15, t, len(lens)))
            outs.append(c.step(q, kn, vn, B, W).float().cpu().numpy())
        ex = [c.export(s, kv=True) for s in range(len(lens))]
        res.append((outs, ex))
        c.sync_status()
    for outs, ex in res[1:]:
        for a, b in zip(outs, res[0][0]):
            assert np.array_equal(a, b)
        for ea, eb in zip(ex, res[0][1]):
            assert np.array_equal(ea["len"], eb["len"])
            for l in range(w.n_layers):
                for h in range(w.n_kv_heads):
                    n = int(ea["len"][l, h])  # rows past len are unset memory
                    for key in ("pos", "score", "K", "V"):
                        assert np.array_equal(ea[key][l, h, :n], eb[key][l, h, :n])


def test_scores_view_matches_export():
    """kvr_cache_scores: the step's scores read in place on the device agree
    with the synchronising export, slot for slot."""
    w = inputs.WORKLOADS["tiny"]
    c, o = harness.make_pair(w, 61, 2, cap=w.prompt + 1)
    harness.lockstep(c, o, w, 61, 5, w.budget, w.window)
    score, pos, state = c.scores_view()
    torch.cuda.synchronize()
    for s in range(2):
        e = c.export(s, kv=False)
        n = e["len"]
        assert np.array_equal(state[s, :, :, 0].cpu().numpy(), n)
        for l in range(c.L):
            for h in range(c.H):
                k = n[l, h]
                assert np.array_equal(score[s, l, h, :k].cpu().numpy(),
                                      e["score"][l, h, :k])
                assert np.array_equal(pos[s, l, h, :k].cpu().numpy(),
                                      e["pos"][l, h, :k])


def test_host_buffer_step_equals_device_step():
    """kvr_decode_step_host (host q/k/v in, host output out, the library
    copying) gives the device call's result bit for bit, with the steps
    alternating over two streams and two staging sets (the library orders
    them), first evictions included."""
    w = inputs.Workload("h", 3, 2, 7, 128, "bf16", 10, 3, 0, 0, sigma=1.0)
    lens = [40, 13, 27]
    c1, _ = harness.make_pair(w, 71, 3, cap=41, prompt_lens=lens, out_dtype="bf16")
    c2, _ = harness.make_pair(w, 71, 3, cap=41, prompt_lens=lens, out_dtype="bf16")
    streams = [torch.cuda.Stream(), torch.cuda.Stream()]
    stage = [None, None]
    hout = [None, None]
    outs = []
    hold = []  # pinned inputs stay alive until the library's copies are done
    for t in range(8):
        q, kn, vn = (harness.dev(a, w.dtype) for a in inputs.step_inputs(w, 71, t, 3))
        outs.append(c1.step(q, kn, vn, w.budget, w.window).cpu())
        j = t % 2
        torch.cuda.synchronize()
        if stage[j] is None:
            stage[j] = tuple(torch.empty_like(x) for x in (q, kn, vn)) + \
                (torch.empty_like(outs[-1], device="cuda"),)
            hout[j] = torch.empty_like(outs[-1]).pin_memory()
        else:
            streams[j].synchronize()  # host buffers of step t - 2 read back
            assert torch.equal(hout[j], outs[t - 2]), f"step {t - 2}"
        hq, hk, hv = (x.cpu().pin_memory() for x in (q, kn, vn))
        hold.append((hq, hk, hv))
        kvr.kvr_decode_step_host(c2.handle, 0, w.n_layers, hq, hk, hv, hout[j],
                                 *stage[j], w.budget, w.window, streams[j])
    torch.cuda.synchronize()
    for t in (6, 7):
        assert torch.equal(hout[t % 2], outs[t]), f"step {t}"
    c1.sync_status()
    c2.sync_status()
    for s in range(3):
        a, b = c1.export(s), c2.export(s)
        assert np.array_equal(a["len"], b["len"]), s
        assert np.array_equal(a["next_pos"], b["next_pos"]), s
        for l in range(w.n_layers):
            for h in range(w.n_kv_heads):
                n = a["len"][l, h]  # slots past the live rows are never read
                for key in ("pos", "score", "K", "V"):
                    assert np.array_equal(a[key][l, h, :n], b[key][l, h, :n]), \
                        (s, l, h, key)


def test_export_import_resumes_bit_for_bit():
    """kvr_cache_import of what kvr_cache_export returned, into another cache
    and into another sequence slot, then decoding on: outputs and live rows
    equal the uninterrupted cache's bit for bit.  Bad states are refused."""
    w = inputs.Workload("imp", 2, 2, 7, 128, "bf16", 10, 3, 0, 0, sigma=1.0)
    c1, _ = harness.make_pair(w, 81, 2, cap=41, prompt_lens=[40, 13],
                              out_dtype="bf16")
    for t in range(3):
        q, kn, vn = (harness.dev(a, w.dtype) for a in inputs.step_inputs(w, 81, t, 2))
        c1.step(q, kn, vn, w.budget, w.window)
    saved = [c1.export(s) for s in range(2)]
    c2, _ = harness.make_pair(w, 82, 2, cap=41, prompt_lens=[5, 7], out_dtype="bf16")
    c2.import_state(0, saved[0])
    c2.import_state(1, saved[1])
    for t in range(3, 8):
        q, kn, vn = (harness.dev(a, w.dtype) for a in inputs.step_inputs(w, 81, t, 2))
        o1 = c1.step(q, kn, vn, w.budget, w.window)
        o2 = c2.step(q, kn, vn, w.budget, w.window)
        torch.cuda.synchronize()
        assert torch.equal(o1, o2), f"step {t}"
    for s in range(2):
        a, b = c1.export(s), c2.export(s)
        assert np.array_equal(a["len"], b["len"]) and np.array_equal(a["next_pos"], b["next_pos"])
        for l in range(w.n_layers):
            for h in range(w.n_kv_heads):
                n = a["len"][l, h]
                for key in ("pos", "score", "K", "V"):
                    assert np.array_equal(a[key][l, h, :n], b[key][l, h, :n]), (s, l, h, key)
    # refused states: a length past the capacity, duplicate live positions,
    # heads of one layer at different lengths
    bad = []
    x = {k: v.copy() for k, v in saved[0].items()}
    x["len"][0, 0] = 42
    bad.append(x)
    x = {k: v.copy() for k, v in saved[0].items()}
    x["pos"][1, 1, 1] = x["pos"][1, 1, 0]
    bad.append(x)
    x = {k: v.copy() for k, v in saved[0].items()}
    x["len"][1, 0] -= 1
    bad.append(x)
    for x in bad:
        with pytest.raises(kvr.KvrError) as e:
            c2.import_state(0, x)
        assert e.value.status == kvr.KVR_EINVAL
