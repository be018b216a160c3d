"""R-KV eviction (kvr_evict_compact_rkv, and the one-launch step
kvr_decode_step_rkv) against the oracle's reading of it (oracle/rkv.py), in
lock-step: every step is kvr_decode_attend_score then the R-KV eviction (or
the fused step) on the CUDA side, and the oracle's step without eviction
then its R-KV eviction on the CPU side.  Outputs, retained scores and the
retained sets are checked after every step (parity.check_and_adopt_rkv)."""
import numpy as np
import pytest
import torch

from oracle import oracle as orc
from oracle import parity, rkv
from paper_2608_15797_gb300 import inputs, kvr
from tests import harness

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    torch.cuda.set_device(0)


def rkv_lockstep(c, o, w, seed, steps, B, W, lam, step0=0, sample=None,
                 fused=False):
    """`steps` R-KV steps on both sides; with `sample` the oracle holds only
    those sequences (harness.make_pair) and only they are checked.  fused:
    the CUDA side runs kvr_decode_step_rkv (one launch where it applies)
    instead of attend+score followed by the R-KV eviction."""
    samp = list(range(c.S)) if sample is None else list(sample)
    stats = parity.Stats()
    for t in range(step0, step0 + steps):
        q, kn, vn = inputs.step_inputs(w, seed, t, c.S)
        qd, kd, vd = (harness.dev(a, w.dtype) for a in (q, kn, vn))
        if fused:
            out = c.step_rkv(qd, kd, vd, B, W, lam)
        else:
            out = c.attend_score(qd, kd, vd)
            c.evict_rkv(B, W, lam)
        ref = o.step(q[samp], kn[samp], vn[samp], evict=False)
        torch.cuda.synchronize()
        parity.check_out(out[samp].float().cpu().numpy(), ref, what=f"out {t}")
        exports = [c.export(s, kv=False) for s in samp]
        stats.merge(parity.check_and_adopt_rkv(o, exports, B, W, lam))
    c.sync_status()
    return stats


@pytest.mark.parametrize("lam", [0.0, 0.1, 0.5, 1.0])
def test_rkv_tiny(lam):
    w = inputs.WORKLOADS["tiny"]
    c, o = harness.make_pair(w, 41, 2, cap=w.prompt + 1)
    st = rkv_lockstep(c, o, w, 41, 30, w.budget, w.window, lam)
    assert st.units > 0


@pytest.mark.parametrize("lam", [0.1, 1.0])
def test_rkv_7b(lam):
    """7B, B = 64, W = 8: the first step evicts a 200-row prompt, then one
    row a step."""
    w = inputs.WORKLOADS["7b_b64"]
    c, o = harness.make_pair(w, 42, 1, cap=201, prompt_lens=[200])
    rkv_lockstep(c, o, w, 42, 12, w.budget, w.window, lam)


def test_rkv_unscaled_keys_and_ragged_lengths():
    """Peaked attention (unscaled keys), sequences of different lengths, a
    budget of 0 and of 1 (first evictions dropping up to 26 rows)."""
    w2 = inputs.Workload("u", 3, 2, 4, 128, "bf16", 1, 3, 0, 0, sigma=1.0)
    for wk, B in ((w2, 1), (w2, 0)):
        c, o = harness.make_pair(wk, 43, 3, cap=40, prompt_lens=[30, 4, 0])
        rkv_lockstep(c, o, wk, 43, 8, B, wk.window, 0.1)


@pytest.mark.parametrize("d,dtype", [(64, "f32"), (128, "bf16")])
def test_rkv_duplicate_and_zero_keys(d, dtype):
    """Keys that repeat, and a zero key: with lambda = 0 the duplicates are
    the most redundant rows and go first; a zero key has cosine 0."""
    n = 24
    rng = np.random.default_rng(44)
    K = inputs.round_to(rng.standard_normal((n, d)).astype(np.float32), dtype)
    K[5] = K[2]
    K[9] = K[2]
    K[14] = 0.0
    V = inputs.round_to(rng.standard_normal((n, d)).astype(np.float32), dtype)
    w = inputs.Workload("z", 1, 1, 2, d, dtype, 10, 2, n, 0, sigma=1.0)
    c = kvr.Cache(1, 1, 1, 2, d, n + 1, kv_dtype=dtype, out_dtype="f32")
    o = orc.OracleCache(1, 1, 1, 2, d, n + 1)
    c.load(0, harness.dev(K[None, None], dtype), harness.dev(V[None, None], dtype))
    o.load(0, K[None, None], V[None, None])
    q, kn, vn = inputs.step_inputs(w, 44, 0, 1)
    c.attend_score(*(harness.dev(a, dtype) for a in (q, kn, vn)))
    o.step(q, kn, vn, evict=False)
    c.evict_rkv(10, 2, 0.0)
    got = set(c.export(0, kv=False)["pos"][0, 0, :12].tolist())
    want = rkv.rkv_keep(o.K[0, 0, 0, :n + 1], o.score[0, 0, 0, :n + 1],
                        o.pos[0, 0, 0, :n + 1], 10, 2, 0.0)
    assert got == want
    assert not {2, 5, 9} <= got


def test_rkv_errors():
    w = inputs.WORKLOADS["tiny"]
    c, _ = harness.make_pair(w, 45, 1, cap=w.prompt + 1)
    for lam in (-0.1, 1.5, float("nan")):
        with pytest.raises(kvr.KvrError) as e:
            c.evict_rkv(w.budget, w.window, lam)
        assert e.value.status == kvr.KVR_EINVAL
    f = kvr.Fork(c, 2, 4)
    with pytest.raises(kvr.KvrError) as e:
        c.evict_rkv(w.budget, w.window, 0.1)
    assert e.value.status == kvr.KVR_ESTATE
    del f


# The one-launch R-KV step at each group shape of the fused kernel: units
# of (B + W + 1) rows staged as T 16-row tiles over U warps (21 rows: T = 2,
# U = 2; 73: T = 5, U = 3; 109: T = 7, U = 4; 8: one warp; 137: T = 9,
# U = 5; 160: T = 10, U = 5).
@pytest.mark.parametrize("B,W,G", [(16, 4, 7), (64, 8, 7), (100, 8, 8),
                                   (5, 2, 3), (128, 8, 7), (151, 8, 8)])
@pytest.mark.parametrize("lam", [0.0, 0.1, 1.0])
def test_rkv_fused_step_shapes(B, W, G, lam):
    w = inputs.Workload("rf", 2, 3, G, 128, "bf16", B, W, B + W, 0, sigma=1.0)
    c, o = harness.make_pair(w, 46 + B, 2, cap=B + W + 1,
                             prompt_lens=[B + W, B + W])
    n0 = c.launch_count()
    st = rkv_lockstep(c, o, w, 46 + B, 10, B, W, lam, fused=True)
    assert c.launch_count() - n0 == 10   # one launch a step
    assert st.units == 10 * 2 * w.n_layers * w.n_kv_heads
    harness.check_guards(c)


def test_rkv_fused_step_7b_scaled_and_first_eviction():
    """7B geometry (N(0, 1/128) inputs): a 200-row prompt's first eviction
    runs the two-launch path, every later step the one-launch step."""
    w = inputs.WORKLOADS["7b_b64"]
    c, o = harness.make_pair(w, 47, 2, cap=201, prompt_lens=[200, 90])
    rkv_lockstep(c, o, w, 47, 1, w.budget, w.window, 0.1, fused=True)
    n0 = c.launch_count()
    rkv_lockstep(c, o, w, 47, 12, w.budget, w.window, 0.1, step0=1,
                 fused=True)
    assert c.launch_count() - n0 == 12


def test_rkv_fused_duplicate_and_zero_keys():
    """Three identical keys and a zero key, one eviction with lambda = 0:
    the duplicates tie exactly as the most redundant rows, so the one at the
    highest position goes; the zero key (cosine 0) stays."""
    n, d, dtype = 24, 128, "bf16"
    rng = np.random.default_rng(48)
    K = inputs.round_to(rng.standard_normal((n, d)).astype(np.float32), dtype)
    K[5] = K[2]
    K[9] = K[2]
    K[14] = 0.0
    V = inputs.round_to(rng.standard_normal((n, d)).astype(np.float32), dtype)
    w = inputs.Workload("z", 1, 1, 2, d, dtype, 22, 2, n, 0, sigma=1.0)
    c = kvr.Cache(1, 1, 1, 2, d, n + 1, kv_dtype=dtype, out_dtype="f32")
    o = orc.OracleCache(1, 1, 1, 2, d, n + 1)
    c.load(0, harness.dev(K[None, None], dtype), harness.dev(V[None, None], dtype))
    o.load(0, K[None, None], V[None, None])
    q, kn, vn = inputs.step_inputs(w, 48, 0, 1)
    n0 = c.launch_count()
    c.step_rkv(*(harness.dev(a, dtype) for a in (q, kn, vn)), 22, 2, 0.0)
    assert c.launch_count() - n0 == 1
    o.step(q, kn, vn, evict=False)
    got = set(c.export(0, kv=False)["pos"][0, 0, :24].tolist())
    want = rkv.rkv_keep(o.K[0, 0, 0, :n + 1], o.score[0, 0, 0, :n + 1],
                        o.pos[0, 0, 0, :n + 1], 22, 2, 0.0)
    assert got == want
    assert 9 not in got and {2, 5, 14} <= got
    c.sync_status()


def test_rkv_fused_errors():
    w = inputs.WORKLOADS["tiny"]
    c, _ = harness.make_pair(w, 49, 1, cap=w.prompt + 1)
    q, kn, vn = (harness.dev(a, w.dtype) for a in inputs.step_inputs(w, 49, 0, 1))
    for lam in (-0.1, 1.5, float("nan")):
        with pytest.raises(kvr.KvrError) as e:
            c.step_rkv(q, kn, vn, w.budget, w.window, lam)
        assert e.value.status == kvr.KVR_EINVAL


def test_rkv_fused_kept_sum_over_a_long_run():
    """The one-launch step keeps each unit's sum of normalised keys across
    steps (the new key added, the evicted one removed): 400 steps with
    peaked attention stay in lock-step with the oracle, which sums the
    live keys afresh every step."""
    w = inputs.Workload("long", 2, 2, 7, 128, "bf16", 64, 8, 72, 0, sigma=1.0)
    c, o = harness.make_pair(w, 50, 1, cap=73, prompt_lens=[72])
    st = rkv_lockstep(c, o, w, 50, 400, w.budget, w.window, 0.1, fused=True)
    assert st.steps == 400


def test_rkv_fused_after_other_calls():
    """Calls that change a unit's rows by other means (a plain decode step,
    an import, a copy into another cache) leave no stale key sum behind:
    the next one-launch R-KV step starts afresh and stays in lock-step."""
    w = inputs.Workload("mix", 2, 2, 7, 128, "bf16", 40, 6, 46, 0, sigma=1.0)
    c, o = harness.make_pair(w, 51, 2, cap=47, prompt_lens=[46, 46])
    B, W = w.budget, w.window
    rkv_lockstep(c, o, w, 51, 3, B, W, 0.1, fused=True)
    harness.lockstep(c, o, w, 51, 2, B, W, step0=3)
    rkv_lockstep(c, o, w, 51, 3, B, W, 0.1, step0=5, fused=True)
    snap = [c.export(s) for s in range(c.S)]
    for s in range(c.S):
        c.import_state(s, snap[s])
    rkv_lockstep(c, o, w, 51, 3, B, W, 0.1, step0=8, fused=True)
    d = harness.guarded_cache(2, w.n_layers, w.n_kv_heads, w.group,
                              w.head_dim, 47, kv_dtype="bf16", out_dtype="f32")
    d.copy_from(c, np.arange(2, dtype=np.int32), np.arange(2, dtype=np.int32))
    rkv_lockstep(d, o, w, 51, 3, B, W, 0.1, step0=11, fused=True)
    harness.check_guards(d)
