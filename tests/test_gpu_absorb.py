"""Absorbing a chunk of tokens (kvr_absorb_chunk) against the oracle: c
tokens attended causally in one call, scores accumulated from every token,
one eviction to B + W at the end; then ordinary decode steps continue from
the resulting state in lock-step."""
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


def absorb_lockstep(c, o, w, seed, chunk, B, W, evict=True, step0=20_000,
                    sample=None):
    """One absorb call on both sides, checking every token's output, then the
    retained rows and scores of every unit (of the sequences `sample` only,
    when the oracle holds just those)."""
    S = c.S
    samp = list(range(S)) if sample is None else list(sample)
    toks = [inputs.step_inputs(w, seed, step0 + j, S) for j in range(chunk)]
    q, kn, vn = (np.stack([t[i] for t in toks], axis=2) for i in range(3))
    out = c.absorb(harness.dev(q, w.dtype), harness.dev(kn, w.dtype),
                   harness.dev(vn, w.dtype), B, W, evict=evict)
    ref = o.absorb(q[samp], kn[samp], vn[samp], B=B, W=W, evict=False)
    torch.cuda.synchronize()
    got = out[samp].float().cpu().numpy()
    for j in range(chunk):
        parity.check_out(got[:, :, j], ref[:, :, j], what=f"token {j} of the chunk")
    exports = [c.export(s, kv=False) for s in samp]
    st = parity.check_and_adopt(o, exports, B, W, evict=evict)
    c.sync_status()
    return st


# The absorb paths: the one-launch kernel on tcgen05 (default) or mma.sync,
# and the token-by-token path (one attend+score launch a token, then one
# eviction).
PATHS = {"tc": (True, 0), "mma": (True, 1), "tokenwise": (False, 0)}


def _pair(w, seed, S, cap, prompt_lens, path):
    fused, kernel = PATHS[path]
    c, o = harness.make_pair(w, seed, S, cap=cap, prompt_lens=prompt_lens,
                             fused=fused)
    c.set_absorb_kernel(kernel)
    return c, o


@pytest.mark.parametrize("path", list(PATHS))
@pytest.mark.parametrize("G,d,dtype", [(7, 128, "bf16"), (1, 128, "bf16"),
                                       (8, 128, "bf16"), (3, 64, "f32")])
@pytest.mark.parametrize("chunk", [1, 5, 33, 64])
def test_absorb_shapes(G, d, dtype, chunk, path):
    """Ragged units (an empty one included), chunks crossing tile ends, then
    three decode steps."""
    B, W = 12, 4
    w = inputs.Workload("ab", 2, 2, G, d, dtype, B, W, 20, 0, sigma=1.0)
    c, o = _pair(w, 50, 3, 20 + chunk + 4, [20, 0, 9], path)
    absorb_lockstep(c, o, w, 50, chunk, B, W)
    # The one-launch kernels take bf16 with d = 128; the rest runs token by
    # token.
    one_launch = d == 128 and dtype == "bf16" and path != "tokenwise"
    assert c.last_absorb_kernel() == (PATHS[path][1] if one_launch else 2)
    harness.lockstep(c, o, w, 50, 3, B, W, step0=100)


@pytest.mark.parametrize("path", list(PATHS))
def test_absorb_without_eviction_grows_every_unit(path):
    w = inputs.Workload("ab", 1, 2, 4, 128, "bf16", 8, 2, 10, 0, sigma=1.0)
    c, o = _pair(w, 51, 2, 40, [10, 3], path)
    absorb_lockstep(c, o, w, 51, 17, 8, 2, evict=False)
    assert c.lengths().tolist() == [[27], [20]]


@pytest.mark.parametrize("path", list(PATHS))
def test_absorb_7b_helper_step(path):
    """7B geometry (28 layers, G=7), an evicted cache at B+W = 72 rows absorbs
    an accepted 64-token step in one call, evicts back to 72, then decodes."""
    w = inputs.WORKLOADS["7b_unscaled"]
    B, W = w.budget, w.window
    c, o = _pair(w, 52, 2, B + W + 64 + 1, [B + W, B + W - 30], path)
    n0 = c.launch_count()
    absorb_lockstep(c, o, w, 52, 64, B, W)
    if PATHS[path][0]:
        assert c.launch_count() - n0 == 1  # one launch for the whole chunk
    assert (c.lengths() <= B + W).all()
    harness.lockstep(c, o, w, 52, 4, B, W, step0=200)


def test_absorb_prompt_seeds_scores():
    """An empty cache absorbs a 200-token prompt: the scores it keeps are the
    prompt's own causal attention (not zeros), and the cut to B + W keeps
    the window and the best-attended rows."""
    w = inputs.Workload("pp", 2, 2, 7, 128, "bf16", 24, 8, 0, 0, sigma=1.0)
    c, o = harness.make_pair(w, 53, 2, cap=201, prompt_lens=[0, 0])
    absorb_lockstep(c, o, w, 53, 200, w.budget, w.window)
    e = c.export(0, kv=False)
    assert (e["len"] == 32).all()
    assert (e["score"][:, :, :32] > 0).all()


def test_absorb_errors():
    w = inputs.Workload("er", 1, 1, 2, 128, "bf16", 4, 2, 8, 0, sigma=1.0)
    c, _ = harness.make_pair(w, 54, 1, cap=12)
    q = torch.zeros(1, 1, 5, 2, 128, dtype=torch.bfloat16, device="cuda")
    k = torch.zeros(1, 1, 5, 1, 128, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(kvr.KvrError) as e:
        c.absorb(q, k, k, 4, 2)
    assert e.value.status == kvr.KVR_ECAPACITY
    with pytest.raises(kvr.KvrError) as e:
        kvr.kvr_absorb_chunk(c.handle, 0, 1, 0, q, k, k, q, 4, 2)
    assert e.value.status == kvr.KVR_EINVAL
    assert c.lengths().tolist() == [[8]]


@pytest.mark.parametrize("path", list(PATHS))
def test_absorb_into_a_longer_than_budget_unit(path):
    """Units above B + W before the chunk (a prompt loaded with zero scores):
    the cut moves surviving old rows as well as placing new ones."""
    w = inputs.Workload("lo", 1, 2, 5, 128, "bf16", 16, 4, 60, 0, sigma=1.0)
    c, o = _pair(w, 55, 2, 100, [60, 25], path)
    absorb_lockstep(c, o, w, 55, 40, w.budget, w.window)
    harness.lockstep(c, o, w, 55, 2, w.budget, w.window, step0=300)


@pytest.mark.parametrize("path", ["tc", "mma"])
def test_absorb_full_unit_and_128_row_tiles(path):
    """The largest unit the one-launch kernels take (128 old rows + a
    64-token chunk = 192 rows) and G = 8, so the 512 query rows fill four
    128-row tiles exactly."""
    w = inputs.Workload("fu", 2, 2, 8, 128, "bf16", 100, 8, 128, 0, sigma=1.0)
    c, o = _pair(w, 56, 2, 192, [128, 127], path)
    absorb_lockstep(c, o, w, 56, 64, w.budget, w.window)
    harness.lockstep(c, o, w, 56, 2, w.budget, w.window, step0=400)


@pytest.mark.parametrize("G", [2, 4, 5, 6])
@pytest.mark.parametrize("chunk", [37, 64])
def test_absorb_tc_tiles_of_whole_tokens(G, chunk):
    """Each query tile of the tensor-memory kernel holds 128 // G whole
    tokens (one q box per 64-column half): G = 5 and 6 leave the tile's last
    rows unused (125 and 126 rows), and a 37-token chunk leaves a ragged last
    tile whose box reaches into the next unit's tokens (or past the end of
    q for the last unit)."""
    w = inputs.Workload("tg", 2, 2, G, 128, "bf16", 60, 8, 72, 0, sigma=1.0)
    c, o = _pair(w, 70 + G, 2, 72 + chunk + 1, [72, 50], "tc")
    absorb_lockstep(c, o, w, 70 + G, chunk, w.budget, w.window)
    assert c.last_absorb_kernel() == 0
    harness.lockstep(c, o, w, 70 + G, 2, w.budget, w.window, step0=600)


@pytest.mark.parametrize("G,old", [(8, 80), (7, 72), (3, 79)])
def test_absorb_tc_largest_unit(G, old):
    """The tensor-memory kernel's largest units (old rows + a 64-token chunk
    up to its 144-row limit; with G = 8 the 512 query rows fill four 128-row
    tiles), units of unequal length in one launch, and a 145-row unit
    routed to the mma.sync kernel in the same way."""
    w = inputs.Workload("tl", 2, 2, G, 128, "bf16", 60, 8, old, 0, sigma=1.0)
    c, o = _pair(w, 57 + G, 2, old + 64 + 1, [old, old - 9], "tc")
    absorb_lockstep(c, o, w, 57 + G, 64, w.budget, w.window)
    assert c.last_absorb_kernel() == 0
    harness.lockstep(c, o, w, 57 + G, 2, w.budget, w.window, step0=500)
    c, o = _pair(w, 60 + G, 1, 146, [81], "tc")
    assert c.last_absorb_kernel() == -1
    absorb_lockstep(c, o, w, 60 + G, 64, w.budget, w.window)
    assert c.last_absorb_kernel() == 1
