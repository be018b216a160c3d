"""The q = 0 closed form through every step kernel, at the benchmarked sizes.

With every query row zero, every logit is exactly 0, so each of the n live
rows gets probability exactly 1/n (Eq. 1 Attn), each output is the plain
mean of the live values, and every live row's accumulated score (Sec. 2.1)
grows by 1/n a step.  Rows of the same age then hold exactly equal scores,
and which of them survive is decided by the tie rule alone: Eq. 1's TopB
with ties kept at the lower position.  From a prompt of P rows at score 0:

* step 1 (n = P + 1): every row gets 1/(P + 1); the W most recent positions
  stay and, of the rest (all tied), the B lowest positions 0 .. B-1;
* step t >= 2 (n = B + W + 1): every live row gets 1/(B + W + 1); the row
  that leaves the window ties with positions 0 .. B-1 while it is a prompt
  row (t <= W) and is younger, so lower, after that.

So after step t the retained positions are exactly {0 .. B-1} plus the W
most recent, the score of position p is the sum of 1/n over the steps it
has lived through, and the output of step t is the mean of the values at
{0 .. B-1} and the W + 1 most recent positions.  None of this needs the
oracle: the expected values are computed here in float64 from those
formulas and the inputs.

The prompt rows are imported in a random slot order per unit, so the lower
position is not the lower slot.  The cases run the kernel each budget
dispatches to at the benchmarked geometry: the fused step (7B, 64 sequences
x 28 layers x 4 KV heads, B = 64 and 128: five and nine row tiles a unit),
the chunked step (B = 256, 512; the same 7,168 units a launch, so each
persistent CTA takes many units), the
streaming step (units of 1,409 rows) and the generic pair; a prompt longer
than B + W makes step 1 the generic first eviction.  The candidate case
forks a fresh 72B parent into 8 candidates and commits one: its cut from
B + W + T rows to B + W is again decided by ties among the parent rows.

Inputs: seeded N(0, 1/128) keys and values from paper_2608_15797_gb300.inputs
(7B / 72B geometry, bf16), queries zero.
"""
import dataclasses

import numpy as np
import pytest
import torch

from oracle import parity
from paper_2608_15797_gb300 import inputs, kvr

pytestmark = pytest.mark.gpu

W = 8


@pytest.fixture(autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    torch.cuda.set_device(0)


def _scrambled_cache(w, S, P, cap, seed, fused=True):
    """A cache whose units each hold prompt positions 0..P-1 at score 0 in a
    random slot order.  Returns (cache, V by position [S][L][H][P][d])."""
    c = kvr.Cache(S, w.n_layers, w.n_kv_heads, w.group, w.head_dim, cap,
                  kv_dtype=w.dtype, out_dtype="f32")
    c.set_fused(fused)
    rng = np.random.default_rng(seed)
    L, H, d = w.n_layers, w.n_kv_heads, w.head_dim
    vpos = np.zeros((S, L, H, P, d), np.float32)
    for s in range(S):
        k, v = inputs.prompt(w, seed, s, P)
        vpos[s] = v
        perm = np.argsort(rng.random((L, H, P)), axis=-1).astype(np.int32)
        hk = np.zeros((L, H, cap, d), np.float32)
        hv = np.zeros((L, H, cap, d), np.float32)
        hk[:, :, :P] = np.take_along_axis(k, perm[..., None], axis=2)
        hv[:, :, :P] = np.take_along_axis(v, perm[..., None], axis=2)
        pos = np.zeros((L, H, cap), np.int32)
        pos[:, :, :P] = perm
        c.import_state(s, {"K": hk, "V": hv,
                           "score": np.zeros((L, H, cap), np.float32),
                           "pos": pos,
                           "len": np.full((L, H), P, np.int32),
                           "next_pos": np.full((L, H), P, np.int32)})
    return c, vpos


def _expected_scores(P, B, t, positions):
    """Closed-form score of each position after step t (see the module
    docstring): the sum of 1/n over the steps the row has lived through."""
    m = B + W
    out = np.zeros(len(positions), np.float64)
    for i, p in enumerate(positions):
        enter = 1 if p < P else p - P + 1
        out[i] = sum((1.0 / (P + 1)) if tau == 1 else 1.0 / (m + 1)
                     for tau in range(enter, t + 1))
    return out


def _check_state(c, B, P, t, where):
    """Retained positions exactly {0..B-1} + the W most recent, scores as
    the closed form, in every unit."""
    sc, ps, st = c.scores_view()
    torch.cuda.synchronize()
    m = B + W
    ln = st[..., 0].cpu().numpy()
    assert (ln == m).all(), f"{where}: live lengths {np.unique(ln)}"
    pos = ps[..., :m].cpu().numpy()
    score = sc[..., :m].cpu().numpy().astype(np.float64)
    order = np.argsort(pos, axis=-1)
    pos = np.take_along_axis(pos, order, axis=-1)
    score = np.take_along_axis(score, order, axis=-1)
    want = np.concatenate([np.arange(B), np.arange(P + t - W, P + t)])
    bad = np.nonzero((pos != want).any(axis=-1).reshape(-1))[0]
    if bad.size:
        u = np.unravel_index(bad[0], pos.shape[:-1])
        raise parity.ParityError(
            f"{where}: unit {u} retained {sorted(set(pos[u]) ^ set(want))[:8]}"
            f" (symmetric difference with the tie rule's set)")
    ref = _expected_scores(P, B, t, want)
    rel = np.abs(score - ref) / np.maximum(ref, parity.SCORE_FLOOR)
    assert rel.max() <= parity.SCORE_RTOL, f"{where}: score rel {rel.max():.3g}"
    return float(rel.max())


@pytest.mark.parametrize("B,S,L,extra,fused", [
    (64, 64, 28, 0, True),      # fused step at the headline's size
    (64, 64, 28, 40, True),     # generic first eviction, then fused
    (128, 64, 28, 0, True),     # fused step, nine row tiles
    (200, 16, 28, 0, True),     # chunked step (209 rows)
    (256, 64, 28, 0, True),
    (512, 64, 28, 0, True),
    (1400, 2, 4, 0, True),      # streaming step (1,409 rows)
    (64, 4, 4, 0, False),       # generic attend + evict
])
def test_zero_query_keeps_the_lowest_positions(B, S, L, extra, fused):
    w = dataclasses.replace(inputs.WORKLOADS["7b_b64"], budget=B, window=W,
                            n_layers=L, n_seq=S)
    P = B + W + extra
    seed = 70 + B + extra
    c, vpos = _scrambled_cache(w, S, P, cap=P + 1, seed=seed, fused=fused)
    H, G, d = w.n_kv_heads, w.group, w.head_dim
    q = torch.zeros(S, L, H * G, d, dtype=torch.bfloat16, device="cuda")
    steps = W + 4
    vnew = []
    launches0 = c.launch_count()
    head = np.sum(vpos[:, :, :, :B], axis=3, dtype=np.float64)   # [S,L,H,d]
    every = np.sum(vpos, axis=3, dtype=np.float64)

    def value(p):
        return vpos[:, :, :, p] if p < P else vnew[p - P]

    for t in range(1, steps + 1):
        _, kn, vn = inputs.step_inputs(w, seed, t, S)
        vnew.append(vn)
        out = c.step(q, torch.from_numpy(kn).to("cuda", torch.bfloat16),
                     torch.from_numpy(vn).to("cuda", torch.bfloat16), B, W)
        torch.cuda.synchronize()
        # Output: the mean of the live values, {0..B-1} and the W+1 most
        # recent positions (every row at step 1).
        if t == 1:
            ref = (every + vn) / (P + 1)
        else:
            recent = sum(value(p).astype(np.float64)
                         for p in range(P + t - 1 - W, P + t))
            ref = (head + recent) / (B + W + 1)
        parity.check_out(out.cpu().numpy(), np.repeat(ref, G, axis=2),
                         what=f"out at step {t}")
        _check_state(c, B, P, t, f"B={B} step {t}")
    c.sync_status()
    # One launch a step; the generic path (and a first eviction of many
    # rows) runs attend+score and the eviction as two.
    want = steps + (1 if extra else 0) if fused else 2 * steps
    assert c.launch_count() - launches0 == want


def test_zero_query_candidates_commit_the_lowest_positions():
    """72B, the bench's 4 sequences x 80 layers x 8 KV heads, 8 candidates:
    a fresh parent of B + W prompt rows (score 0) forks, every candidate
    decodes T tokens with q = 0, and the commit cuts the chosen one from
    B + W + T rows back to B + W.  Every parent row has lived T tokens and
    holds the same score, above every tail row's, so the commit keeps
    positions 0 .. B-1 and the W most recent tail rows."""
    w = inputs.WORKLOADS["72b_bon8"]
    S, B, N, T = 4, w.budget, w.n_cand, 20
    m = B + W
    c, vpos = _scrambled_cache(w, S, m, cap=m + T + 1, seed=77)
    L, H, G, d = w.n_layers, w.n_kv_heads, w.group, w.head_dim
    f = kvr.Fork(c, N, T)
    q = torch.zeros(N, S, L, H * G, d, dtype=torch.bfloat16, device="cuda")
    tails = []
    for t in range(T):
        per = [inputs.step_inputs(w, 77, 10_000 + t, S, cand=k + 1)
               for k in range(N)]
        K = np.stack([p[1] for p in per])
        V = np.stack([p[2] for p in per])        # [N][S][L][H][d]
        tails.append(V)
        out = f.attend_score(q, torch.from_numpy(K).to("cuda", torch.bfloat16),
                             torch.from_numpy(V).to("cuda", torch.bfloat16))
        torch.cuda.synchronize()
        # candidate k: mean over the m parent rows and its t+1 tail rows
        tot = vpos.astype(np.float64).sum(axis=3)[None]           # [1,S,L,H,d]
        tot = tot + np.stack(tails).astype(np.float64).sum(axis=0)
        ref = np.repeat(tot / (m + t + 1), G, axis=3)
        parity.check_out(out.cpu().numpy(), ref, what=f"candidate token {t}")
    chosen = inputs.candidate_pick(77, 0, S, N)
    f.commit(chosen, B, W)
    del f
    sc, ps, st = c.scores_view()
    torch.cuda.synchronize()
    assert (st[..., 0].cpu().numpy() == m).all()
    pos = np.sort(ps[..., :m].cpu().numpy(), axis=-1)
    want = np.concatenate([np.arange(B), np.arange(m + T - W, m + T)])
    assert (pos == want).all(), "commit broke the tie rule"
    order = np.argsort(ps[..., :m].cpu().numpy(), axis=-1)
    score = np.take_along_axis(sc[..., :m].cpu().numpy(), order, axis=-1)
    inv = [1.0 / (m + t + 1) for t in range(T)]
    ref = np.array([sum(inv)] * B + [sum(inv[p - m:]) for p in want[B:]])
    rel = np.abs(score - ref) / ref
    assert rel.max() <= parity.SCORE_RTOL
    c.sync_status()
