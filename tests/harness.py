"""Drivers that run the CUDA path and the fp64 oracle side by side.

Test infrastructure: used by the GPU parity tests and by
``__graft_entry__.smoke()``.  Inputs come from the seeded generators of
``paper_2608_15797_gb300.inputs``; the CUDA path is driven through the C ABI
(via the ctypes binding), the oracle through ``oracle.oracle``.
"""
from __future__ import annotations

import numpy as np
import torch

from oracle import oracle as orc
from oracle import parity
from paper_2608_15797_gb300 import inputs, kvr


# Canary guard regions: every device buffer the parity runs hand to the
# library sits between two GUARD-byte regions filled with CANARY, and the
# regions are checked after each run, so a write past either end of a
# caller buffer fails the test that made it.
GUARD, CANARY = 4096, 0xA5


class Guarded:
    """A uint8 device buffer of nbytes with canary regions on both sides
    (the buffer keeps the allocation's 256-byte alignment)."""

    def __init__(self, nbytes, device="cuda"):
        self.raw = torch.full((nbytes + 2 * GUARD,), CANARY, dtype=torch.uint8,
                              device=device)
        self.buf = self.raw[GUARD:GUARD + nbytes]

    def intact(self) -> bool:
        return bool((self.raw[:GUARD] == CANARY).all().item() and
                    (self.raw[GUARD + self.buf.numel():] == CANARY).all().item())


def guarded_tensor(shape, dtype, owner=None, device="cuda"):
    """An uninitialised tensor inside a Guarded buffer; the guard is kept on
    `owner._guards` for check_guards."""
    n = int(np.prod(shape)) * torch.empty((), dtype=dtype).element_size()
    g = Guarded(n, device)
    if owner is not None:
        owner.__dict__.setdefault("_guards", []).append(g)
    return g.buf.view(dtype).view(*shape)


def check_guards(*owners):
    """Every canary region of the owners' buffers is unchanged."""
    torch.cuda.synchronize()
    for o in owners:
        for g in o.__dict__.get("_guards", []):
            if not g.intact():
                raise parity.ParityError("a canary region next to a caller "
                                         "buffer was overwritten")


def guarded_cache(*args, **kw) -> kvr.Cache:
    """kvr.Cache in a Guarded buffer."""
    probe = kvr.make_desc(*args[:6], kw.get("kv_dtype", "bf16"),
                          kw.get("out_dtype", "bf16"))
    g = Guarded(kvr.kvr_cache_required_bytes(probe))
    c = kvr.Cache(*args, buf=g.buf, **kw)
    c._guards = [g]
    return c


def guarded_fork(c: kvr.Cache, n_cand, tail_cap, kernel=0) -> kvr.Fork:
    g = Guarded(kvr.kvr_fork_required_bytes(c.handle, n_cand, tail_cap))
    f = kvr.Fork(c, n_cand, tail_cap, kernel=kernel, buf=g.buf)
    f._guards = [g]
    return f


def dev(x: np.ndarray, dtype: str) -> torch.Tensor:
    """Element-type-exact float32 host values -> device tensor of dtype."""
    return torch.from_numpy(np.ascontiguousarray(x)).to(
        device="cuda", dtype=kvr.TORCH_DTYPES[dtype])


def make_pair(w: inputs.Workload, seed: int, S: int, cap: int,
              prompt_lens=None, out_dtype="f32", first_pos=None, fused=True,
              chunk=(0, 0), sample=None):
    """A CUDA cache and an oracle cache loaded with the same prompts.
    fused=False restricts the CUDA cache to the generic kernels; chunk is
    the chunked kernel's (groups, stages) tuning, groups -1 turning it off.
    With `sample` (a list of sequence indices) the oracle holds only those
    sequences, in that order; the others get device-drawn prompts of the
    same lengths, which no check reads (sequences are independent)."""
    c = guarded_cache(S, w.n_layers, w.n_kv_heads, w.group, w.head_dim, cap,
                      kv_dtype=w.dtype, out_dtype=out_dtype)
    c.set_fused(fused)
    c.set_chunk_tuning(*chunk)
    samp = list(range(S)) if sample is None else list(sample)
    o = orc.OracleCache(len(samp), w.n_layers, w.n_kv_heads, w.group,
                        w.head_dim, cap)
    lens = [w.prompt] * S if prompt_lens is None else list(prompt_lens)
    gen = torch.Generator(device="cuda")
    gen.manual_seed(seed + 1_000_003)
    for s in range(S):
        n = int(lens[s])
        fp = 0 if first_pos is None else int(first_pos[s])
        if s in samp:
            k, v = inputs.prompt(w, seed, s, n)
            c.load(s, dev(k, w.dtype), dev(v, w.dtype), first_pos=fp)
            o.load(samp.index(s), k, v, first_pos=fp)
        else:
            shape = (w.n_layers, w.n_kv_heads, n, w.head_dim)
            k, v = (torch.randn(shape, generator=gen, device="cuda")
                    .mul_(w.sigma).to(kvr.TORCH_DTYPES[w.dtype])
                    for _ in range(2))
            c.load(s, k, v, first_pos=fp)
    return c, o


def lockstep(c: kvr.Cache, o: orc.OracleCache, w: inputs.Workload, seed: int,
             steps: int, budget: int, window: int, fused: bool = True,
             step0: int = 0, layers=None, evict: bool = True,
             sample=None) -> parity.Stats:
    """Run `steps` decode steps on both sides, checking after every step
    (the sequences `sample` only, when the oracle holds just those)."""
    S = c.S
    samp = list(range(S)) if sample is None else list(sample)
    stats = parity.Stats()
    lb, le = (0, c.L) if layers is None else layers
    for t in range(step0, step0 + steps):
        q, kn, vn = inputs.step_inputs(w, seed, t, S, n_layers=le - lb)
        qd, kd, vd = (dev(a, w.dtype) for a in (q, kn, vn))
        if t == step0:
            out_buf = guarded_tensor((S, le - lb, c.H * c.G, c.d),
                                     c.out_torch_dtype, owner=c)
        out = out_buf
        if not evict:
            c.attend_score(qd, kd, vd, out=out, layers=(lb, le))
        elif fused:
            c.step(qd, kd, vd, budget, window, out=out, layers=(lb, le))
        else:
            c.attend_score(qd, kd, vd, out=out, layers=(lb, le))
            c.evict(budget, window, layers=(lb, le))
        ref = o.step(q[samp], kn[samp], vn[samp], evict=False, layer_begin=lb,
                     layer_end=le)
        torch.cuda.synchronize()
        stats.max_out_excess = max(stats.max_out_excess, parity.check_out(
            out[samp].float().cpu().numpy(), ref, what=f"out at step {t}"))
        exports = [c.export(s, kv=False) for s in samp]
        st = parity.check_and_adopt(o, exports, budget, window, evict=evict,
                                    layers=(lb, le))
        stats.merge(st)
        stats.steps = t - step0 + 1
    c.sync_status()
    check_guards(c)
    return stats


def _unit_map(pos, score):
    return dict(zip(np.asarray(pos).tolist(), np.asarray(score, np.float64).tolist()))


def fork_lockstep(c: kvr.Cache, o: orc.OracleCache, w: inputs.Workload,
                  seed: int, n_cand: int, steps: int, budget: int, window: int,
                  pick_step: int = 0, tail_cap=None, kernel: int = 0):
    """Fork both sides into n_cand candidates, decode `steps` tokens per
    candidate checking every candidate after every token (outputs; scores of
    every prefix and tail row, by position), then commit a seeded pick (the
    stand-in for the PRM argmax of Eq. 2) on both sides and check the parent.
    Returns (oracle after commit, chosen, stats); stats.kernels lists the
    kernel that ran each token (kvr_fork_last_kernel)."""
    S = c.S
    parent_pos = [c.export(s, kv=False) for s in range(S)]
    f = guarded_fork(c, n_cand, tail_cap or steps, kernel=kernel)
    cands = o.fork(n_cand)
    stats = parity.Stats()
    stats.kernels = []
    for t in range(steps):
        per = [inputs.step_inputs(w, seed, 10_000 + t, S, cand=k + 1)
               for k in range(n_cand)]
        Q, K, V = (np.stack([p[i] for p in per]) for i in range(3))
        if t == 0:
            out_buf = guarded_tensor((n_cand, S, c.L, c.H * c.G, c.d),
                                     c.out_torch_dtype, owner=f)
        out = f.attend_score(dev(Q, w.dtype), dev(K, w.dtype), dev(V, w.dtype),
                             out=out_buf)
        stats.kernels.append(f.last_kernel())
        torch.cuda.synchronize()
        out = out.float().cpu().numpy()
        for k in range(n_cand):
            ref = cands[k].step(*per[k], evict=False)
            stats.max_out_excess = max(stats.max_out_excess, parity.check_out(
                out[k], ref, what=f"candidate {k} out at token {t}"))
            for s in range(S):
                ex = f.export(k, s)
                for l in range(c.L):
                    for h in range(c.H):
                        n_p = parent_pos[s]["len"][l, h]
                        n_t = ex["tail_len"][l, h]
                        got = _unit_map(parent_pos[s]["pos"][l, h, :n_p],
                                        ex["prefix_score"][l, h, :n_p])
                        got.update(_unit_map(ex["tail_pos"][l, h, :n_t],
                                             ex["tail_score"][l, h, :n_t]))
                        p_ref, s_ref, _, _ = cands[k].unit_rows(s, l, h)
                        want = _unit_map(p_ref, s_ref)
                        if got.keys() != want.keys():
                            raise parity.ParityError(
                                f"candidate {k} seq {s} layer {l} head {h}: "
                                f"rows differ at token {t}")
                        a = np.array([got[p] for p in want])
                        b = np.array([want[p] for p in want])
                        rel = np.abs(a - b) / np.maximum(np.abs(b), parity.SCORE_FLOOR)
                        if rel.max() > parity.SCORE_RTOL:
                            raise parity.ParityError(
                                f"candidate {k} seq {s} layer {l} head {h}: score"
                                f" rel {rel.max():.3g} at token {t}")
                        stats.max_score_rel = max(stats.max_score_rel, float(rel.max()))
        stats.steps += 1
    chosen = inputs.candidate_pick(seed, pick_step, S, n_cand)
    f.commit(chosen, budget, window)
    committed = o.copy()
    for s in range(S):
        src = cands[int(chosen[s])]
        for name in ("K", "V", "score", "pos", "len", "next_pos"):
            getattr(committed, name)[s] = getattr(src, name)[s]
    exports = [c.export(s, kv=False) for s in range(S)]
    kernels = stats.kernels
    stats.merge(parity.check_and_adopt(committed, exports, budget, window))
    stats.kernels = kernels
    c.sync_status()
    check_guards(c, f)
    return committed, chosen, stats
