"""Lock-step parity checks of the CUDA path against the fp64 oracle.

TEST INFRASTRUCTURE ONLY (tests, smoke check).  It compares host copies of
the CUDA cache state with an ``OracleCache`` after each step:

* attention outputs: |out - ref| <= 2e-3 + 1e-2 |ref| elementwise
  (bf16 inputs, fp32 accumulation against fp64);
* importance scores of every retained row: |s - s_ref| <= 1e-4 max(|s_ref|,
  1e-6);
* retained sets: equal to the oracle's TopB-with-window set, except for
  swaps between rows whose oracle scores lie within 1e-4 relative of each
  other; between rows of exactly equal oracle score the lower position must
  be the one kept (``check_swaps``).  After a valid but different set the
  oracle adopts the CUDA set, so both continue from the same state; the
  number of adoptions is reported.
"""
from __future__ import annotations

import dataclasses

import numpy as np

from . import oracle as orc

OUT_ATOL, OUT_RTOL = 2e-3, 1e-2
SCORE_RTOL, SCORE_FLOOR = 1e-4, 1e-6
SWAP_RTOL = 1e-4


class ParityError(AssertionError):
    pass


@dataclasses.dataclass
class Stats:
    steps: int = 0
    units: int = 0
    adoptions: int = 0
    max_out_excess: float = 0.0   # max of |d| / (atol + rtol |ref|)
    max_score_rel: float = 0.0

    def merge(self, o: "Stats"):
        self.steps += o.steps
        self.units += o.units
        self.adoptions += o.adoptions
        self.max_out_excess = max(self.max_out_excess, o.max_out_excess)
        self.max_score_rel = max(self.max_score_rel, o.max_score_rel)


def check_out(out, ref, what="out") -> float:
    out = np.asarray(out, np.float64)
    ref = np.asarray(ref, np.float64)
    if out.shape != ref.shape:
        raise ParityError(f"{what}: shape {out.shape} != {ref.shape}")
    if not np.isfinite(out).all():
        raise ParityError(f"{what}: non-finite values")
    excess = np.abs(out - ref) / (OUT_ATOL + OUT_RTOL * np.abs(ref))
    worst = float(excess.max()) if excess.size else 0.0
    if worst > 1.0:
        i = np.unravel_index(int(excess.argmax()), excess.shape)
        raise ParityError(f"{what}: {out[i]} vs {ref[i]} at {i} "
                          f"(|d|={abs(out[i] - ref[i]):.3g})")
    return worst


def _window_positions(pos, W):
    if W == 0:
        return set()
    return set(np.sort(pos)[::-1][:W].tolist())


def check_swaps(kept, dropped, slack, where, what, relative):
    """A retained set that differs from the oracle's TopB is valid only if
    every dropped candidate ranks at most a near-tie above the lowest kept
    one, and exact ties follow the order of Eq. 1's TopB as read here:
    between two rows of equal oracle value the lower position is kept.

    kept, dropped: (value, position) pairs of the non-window rows.  With
    `relative`, a near-tie is value_dropped <= lowest_kept * (1 + SWAP_RTOL);
    otherwise value_dropped <= lowest_kept + slack."""
    if not kept:
        return
    lo = min(v for v, _ in kept)
    for v, p in dropped:
        bound = lo * (1.0 + SWAP_RTOL) if relative else lo + slack
        if v > bound:
            raise ParityError(
                f"{where}: evicted pos {p} ({what} {v:.9g}) while keeping a "
                f"row of {what} {lo:.9g}: not a near-tie")
    # Exact ties: a kept row may not sit above a dropped row of the same
    # value (the lower position wins).
    top = {}
    for v, p in kept:
        top[v] = max(top.get(v, -1), p)
    for v, p in dropped:
        if v in top and top[v] > p:
            raise ParityError(
                f"{where}: exact tie at {what} {v:.17g}: kept pos {top[v]} "
                f"and evicted the lower pos {p}")


def check_unit(o_pos, o_score, g_pos, g_score, B, W, evict, where=""):
    """Compare one unit.  o_*: oracle rows before eviction (all n rows);
    g_*: CUDA rows after the step.  Returns (adopted, max_score_rel)."""
    n = len(o_pos)
    if evict:
        keep = orc.select_unit(o_score, o_pos, B, W)
        want = set(o_pos[keep].tolist())
        target = min(n, B + W)
    else:
        want = set(o_pos.tolist())
        target = n
    got = set(g_pos.tolist())
    if len(g_pos) != target or len(got) != target:
        raise ParityError(f"{where}: retained {len(g_pos)} rows "
                          f"({len(got)} distinct), expected {target}")
    if not got <= set(o_pos.tolist()):
        raise ParityError(f"{where}: unknown positions {sorted(got - set(o_pos.tolist()))[:5]}")
    window = _window_positions(o_pos, W) if evict else set()
    if not window <= got:
        raise ParityError(f"{where}: window positions evicted "
                          f"{sorted(window - got)}")
    ref = dict(zip(o_pos.tolist(), o_score.tolist()))
    adopted = False
    if got != want:
        kept = [(ref[p], p) for p in got - window]
        dropped = [(ref[p], p) for p in set(o_pos.tolist()) - got]
        check_swaps(kept, dropped, 0.0, where, "score", relative=True)
        adopted = True
    # Scores of the retained rows.
    s_ref = np.array([ref[p] for p in g_pos.tolist()])
    rel = np.abs(g_score - s_ref) / np.maximum(np.abs(s_ref), SCORE_FLOOR)
    worst = float(rel.max()) if rel.size else 0.0
    if worst > SCORE_RTOL:
        i = int(rel.argmax())
        raise ParityError(f"{where}: score of pos {g_pos[i]}: {g_score[i]:.9g} "
                          f"vs {s_ref[i]:.9g} (rel {worst:.3g})")
    return adopted, worst, got


def check_and_adopt(o: orc.OracleCache, exports, B, W, evict=True,
                    layers=None) -> Stats:
    """Check every unit of layers [lb, le) after one step and make the oracle
    (which holds the pre-eviction state) adopt the CUDA retained sets.

    exports[s] is the dict returned by ``Cache.export(s, kv=False)``.
    """
    lb, le = (0, o.L) if layers is None else layers
    st = Stats(steps=1)
    keep_sets = [[[None] * o.H for _ in range(o.L)] for _ in range(o.S)]
    for s in range(o.S):
        ex = exports[s]
        for l in range(o.L):
            for h in range(o.H):
                n = o.len[s, l, h]
                if not (lb <= l < le):
                    keep_sets[s][l][h] = o.pos[s, l, h, :n].tolist()
                    continue
                g_n = ex["len"][l, h]
                adopted, worst, got = check_unit(
                    o.pos[s, l, h, :n], o.score[s, l, h, :n],
                    ex["pos"][l, h, :g_n], ex["score"][l, h, :g_n].astype(np.float64),
                    B, W, evict, where=f"seq {s} layer {l} head {h}")
                st.units += 1
                st.adoptions += int(adopted)
                st.max_score_rel = max(st.max_score_rel, worst)
                keep_sets[s][l][h] = got
    o.keep_positions(keep_sets)
    return st


# R-KV eviction (oracle/rkv.py): z differs from the oracle's by the fp32
# rounding of the normalised score (the scores carry up to 1e-4 relative)
# and of the mean cosines (about 1e-6 absolute); swaps within this bound
# are near-ties.
RKV_SWAP_ATOL = 2e-5


def check_and_adopt_rkv(o: orc.OracleCache, exports, B, W, lam,
                        layers=None) -> Stats:
    """As check_and_adopt, for one R-KV eviction after the step: every
    unit's CUDA retained set must be a TopB set of the oracle's z (window
    kept, every kept candidate ranked before every evicted one, up to
    near-ties of z), and the retained scores must match."""
    from . import rkv
    lb, le = (0, o.L) if layers is None else layers
    st = Stats(steps=1)
    sets = [[[None] * o.H for _ in range(o.L)] for _ in range(o.S)]
    for s in range(o.S):
        ex = exports[s]
        for l in range(o.L):
            for h in range(o.H):
                n = o.len[s, l, h]
                pos = o.pos[s, l, h, :n]
                if not (lb <= l < le):
                    sets[s][l][h] = pos.tolist()
                    continue
                where = f"seq {s} layer {l} head {h}"
                g_n = ex["len"][l, h]
                g_pos = ex["pos"][l, h, :g_n]
                g_score = ex["score"][l, h, :g_n].astype(np.float64)
                got = set(g_pos.tolist())
                target = min(n, B + W)
                if g_n != target or len(got) != target:
                    raise ParityError(f"{where}: retained {g_n} rows, "
                                      f"expected {target}")
                if not got <= set(pos.tolist()):
                    raise ParityError(f"{where}: unknown positions")
                adopted = False
                if n > B + W:
                    want = rkv.rkv_keep(o.K[s, l, h, :n], o.score[s, l, h, :n],
                                        pos, B, W, lam)
                    if got != want:
                        cand, z = rkv.rkv_scores(o.K[s, l, h, :n],
                                                 o.score[s, l, h, :n], pos, W,
                                                 lam)
                        if not set(pos[~cand].tolist()) <= got:
                            raise ParityError(f"{where}: window evicted")
                        zc = z[cand]
                        tol = RKV_SWAP_ATOL * float(np.abs(zc).max()) + 1e-9
                        ci = np.nonzero(cand)[0]
                        kept = [(float(z[i]), int(pos[i])) for i in ci
                                if pos[i] in got]
                        dropped = [(float(z[i]), int(pos[i])) for i in ci
                                   if pos[i] not in got]
                        check_swaps(kept, dropped, tol, where, "z",
                                    relative=False)
                        adopted = True
                ref = dict(zip(pos.tolist(), o.score[s, l, h, :n].tolist()))
                s_ref = np.array([ref[p] for p in g_pos.tolist()])
                rel = np.abs(g_score - s_ref) / np.maximum(np.abs(s_ref),
                                                           SCORE_FLOOR)
                worst = float(rel.max()) if rel.size else 0.0
                if worst > SCORE_RTOL:
                    raise ParityError(f"{where}: score rel error {worst:.3g}")
                st.units += 1
                st.adoptions += int(adopted)
                st.max_score_rel = max(st.max_score_rel, worst)
                sets[s][l][h] = got
    o.keep_positions(sets)
    return st
