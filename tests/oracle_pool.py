"""The fp64 oracle of a candidate step (Sec. 2.2 Eq. 2; App. C best-of-N)
spread over spawned worker processes, for full-length lock-step runs.

TEST INFRASTRUCTURE ONLY.  Every candidate is an independent copy of the
committed parent (the paper forks by copying the live KV slots), and layers
never interact, so worker (k, part) holds candidate k's oracle state for one
contiguous range of layers.  Per candidate token each worker draws its
candidate's inputs from ``paper_2608_15797_gb300.inputs`` (the same seeded
draws the CUDA side uploads), steps its oracle, and compares the CUDA
candidate's outputs and scores, which the driving process leaves in shared
memory.  At the commit, the workers of the chosen candidate check the
CUDA parent against their state (``oracle.parity.check_and_adopt``: TopB
with ties at the lower position, near-ties adopted) and publish the adopted
state as the next parent.

Workers are started with the ``spawn`` method, so no worker inherits the
driving process's CUDA context.  Nothing here imports the CUDA binding.
"""
from __future__ import annotations

import multiprocessing as mp
import os
import traceback
from multiprocessing import shared_memory

import numpy as np

from oracle import oracle as orc
from oracle import parity
from paper_2608_15797_gb300 import inputs

_SEG_DTYPES = {"f4": np.float32, "f8": np.float64, "i4": np.int32}


class _Shared:
    """Named numpy arrays over one shared-memory block."""

    def __init__(self, spec, name=None):
        self.spec = spec            # [(key, shape, dtype code)]
        offs, off = {}, 0
        for key, shape, dt in spec:
            offs[key] = off
            off += int(np.prod(shape)) * np.dtype(_SEG_DTYPES[dt]).itemsize
            off = (off + 63) // 64 * 64
        self.shm = (shared_memory.SharedMemory(create=True, size=max(off, 64))
                    if name is None else shared_memory.SharedMemory(name=name))
        self.a = {key: np.ndarray(shape, _SEG_DTYPES[dt], self.shm.buf,
                                  offs[key]) for key, shape, dt in spec}

    def close(self, unlink=False):
        self.a = {}
        self.shm.close()
        if unlink:
            self.shm.unlink()


def _layer_ranges(L, parts):
    b = np.linspace(0, L, parts + 1).round().astype(int)
    return [(int(b[i]), int(b[i + 1])) for i in range(parts)]


def _spec(w, N, cap_p, tcap):
    L, H, G, d = w.n_layers, w.n_kv_heads, w.group, w.head_dim
    return [
        ("q", (N, L, H * G, d), "f4"), ("kn", (N, L, H, d), "f4"),
        ("vn", (N, L, H, d), "f4"),
        ("out", (N, L, H * G, d), "f4"),                  # CUDA outputs
        ("pscore", (N, L, H, cap_p), "f4"),               # CUDA prefix scores
        ("tscore", (N, L, H, tcap), "f4"), ("tpos", (N, L, H, tcap), "i4"),
        ("tlen", (N, L, H), "i4"),
        ("gpos", (L, H, cap_p), "i4"), ("glen", (L, H), "i4"),  # CUDA parent
        ("gscore", (L, H, cap_p), "f4"),
        # oracle parent (compacted, cap_p rows)
        ("K", (L, H, cap_p, d), "f8"), ("V", (L, H, cap_p, d), "f8"),
        ("score", (L, H, cap_p), "f8"), ("pos", (L, H, cap_p), "i4"),
        ("len", (L, H), "i4"), ("next_pos", (L, H), "i4"),
    ]


def _worker(conn, shm_name, w, N, cap_p, tcap, seed, k, lb, le):
    sh = _Shared(_spec(w, N, cap_p, tcap), shm_name)
    a = sh.a
    H, G, d = w.n_kv_heads, w.group, w.head_dim
    nl = le - lb
    cand = None
    ref = None
    try:
        while True:
            msg = conn.recv()
            cmd = msg[0]
            if cmd == "stop":
                break
            try:
                if cmd == "fork":
                    cand = orc.OracleCache(1, nl, H, G, d, cap_p + tcap)
                    cand.K[0, :, :, :cap_p] = a["K"][lb:le]
                    cand.V[0, :, :, :cap_p] = a["V"][lb:le]
                    cand.score[0, :, :, :cap_p] = a["score"][lb:le]
                    cand.pos[0, :, :, :cap_p] = a["pos"][lb:le]
                    cand.len[0] = a["len"][lb:le]
                    cand.next_pos[0] = a["next_pos"][lb:le]
                    conn.send(("ok",))
                elif cmd == "token":
                    step = msg[1]
                    q, kn, vn = inputs.step_inputs(w, seed, step, 1, cand=k + 1)
                    if lb == 0:   # one worker per candidate publishes them
                        a["q"][k] = q[0]
                        a["kn"][k] = kn[0]
                        a["vn"][k] = vn[0]
                    conn.send(("in",))
                    ref = cand.step(q[:, lb:le], kn[:, lb:le], vn[:, lb:le],
                                    evict=False)
                elif cmd == "check":
                    st = parity.Stats(steps=1)
                    st.max_out_excess = parity.check_out(
                        a["out"][k, lb:le], ref[0], what=f"candidate {k} out "
                        f"at token {msg[1]} (layers {lb}-{le})")
                    st.max_score_rel = _check_scores(a, cand, k, lb, le, msg[1])
                    conn.send(("ok", st))
                elif cmd == "commit":
                    chosen, B, W = msg[1], msg[2], msg[3]
                    st = parity.Stats()
                    if chosen == k:
                        ex = {"pos": a["gpos"][lb:le], "score": a["gscore"][lb:le],
                              "len": a["glen"][lb:le]}
                        st = parity.check_and_adopt(cand, [ex], B, W)
                        n = int(cand.len.max())
                        a["K"][lb:le] = 0.0
                        a["V"][lb:le] = 0.0
                        a["K"][lb:le, :, :n] = cand.K[0, :, :, :n]
                        a["V"][lb:le, :, :n] = cand.V[0, :, :, :n]
                        a["score"][lb:le] = 0.0
                        a["score"][lb:le, :, :n] = cand.score[0, :, :, :n]
                        a["pos"][lb:le] = 0
                        a["pos"][lb:le, :, :n] = cand.pos[0, :, :, :n]
                        a["len"][lb:le] = cand.len[0]
                        a["next_pos"][lb:le] = cand.next_pos[0]
                    conn.send(("ok", st))
                else:
                    raise ValueError(f"unknown command {cmd}")
            except Exception:   # reported to the driving process
                conn.send(("err", traceback.format_exc()))
    finally:
        sh.close()


def _check_scores(a, cand, k, lb, le, token):
    """Every row's score of candidate k (parent rows and tail rows), matched
    by position, within 1e-4 relative; the row sets must agree exactly."""
    nl = le - lb
    big = np.iinfo(np.int32).max
    glen = a["glen"][lb:le]
    tlen = a["tlen"][k, lb:le]
    cap_p, tcap = a["gpos"].shape[-1], a["tpos"].shape[-1]
    slot_p = np.arange(cap_p)[None, None, :] < glen[..., None]
    slot_t = np.arange(tcap)[None, None, :] < tlen[..., None]
    gp = np.concatenate([np.where(slot_p, a["gpos"][lb:le], big),
                         np.where(slot_t, a["tpos"][k, lb:le], big)], axis=-1)
    gs = np.concatenate([np.where(slot_p, a["pscore"][k, lb:le], 0.0),
                         np.where(slot_t, a["tscore"][k, lb:le], 0.0)], axis=-1)
    o_n = cand.len[0]
    width = gp.shape[-1]
    op = np.full((nl, cand.H, width), big, np.int64)
    osc = np.zeros((nl, cand.H, width), np.float64)
    m = min(width, cand.cap)
    live = np.arange(m)[None, None, :] < o_n[..., None]
    op[..., :m] = np.where(live, cand.pos[0, :, :, :m], big)
    osc[..., :m] = np.where(live, cand.score[0, :, :, :m], 0.0)
    go = np.argsort(gp, axis=-1, kind="stable")
    oo = np.argsort(op, axis=-1, kind="stable")
    gp, gs = (np.take_along_axis(x, go, axis=-1) for x in (gp, gs))
    op, osc = (np.take_along_axis(x, oo, axis=-1) for x in (op, osc))
    if (gp != op).any() or ((glen + tlen) != o_n).any():
        bad = np.argwhere((gp != op).any(axis=-1))[:1]
        raise parity.ParityError(f"candidate {k} token {token}: row sets "
                                 f"differ (layer {lb + int(bad[0][0]) if len(bad) else '?'})")
    livem = gp != big
    rel = np.abs(gs - osc) / np.maximum(np.abs(osc), parity.SCORE_FLOOR)
    rel = np.where(livem, rel, 0.0)
    worst = float(rel.max()) if rel.size else 0.0
    if worst > parity.SCORE_RTOL:
        raise parity.ParityError(f"candidate {k} token {token}: score rel "
                                 f"{worst:.3g}")
    return worst


class CandidateOraclePool:
    """Oracle workers for N candidates of one sequence (S = 1) of workload
    w: N x parts processes, `parts` layer ranges per candidate."""

    def __init__(self, w, N, cap_p, tcap, seed, parts=None):
        self.w, self.N, self.cap_p, self.tcap = w, N, cap_p, tcap
        if parts is None:
            parts = max(1, min(4, (os.cpu_count() or 1) // N))
        self.ranges = _layer_ranges(w.n_layers, parts)
        self.sh = _Shared(_spec(w, N, cap_p, tcap))
        ctx = mp.get_context("spawn")
        self.procs, self.conns = [], []
        for k in range(N):
            for lb, le in self.ranges:
                a, b = ctx.Pipe()
                p = ctx.Process(target=_worker, args=(
                    b, self.sh.shm.name, w, N, cap_p, tcap, seed, k, lb, le),
                    daemon=True)
                p.start()
                self.procs.append(p)
                self.conns.append((k, lb, a))

    @property
    def a(self):
        return self.sh.a

    def _gather(self, which=None):
        res = []
        for k, lb, c in self.conns:
            if which is not None and (k, lb) not in which:
                continue
            r = c.recv()
            if r[0] == "err":
                raise parity.ParityError(f"oracle worker ({k}, {lb}):\n{r[1]}")
            res.append(r)
        return res

    def _send(self, msg):
        for _, _, c in self.conns:
            c.send(msg)

    def set_parent(self, o: orc.OracleCache):
        """The oracle parent (sequence 0 of `o`, at most cap_p live rows)."""
        n = int(o.len.max())
        if n > self.cap_p:
            raise ValueError("parent longer than the pool's capacity")
        a = self.a
        for key in ("K", "V", "score", "pos"):
            a[key][...] = 0
            a[key][:, :, :n] = getattr(o, key)[0, :, :, :n]
        a["len"][...] = o.len[0]
        a["next_pos"][...] = o.next_pos[0]

    def fork(self):
        self._send(("fork",))
        self._gather()

    def token_inputs(self, step):
        """Ask every worker for its candidate's token; returns once the
        inputs (a["q"], a["kn"], a["vn"], [N][L][..][d]) are published.  The
        workers then step their oracles."""
        self._send(("token", step))
        self._gather()

    def check(self, token) -> parity.Stats:
        """Compare after the CUDA side has filled out, pscore, tscore,
        tpos, tlen (and gpos / glen for the parent rows)."""
        self._send(("check", token))
        st = parity.Stats()
        for r in self._gather():
            st.max_out_excess = max(st.max_out_excess, r[1].max_out_excess)
            st.max_score_rel = max(st.max_score_rel, r[1].max_score_rel)
        st.steps = 1
        return st

    def commit(self, chosen, B, W) -> parity.Stats:
        """Check the CUDA parent (gpos, gscore, glen) against the chosen
        candidate cut to B + W, and make the adopted state the parent."""
        self._send(("commit", int(chosen), B, W))
        st = parity.Stats()
        for r in self._gather():
            st.merge(r[1])
        st.steps = 1
        return st

    def close(self):
        for _, _, c in self.conns:
            try:
                c.send(("stop",))
            except (BrokenPipeError, OSError):
                pass
        for p in self.procs:
            p.join(timeout=10)
            if p.is_alive():
                p.terminate()
        self.sh.close(unlink=True)
