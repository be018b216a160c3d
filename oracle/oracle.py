"""fp64 CPU oracle of the evicted-KV decode step (KV-Rescue, arXiv 2608.15797).

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` leg of ``bench.py`` may use this module; the product path
(the ``paper_2608_15797_gb300`` package) never imports it.  It shares no code
with the CUDA library.

The arithmetic lives in ``kvr_oracle.c`` (plain C, double precision); this
module compiles it with gcc, marshals numpy arrays to it and keeps the
per-unit cache state:

* ``OracleCache.step``   -- Eq. 1 (Sec. 2.1): append the step's key/value,
  attend over every live row, add the mean over the G query heads of the
  attention probability to each row's accumulated-attention score, and, when
  the live length exceeds B' = B + W (App. D), keep the W most recent rows
  (Sec. 4.1 window) plus the B best-scored others (ties: lower position).
* ``OracleCache.fork``   -- App. C, "Best-of-(N+N)": a candidate is a
  physical copy of the parent's live rows.
* ``OracleCache.evict``  -- TopB of Eq. 1 on the current state.

Parity pins of every function are in ``tests/test_oracle_pins.py``.
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "kvr_oracle.c")
_LIB_PATH = os.path.join(_HERE, "libkvr_oracle.so")
_lib = None


def build(force: bool = False) -> str:
    """Compile kvr_oracle.c into a shared library next to it (gcc, IEEE fp)."""
    if force or not os.path.exists(_LIB_PATH) or (
            os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC)):
        tmp = _LIB_PATH + ".tmp%d" % os.getpid()
        subprocess.run(["gcc", "-O2", "-std=c11", "-shared", "-fPIC",
                        "-fno-fast-math", "-o", tmp, _SRC, "-lm"], check=True)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        P = ctypes.c_void_p
        I = ctypes.c_int
        D = ctypes.c_double
        lib.kvro_attend_unit.argtypes = [I, I, I, D, P, P, P, P, P]
        lib.kvro_select_unit.argtypes = [I, P, P, I, I, P]
        lib.kvro_step.argtypes = [I, I, I, I, D, P, P, P, P, P, P, P, P, P,
                                  I, I, I, P]
        lib.kvro_evict.argtypes = [I, I, I, P, P, P, P, P, I, I]
        lib.kvro_keep_rows.argtypes = [I, I, I, P, P, P, P, P, P]
        for f in (lib.kvro_attend_unit, lib.kvro_select_unit, lib.kvro_step,
                  lib.kvro_evict, lib.kvro_keep_rows):
            f.restype = ctypes.c_int
        _lib = lib
    return _lib


def _p(a: np.ndarray):
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data_as(ctypes.c_void_p)


def attend_unit(K, V, q, scale=None):
    """Eq. 1 Attn for one KV head: returns (out [G,d], prob [G,n])."""
    K = np.ascontiguousarray(K, dtype=np.float64)
    V = np.ascontiguousarray(V, dtype=np.float64)
    q = np.ascontiguousarray(q, dtype=np.float64)
    n, d = K.shape
    G = q.shape[0]
    scale = 1.0 / math.sqrt(d) if scale is None else float(scale)
    out = np.zeros((G, d), np.float64)
    prob = np.zeros((G, n), np.float64)
    rc = _load().kvro_attend_unit(n, d, G, scale, _p(K), _p(V), _p(q),
                                  _p(out), _p(prob))
    if rc:
        raise ValueError("kvro_attend_unit failed")
    return out, prob


def select_unit(score, pos, B, W):
    """TopB with protected window: boolean keep mask over the n rows."""
    score = np.ascontiguousarray(score, dtype=np.float64)
    pos = np.ascontiguousarray(pos, dtype=np.int32)
    keep = np.zeros(score.shape[0], np.uint8)
    rc = _load().kvro_select_unit(score.shape[0], _p(score), _p(pos), int(B),
                                  int(W), _p(keep))
    if rc < 0:
        raise ValueError("kvro_select_unit failed")
    return keep.astype(bool)


class OracleCache:
    """Per-unit fp64 cache state: S sequences x L layers x H KV heads.

    Rows of a unit live compacted in slots [0, len) in entry order.
    """

    def __init__(self, S, L, H, G, d, cap, scale=None):
        self.S, self.L, self.H, self.G, self.d, self.cap = S, L, H, G, d, cap
        self.scale = 1.0 / math.sqrt(d) if scale is None else float(scale)
        self.K = np.zeros((S, L, H, cap, d), np.float64)
        self.V = np.zeros((S, L, H, cap, d), np.float64)
        self.score = np.zeros((S, L, H, cap), np.float64)
        self.pos = np.zeros((S, L, H, cap), np.int32)
        self.len = np.zeros((S, L, H), np.int32)
        self.next_pos = np.zeros((S, L, H), np.int32)

    @property
    def n_units(self):
        return self.S * self.L * self.H

    def copy(self) -> "OracleCache":
        c = OracleCache.__new__(OracleCache)
        c.__dict__.update({k: (v.copy() if isinstance(v, np.ndarray) else v)
                           for k, v in self.__dict__.items()})
        return c

    def resized(self, cap) -> "OracleCache":
        """The same state in a cache of capacity `cap` (at least every live
        length); rows are compacted, so only slots [0, cap) are kept.  Data
        movement only: lets long runs fork small copies after the first
        eviction."""
        if cap < int(self.len.max(initial=0)):
            raise ValueError("capacity below a live length")
        c = OracleCache(self.S, self.L, self.H, self.G, self.d, cap, self.scale)
        k = min(cap, self.cap)
        c.K[..., :k, :] = self.K[..., :k, :]
        c.V[..., :k, :] = self.V[..., :k, :]
        c.score[..., :k] = self.score[..., :k]
        c.pos[..., :k] = self.pos[..., :k]
        c.len[...] = self.len
        c.next_pos[...] = self.next_pos
        return c

    def load(self, seq, k, v, first_pos=0, scores=None):
        """Prompt rows [L][H][n][d] with positions first_pos.. and score 0."""
        n = k.shape[2]
        if n > self.cap:
            raise ValueError("prompt longer than capacity")
        self.K[seq, :, :, :n] = k
        self.V[seq, :, :, :n] = v
        self.score[seq, :, :, :n] = 0.0 if scores is None else scores
        self.pos[seq, :, :, :n] = first_pos + np.arange(n, dtype=np.int32)
        self.len[seq] = n
        self.next_pos[seq] = first_pos + n

    def _layers(self, layer_begin, layer_end):
        lb = 0 if layer_begin is None else layer_begin
        le = self.L if layer_end is None else layer_end
        return lb, le

    def step(self, q, k_new, v_new, B=0, W=0, evict=True, layer_begin=None,
             layer_end=None):
        """One decode step over layers [lb, le) of every sequence.

        q: [S][nl][H*G][d]; k_new, v_new: [S][nl][H][d].  Returns out
        [S][nl][H*G][d].  With evict, each unit is cut back to B + W rows.
        """
        lb, le = self._layers(layer_begin, layer_end)
        nl = le - lb
        S, H, G, d, cap = self.S, self.H, self.G, self.d, self.cap
        sub = [np.ascontiguousarray(a[:, lb:le]) for a in
               (self.K, self.V, self.score, self.pos, self.len, self.next_pos)]
        K, V, sc, pos, ln, npos = sub
        qq = np.ascontiguousarray(q, dtype=np.float64).reshape(S, nl, H, G, d)
        kn = np.ascontiguousarray(k_new, dtype=np.float64)
        vn = np.ascontiguousarray(v_new, dtype=np.float64)
        out = np.zeros((S, nl, H, G, d), np.float64)
        newp = np.ascontiguousarray(npos)
        rc = _load().kvro_step(S * nl * H, cap, d, G, self.scale, _p(K), _p(V),
                               _p(sc), _p(pos), _p(ln), _p(qq), _p(kn),
                               _p(vn), _p(newp), int(B), int(W),
                               1 if evict else 0, _p(out))
        if rc:
            raise ValueError("kvro_step: a unit is full")
        npos = npos + 1
        for arr, new in zip((self.K, self.V, self.score, self.pos, self.len,
                             self.next_pos), (K, V, sc, pos, ln, npos)):
            arr[:, lb:le] = new
        return out.reshape(S, nl, H * G, d)

    def absorb(self, q, k_new, v_new, B=0, W=0, evict=True, layer_begin=None,
               layer_end=None):
        """c tokens of every sequence in one call: the reading of Alg. 1's
        single forward pass of the base model over an accepted helper step
        (and of a prompt prefill whose attention seeds the scores).  Token j
        is appended and attends every live row and the chunk's rows 0..j
        (causal), adding its head-mean probabilities to the scores of every
        row it attends -- c decode steps with the eviction to B + W applied
        once, after the last.

        q: [S][nl][c][H*G][d]; k_new, v_new: [S][nl][c][H][d].  Returns out
        [S][nl][c][H*G][d].
        """
        lb, le = self._layers(layer_begin, layer_end)
        c = q.shape[2]
        outs = [self.step(q[:, :, j], k_new[:, :, j], v_new[:, :, j],
                          evict=False, layer_begin=lb, layer_end=le)
                for j in range(c)]
        if evict:
            self.evict(B, W, lb, le)
        return np.stack(outs, axis=2)

    def evict(self, B, W, layer_begin=None, layer_end=None):
        lb, le = self._layers(layer_begin, layer_end)
        sub = [np.ascontiguousarray(a[:, lb:le]) for a in
               (self.K, self.V, self.score, self.pos, self.len)]
        K, V, sc, pos, ln = sub
        n_units = self.S * (le - lb) * self.H
        _load().kvro_evict(n_units, self.cap, self.d, _p(K), _p(V), _p(sc),
                           _p(pos), _p(ln), int(B), int(W))
        for arr, new in zip((self.K, self.V, self.score, self.pos, self.len),
                            (K, V, sc, pos, ln)):
            arr[:, lb:le] = new

    def keep_positions(self, keep_pos_sets):
        """Adopt a retained set per unit: keep_pos_sets[s][l][h] is an iterable
        of positions; rows at other positions are dropped (stable)."""
        keep = np.zeros((self.S, self.L, self.H, self.cap), np.uint8)
        for s in range(self.S):
            for l in range(self.L):
                for h in range(self.H):
                    n = self.len[s, l, h]
                    want = np.asarray(sorted(keep_pos_sets[s][l][h]),
                                      dtype=np.int32)
                    keep[s, l, h, :n] = np.isin(self.pos[s, l, h, :n], want)
        _load().kvro_keep_rows(self.n_units, self.cap, self.d, _p(self.K),
                               _p(self.V), _p(self.score), _p(self.pos),
                               _p(self.len), _p(keep))

    def copy_sequences(self, src: "OracleCache", src_seqs, dst_seqs):
        """App. C "Best-of-(N+N)": a candidate is forked by physically copying
        the live (post-eviction) KV slots of the accepted sequence, and the
        chosen candidate becomes the persistent sequence.  Sequence
        dst_seqs[i] of this cache takes the whole state (rows, scores,
        positions, length, position counter) of sequence src_seqs[i] of
        `src`, every layer and KV head.  Data movement only."""
        if (src.L, src.H, src.d) != (self.L, self.H, self.d):
            raise ValueError("geometry differs")
        moved = [(int(a), int(b)) for a, b in zip(src_seqs, dst_seqs)]
        for a, b in moved:
            n = int(src.len[a].max(initial=0))
            if n > self.cap:
                raise ValueError("a live length exceeds the capacity")
        snap = {a: (src.K[a, :, :, :min(src.cap, self.cap)].copy(),
                    src.V[a, :, :, :min(src.cap, self.cap)].copy(),
                    src.score[a, :, :, :min(src.cap, self.cap)].copy(),
                    src.pos[a, :, :, :min(src.cap, self.cap)].copy(),
                    src.len[a].copy(), src.next_pos[a].copy())
                for a, _ in moved}
        for a, b in moved:
            K, V, sc, ps, ln, nx = snap[a]
            k = K.shape[2]
            self.K[b] = 0.0
            self.V[b] = 0.0
            self.score[b] = 0.0
            self.pos[b] = 0
            self.K[b, :, :, :k] = K
            self.V[b, :, :, :k] = V
            self.score[b, :, :, :k] = sc
            self.pos[b, :, :, :k] = ps
            self.len[b] = ln
            self.next_pos[b] = nx

    def fork(self, n_cand):
        """App. C "Best-of-(N+N)": N physical copies of the live state."""
        return [self.copy() for _ in range(n_cand)]

    def unit_rows(self, s, l, h):
        """(pos, score, K, V) of the live rows of one unit, sorted by pos."""
        n = self.len[s, l, h]
        order = np.argsort(self.pos[s, l, h, :n], kind="stable")
        return (self.pos[s, l, h, :n][order], self.score[s, l, h, :n][order],
                self.K[s, l, h, :n][order], self.V[s, l, h, :n][order])
