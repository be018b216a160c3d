"""fp64 oracle of the redundancy-aware eviction score (R-KV) used by the
paper's base model.

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` leg of ``bench.py`` may use this module; the product path
never imports it.  It shares no code with the CUDA library.

PARITY UNPINNED against the paper: App. C says only that R-KV scores the
cached tokens "with a mix of query-attention importance and key redundancy
(cosine similarity)", keeps the top B plus a recent window, and uses a mix
weight lambda = 0.1; App. D adds that an eviction makes a key-similarity
pass and a top-k selection over the B' physical tokens.  No formula is
printed.  The reading implemented here, for one (sequence, layer, KV head)
unit with live rows L (n = |L|), window rows Wset (the W largest positions)
and candidates C = L minus Wset:

1. cos(k_i, k_j) = k_i . k_j / (|k_i| |k_j|), and 0 when either norm is 0.
2. redundancy r_i = (1 / (n - 1)) sum over j in L, j != i of cos(k_i, k_j).
3. R_i = softmax over C of r (so sum over C of R = 1).
4. importance I_i = s_i / sum over C of s (the accumulated attention score
   of Sec. 2.1, the library's importance), 0 for all if that sum is 0.
5. z_i = lambda * I_i - (1 - lambda) * R_i.
6. Keep Wset and the B candidates ranked first by (z descending, position
   ascending); evict the rest.

With lambda = 1 this is the accumulated-attention TopB of Eq. 1.  The pins
(``tests/test_rkv_oracle_pins.py``) fix the reading's arithmetic: torch's
cosine_similarity, the lambda = 1 reduction to ``OracleCache.evict``, a
hand-worked example (``tests/golden/rkv_worked.json``), invariances and
planted mistakes.
"""
from __future__ import annotations

import numpy as np


def cosine_matrix(K) -> np.ndarray:
    """n x n cosine similarities of the rows of K (0 where a norm is 0)."""
    K = np.asarray(K, dtype=np.float64)
    nrm = np.sqrt((K * K).sum(axis=1))
    G = K @ K.T
    den = np.outer(nrm, nrm)
    with np.errstate(divide="ignore", invalid="ignore"):
        return np.where(den > 0, G / np.where(den > 0, den, 1.0), 0.0)


def rkv_scores(K, score, pos, W, lam):
    """(cand, z): the candidate mask of the live rows and z for every live
    row (NaN outside the candidates), steps 1-5 above."""
    K = np.asarray(K, dtype=np.float64)
    score = np.asarray(score, dtype=np.float64)
    pos = np.asarray(pos)
    n = len(pos)
    order = np.argsort(-pos, kind="stable")
    cand = np.ones(n, bool)
    cand[order[:min(W, n)]] = False
    z = np.full(n, np.nan)
    if not cand.any():
        return cand, z
    C = cosine_matrix(K)
    off = C.sum(axis=1) - np.diag(C)
    r = off / (n - 1) if n > 1 else np.zeros(n)
    rc = r[cand]
    e = np.exp(rc - rc.max())
    R = e / e.sum()
    tot = score[cand].sum()
    I = score[cand] / tot if tot > 0 else np.zeros(cand.sum())
    z[cand] = lam * I - (1.0 - lam) * R
    return cand, z


def rkv_keep(K, score, pos, B, W, lam):
    """Positions kept by one R-KV eviction (step 6); all if n <= B + W."""
    pos = np.asarray(pos)
    n = len(pos)
    if n <= B + W:
        return set(pos.tolist())
    cand, z = rkv_scores(K, score, pos, W, lam)
    idx = np.nonzero(cand)[0]
    ranked = sorted(idx.tolist(), key=lambda i: (-z[i], pos[i]))
    keep = set(pos[~cand].tolist()) | set(pos[ranked[:B]].tolist())
    return keep


def evict_rkv(o, B, W, lam, layer_begin=None, layer_end=None):
    """R-KV eviction of every unit of an ``OracleCache`` (layers [lb, le))."""
    lb = 0 if layer_begin is None else layer_begin
    le = o.L if layer_end is None else layer_end
    sets = [[[None] * o.H for _ in range(o.L)] for _ in range(o.S)]
    for s in range(o.S):
        for l in range(o.L):
            for h in range(o.H):
                n = o.len[s, l, h]
                pos = o.pos[s, l, h, :n]
                if lb <= l < le:
                    sets[s][l][h] = rkv_keep(o.K[s, l, h, :n],
                                             o.score[s, l, h, :n], pos, B, W,
                                             lam)
                else:
                    sets[s][l][h] = set(pos.tolist())
    o.keep_positions(sets)
