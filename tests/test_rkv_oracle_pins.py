"""Pins of the R-KV oracle (oracle/rkv.py).

The paper prints no formula for R-KV, so these pins fix the library's
reading of it (stated in oracle/rkv.py) rather than the paper: torch's
cosine_similarity for the key similarities, the lambda = 1 case against the
already pinned accumulated-attention eviction, a hand-worked example, the
defining order property of the kept set, invariances, and planted mistakes
that each fail a pin.
"""
import json
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import oracle as orc
from oracle import rkv
from paper_2608_15797_gb300 import inputs


def _golden(golden_dir):
    with open(os.path.join(golden_dir, "rkv_worked.json")) as f:
        return json.load(f)


def _check_cosine(cosine_matrix):
    rng = np.random.default_rng(1)
    K = rng.standard_normal((9, 16))
    K[3] = 0.0
    want = F.cosine_similarity(torch.from_numpy(K)[:, None, :],
                               torch.from_numpy(K)[None, :, :], dim=-1,
                               eps=1e-300).numpy()
    return np.allclose(cosine_matrix(K), want, rtol=0, atol=1e-12)


def _check_golden(scores_fn, keep_fn, g):
    K = np.asarray(g["keys"], np.float64)
    s = np.asarray(g["score"], np.float64)
    p = np.asarray(g["pos"])
    for case in g["cases"]:
        cand, z = scores_fn(K, s, p, g["W"], case["lambda"])
        if not np.allclose(z[cand], case["z"], rtol=0, atol=2e-7):
            return False
        for B, want in case["keep"].items():
            if keep_fn(K, s, p, int(B), g["W"], case["lambda"]) != set(want):
                return False
    return True


def test_cosine_matrix_equals_torch():
    assert _check_cosine(rkv.cosine_matrix)


def test_golden_rkv_worked_example(golden_dir):
    assert _check_golden(rkv.rkv_scores, rkv.rkv_keep, _golden(golden_dir))


def test_lambda_one_is_accumulated_attention_topb():
    """With lambda = 1, z is the normalised accumulated score, so the kept
    set is the TopB of Eq. 1 that OracleCache.evict computes."""
    w = inputs.WORKLOADS["tiny"]
    o = orc.OracleCache(1, w.n_layers, w.n_kv_heads, w.group, w.head_dim,
                        cap=64)
    k, v = inputs.prompt(w, 4, 0, 40)
    o.load(0, k, v)
    for t in range(3):
        o.step(*inputs.step_inputs(w, 4, t, 1), evict=False)
    ref = o.copy()
    ref.evict(w.budget, w.window)
    o2 = o.copy()
    rkv.evict_rkv(o2, w.budget, w.window, 1.0)
    for l in range(o.L):
        for h in range(o.H):
            assert set(ref.pos[0, l, h, :ref.len[0, l, h]].tolist()) == \
                set(o2.pos[0, l, h, :o2.len[0, l, h]].tolist())


def test_kept_set_order_property_and_invariances():
    rng = np.random.default_rng(7)
    for trial in range(30):
        n = int(rng.integers(3, 40))
        d = int(rng.integers(2, 9))
        K = rng.standard_normal((n, d))
        K[rng.integers(0, n)] = K[rng.integers(0, n)]  # a duplicate key
        s = rng.random(n)
        p = rng.permutation(1000)[:n]
        W = int(rng.integers(0, 4))
        B = int(rng.integers(0, max(1, n - W)))
        lam = float(rng.choice([0.0, 0.1, 0.5, 1.0]))
        cand, z = rkv.rkv_scores(K, s, p, W, lam)
        keep = rkv.rkv_keep(K, s, p, B, W, lam)
        if n <= B + W:
            assert keep == set(p.tolist())
            continue
        assert len(keep) == B + W
        # the W largest positions are kept
        assert set(np.sort(p)[n - W:].tolist()) <= keep if W else True
        # every kept candidate ranks before every evicted one
        kc = [i for i in range(n) if cand[i] and p[i] in keep]
        ec = [i for i in range(n) if cand[i] and p[i] not in keep]
        for i in kc:
            for j in ec:
                assert (z[i], -p[i]) > (z[j], -p[j])
        # R and I each sum to one over the candidates (lambda = 0 / 1)
        _, z0 = rkv.rkv_scores(K, s, p, W, 0.0)
        _, z1 = rkv.rkv_scores(K, s, p, W, 1.0)
        assert abs(z0[cand].sum() + 1.0) < 1e-12
        assert abs(z1[cand].sum() - 1.0) < 1e-12
        # positive scalings of keys and of all scores change nothing
        scale = rng.uniform(0.1, 10.0, size=(n, 1))
        _, zs = rkv.rkv_scores(K * scale, s * 3.7, p, W, lam)
        assert np.allclose(zs[cand], z[cand], rtol=0, atol=1e-12)


# --------------------------------------------------------------------------
# Planted mistakes: copies of the oracle with one plausible error each
# --------------------------------------------------------------------------

def _scores_variant(kind):
    def f(K, score, pos, W, lam):
        K = np.asarray(K, np.float64)
        score = np.asarray(score, np.float64)
        pos = np.asarray(pos)
        n = len(pos)
        order = np.argsort(-pos, kind="stable")
        cand = np.ones(n, bool)
        cand[order[:min(W, n)]] = False
        z = np.full(n, np.nan)
        C = rkv.cosine_matrix(K)
        if kind == "self_included":
            r = C.sum(axis=1) / n
        elif kind == "candidates_only":
            Cc = C[np.ix_(cand, cand)]
            r = np.zeros(n)
            r[cand] = (Cc.sum(axis=1) - np.diag(Cc)) / max(1, cand.sum() - 1)
        else:
            r = (C.sum(axis=1) - np.diag(C)) / (n - 1)
        rc = r[cand]
        if kind == "no_softmax":
            R = rc / rc.sum() if rc.sum() else rc
        else:
            R = np.exp(rc - rc.max())
            R /= R.sum()
        I = score[cand] / score[cand].sum()
        if kind == "plus":
            z[cand] = lam * I + (1 - lam) * R
        elif kind == "swapped":
            z[cand] = (1 - lam) * I - lam * R
        else:
            z[cand] = lam * I - (1 - lam) * R
        return cand, z
    return f


def _keep_with(scores_fn, tie_high=False):
    def f(K, score, pos, B, W, lam):
        pos = np.asarray(pos)
        n = len(pos)
        if n <= B + W:
            return set(pos.tolist())
        cand, z = scores_fn(K, score, pos, W, lam)
        idx = np.nonzero(cand)[0].tolist()
        sign = 1 if tie_high else -1
        ranked = sorted(idx, key=lambda i: (-z[i], -sign * pos[i]))
        return set(pos[~cand].tolist()) | set(pos[ranked[:B]].tolist())
    return f


def test_planted_mistakes_are_caught(golden_dir):
    g = _golden(golden_dir)
    for kind in ("self_included", "candidates_only", "no_softmax", "plus",
                 "swapped"):
        fn = _scores_variant(kind)
        assert not _check_golden(fn, _keep_with(fn), g), kind
    # a tie broken toward the higher position: two identical candidates
    K = np.array([[1.0, 0.0], [1.0, 0.0], [0.0, 1.0]])
    s = np.array([0.3, 0.3, 0.4])
    p = np.array([5, 6, 7])
    good = rkv.rkv_keep(K, s, p, 1, 1, 0.1)
    bad = _keep_with(rkv.rkv_scores, tie_high=True)(K, s, p, 1, 1, 0.1)
    assert good == {5, 7} and bad != good
