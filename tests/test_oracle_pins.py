"""Pins of the fp64 oracle against what the paper and the mathematics fix.

Every function of ``oracle/`` is checked here against something other than
itself: hand-worked examples (tests/golden), a library routine
(torch's scaled_dot_product_attention) in the special case where eviction
never fires, closed forms (zero query), invariants (probabilities sum to one,
score conservation, retained size and window), and brute force by subset
enumeration on tiny inputs.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import oracle as orc
from paper_2608_15797_gb300 import inputs


def _load_json(golden_dir, name):
    with open(os.path.join(golden_dir, name)) as f:
        return json.load(f)


# --------------------------------------------------------------------------
# Hand-worked examples (Eq. 1 Attn, accumulated attention, TopB + window)
# --------------------------------------------------------------------------

def test_golden_attention_worked_example(golden_dir):
    g = _load_json(golden_dir, "attend_worked.json")
    K, V, q = (np.array(g[k], np.float64) for k in ("K", "V", "q"))
    out, prob = orc.attend_unit(K, V, q)
    np.testing.assert_allclose(prob, np.array(g["prob"]), atol=1e-12, rtol=0)
    np.testing.assert_allclose(out, np.array(g["out"]), atol=1e-12, rtol=0)
    # The same rows driven through a decode step: rows 0-1 as the prompt, row 2
    # appended by the step; the step's score increment is the mean over heads.
    c = orc.OracleCache(1, 1, 1, g["G"], g["d"], cap=4)
    c.load(0, K[None, None, :2], V[None, None, :2])
    o = c.step(q[None, None], K[2][None, None, None], V[2][None, None, None],
               evict=False)
    np.testing.assert_allclose(o[0, 0], np.array(g["out"]), atol=1e-12, rtol=0)
    np.testing.assert_allclose(c.score[0, 0, 0, :3], g["score_increment"],
                               atol=1e-12, rtol=0)


def test_golden_eviction_worked_example(golden_dir):
    g = _load_json(golden_dir, "evict_worked.json")
    pos = np.array(g["pos"], np.int32)
    score = np.array(g["score"], np.float64)
    rng = np.random.default_rng(0)
    for case in g["cases"]:
        for trial in range(4):  # slot order must not matter
            perm = np.arange(len(pos)) if trial == 0 else rng.permutation(len(pos))
            keep = orc.select_unit(score[perm], pos[perm], case["B"], case["W"])
            assert sorted(pos[perm][keep].tolist()) == case["kept_pos"], case


# --------------------------------------------------------------------------
# Library special case: with B >= length eviction never fires and the step is
# plain grouped-query decode attention over the whole history.
# --------------------------------------------------------------------------

def _sdpa_gqa(q, K, V, G):
    """q [Hq, d], K/V [H, n, d] -> [Hq, d] via torch SDPA in float64."""
    Kq = torch.from_numpy(K).repeat_interleave(G, dim=0)
    Vq = torch.from_numpy(V).repeat_interleave(G, dim=0)
    o = F.scaled_dot_product_attention(torch.from_numpy(q)[:, None, :], Kq, Vq)
    return o[:, 0, :].numpy()


def test_no_eviction_equals_full_attention_sdpa():
    S, L, H, G, d, P, T = 2, 2, 2, 3, 16, 11, 9
    w = inputs.Workload("t", L, H, G, d, "f32", 1 << 20, 4, P, T, n_seq=S)
    c = orc.OracleCache(S, L, H, G, d, cap=P + T)
    hist_k = np.zeros((S, L, H, P + T, d))
    hist_v = np.zeros((S, L, H, P + T, d))
    for s in range(S):
        k, v = inputs.prompt(w, 7, s, P)
        c.load(s, k, v)
        hist_k[s, :, :, :P] = k
        hist_v[s, :, :, :P] = v
    for t in range(T):
        q, kn, vn = inputs.step_inputs(w, 7, t, S)
        out = c.step(q, kn, vn, B=w.budget, W=w.window)
        n = P + t + 1
        hist_k[:, :, :, n - 1] = kn
        hist_v[:, :, :, n - 1] = vn
        for s in range(S):
            for l in range(L):
                ref = _sdpa_gqa(q[s, l].astype(np.float64),
                                hist_k[s, l, :, :n], hist_v[s, l, :, :n], G)
                np.testing.assert_allclose(out[s, l], ref, rtol=1e-12,
                                           atol=1e-13)
        assert (c.len == n).all()


def test_score_equals_sum_of_library_probabilities():
    """Accumulated attention = sum over steps of the mean over the G heads of
    the attention probability, where the probability is obtained from the
    library's SDPA by attending to the identity matrix as values."""
    L, H, G, d, P, T = 1, 2, 2, 8, 6, 7
    w = inputs.Workload("t", L, H, G, d, "f32", 1 << 20, 0, P, T)
    c = orc.OracleCache(1, L, H, G, d, cap=P + T)
    k, v = inputs.prompt(w, 3, 0, P)
    c.load(0, k, v)
    hk = [list(k[0, h]) for h in range(H)]
    acc = [np.zeros(P + T) for _ in range(H)]
    for t in range(T):
        q, kn, vn = inputs.step_inputs(w, 3, t, 1)
        c.step(q, kn, vn, evict=False)
        for h in range(H):
            hk[h].append(kn[0, 0, h])
            n = len(hk[h])
            Kh = torch.tensor(np.array(hk[h]), dtype=torch.float64)
            eye = torch.eye(n, dtype=torch.float64)
            qh = torch.tensor(q[0, 0, h * G:(h + 1) * G], dtype=torch.float64)
            prob = F.scaled_dot_product_attention(qh[:, None], Kh[None].expand(G, n, d),
                                                  eye[None].expand(G, n, n))[:, 0]
            acc[h][:n] += prob.mean(0).numpy()
    for h in range(H):
        np.testing.assert_allclose(c.score[0, 0, h, :P + T], acc[h], rtol=1e-12,
                                   atol=1e-14)


# --------------------------------------------------------------------------
# Invariants
# --------------------------------------------------------------------------

def test_probabilities_sum_to_one():
    rng = np.random.default_rng(1)
    for n in (1, 2, 5, 33, 200):
        K = rng.standard_normal((n, 32)) * 3
        V = rng.standard_normal((n, 32))
        q = rng.standard_normal((5, 32)) * 3
        _, prob = orc.attend_unit(K, V, q)
        np.testing.assert_allclose(prob.sum(1), 1.0, atol=1e-12, rtol=0)
        assert (prob >= 0).all()


def _run_tracking_evicted(w, seed, steps, S=1):
    """Run the oracle, returning per-unit sums of retained and evicted scores."""
    c = orc.OracleCache(S, w.n_layers, w.n_kv_heads, w.group, w.head_dim,
                        cap=w.prompt + 2)
    for s in range(S):
        k, v = inputs.prompt(w, seed, s, w.prompt)
        c.load(s, k, v)
    evicted = np.zeros(c.len.shape)
    history = []
    for t in range(steps):
        q, kn, vn = inputs.step_inputs(w, seed, t, S)
        c.step(q, kn, vn, evict=False)
        before = c.score.copy(), c.pos.copy(), c.len.copy()
        c.evict(w.budget, w.window)
        for idx in np.ndindex(*c.len.shape):
            n = before[2][idx]
            kept = set(c.pos[idx][:c.len[idx]].tolist())
            for i in range(n):
                if before[1][idx][i] not in kept:
                    evicted[idx] += before[0][idx][i]
        history.append((before, c.pos.copy(), c.len.copy()))
    return c, evicted, history


def test_score_conservation_and_window():
    w = inputs.Workload("t", 2, 2, 4, 16, "f32", 5, 3, 12, 0)
    T = 25
    c, evicted, history = _run_tracking_evicted(w, 11, T)
    retained = np.array([[c.score[0, l, h, :c.len[0, l, h]].sum()
                          for h in range(2)] for l in range(2)])
    # each step adds exactly one unit of attention mass per KV head
    np.testing.assert_allclose(retained + evicted[0], T, rtol=1e-12)
    for t, (before, pos_after, len_after) in enumerate(history):
        n_before = before[2]
        assert (len_after == np.minimum(n_before, w.budget + w.window)).all()
        newest = w.prompt + t
        for idx in np.ndindex(*len_after.shape):
            live = set(pos_after[idx][:len_after[idx]].tolist())
            assert set(range(newest - w.window + 1, newest + 1)) <= live


def test_zero_query_closed_form():
    """q = 0: every live row gets probability 1/n, out is the mean of the live
    values, all candidates tie at the first eviction so the lowest positions
    are kept, and afterwards the oldest rows stay ahead of every newcomer."""
    L, H, G, d, P, B, W, T = 1, 2, 3, 8, 20, 4, 3, 12
    w = inputs.Workload("t", L, H, G, d, "f32", B, W, P, T)
    c = orc.OracleCache(1, L, H, G, d, cap=P + 1)
    k, v = inputs.prompt(w, 5, 0, P)
    c.load(0, k, v)
    expect = {}  # pos -> closed-form score
    n1 = P + 1
    for t in range(T):
        _, kn, vn = inputs.step_inputs(w, 5, t, 1)
        q = np.zeros((1, L, H * G, d))
        live_before = [c.unit_rows(0, 0, h) for h in range(H)]
        out = c.step(q, kn, vn, B=B, W=W)
        n = P + 1 if t == 0 else B + W + 1
        for h in range(H):
            Vlive = np.concatenate([live_before[h][3], vn[0, 0, h][None]])
            np.testing.assert_allclose(out[0, 0, h * G:(h + 1) * G],
                                       np.broadcast_to(Vlive.mean(0), (G, d)),
                                       rtol=0, atol=1e-14)
        newest = P + t
        for p in list(expect):
            expect[p] += 1.0 / n
        if t == 0:
            for p in range(P + 1):
                expect[p] = 1.0 / n1
        else:
            expect[newest] = 1.0 / n
        kept = set(range(B)) | set(range(newest - W + 1, newest + 1))
        expect = {p: s for p, s in expect.items() if p in kept}
        for h in range(H):
            pos, score, _, _ = c.unit_rows(0, 0, h)
            assert pos.tolist() == sorted(kept)
            np.testing.assert_allclose(score, [expect[p] for p in pos.tolist()],
                                       rtol=1e-13)


def test_single_row_returns_its_value():
    rng = np.random.default_rng(2)
    K, V, q = rng.standard_normal((1, 8)), rng.standard_normal((1, 8)), \
        rng.standard_normal((3, 8))
    out, prob = orc.attend_unit(K, V, q)
    assert (prob == 1.0).all()
    assert (out == V[0]).all()


def test_dominant_key():
    rng = np.random.default_rng(3)
    n, d = 40, 32
    K = rng.standard_normal((n, d)) * 0.1
    V = rng.standard_normal((n, d))
    q = rng.standard_normal((1, d))
    j = 17
    K[j] = 50.0 * math.sqrt(d) * q[0] / np.dot(q[0], q[0])  # logit exactly 50
    out, prob = orc.attend_unit(K, V, q)
    # every other logit is below 50 - 40 (|k| ~ 0.1, |q| ~ sqrt(d)), so the
    # rest of the mass is below n * exp(-40)
    assert prob[0, j] >= 1.0 - n * math.exp(-40)
    np.testing.assert_allclose(out[0], V[j], rtol=0, atol=1e-12)


def test_permutation_invariance():
    w = inputs.Workload("t", 1, 2, 2, 16, "f32", 6, 2, 15, 0)
    base = orc.OracleCache(1, 1, 2, 2, 16, cap=16)
    k, v = inputs.prompt(w, 9, 0, 15)
    base.load(0, k, v)
    base.score[0, 0, :, :15] = np.random.default_rng(4).random((2, 15))
    shuf = base.copy()
    perm = np.random.default_rng(5).permutation(15)
    for a in (shuf.K, shuf.V, shuf.score, shuf.pos):
        a[0, 0, :, :15] = a[0, 0][:, perm]
    q, kn, vn = inputs.step_inputs(w, 9, 0, 1)
    o1 = base.step(q, kn, vn, B=w.budget, W=w.window)
    o2 = shuf.step(q, kn, vn, B=w.budget, W=w.window)
    np.testing.assert_allclose(o1, o2, rtol=1e-13, atol=1e-15)
    for h in range(2):
        p1, s1, _, _ = base.unit_rows(0, 0, h)
        p2, s2, _, _ = shuf.unit_rows(0, 0, h)
        assert p1.tolist() == p2.tolist()
        np.testing.assert_allclose(s1, s2, rtol=1e-13)


# --------------------------------------------------------------------------
# Brute force: selection by exhaustive subset enumeration, and a whole tiny
# trajectory with the library's attention and enumerated selection.
# --------------------------------------------------------------------------

def _brute_keep(score, pos, B, W):
    """The unique kept set: the W newest positions, plus the size-B subset S of
    the others such that every member outranks every non-member under
    (higher score, then lower position)."""
    n = len(score)
    if n <= B + W:
        return set(range(n))
    order = sorted(range(n), key=lambda i: -pos[i])
    window = set(order[:W])
    rest = [i for i in range(n) if i not in window]

    def better(i, j):
        return score[i] > score[j] or (score[i] == score[j] and pos[i] < pos[j])

    valid = []
    for sub in itertools.combinations(rest, B):
        sset = set(sub)
        if all(better(i, j) for i in sset for j in rest if j not in sset):
            valid.append(sset)
    assert len(valid) == 1
    return window | valid[0]


def test_selection_matches_subset_enumeration():
    rng = np.random.default_rng(6)
    for _ in range(300):
        n = int(rng.integers(1, 10))
        score = rng.choice([0.0, 0.1, 0.25, 0.5, 0.7], size=n)  # forces ties
        pos = rng.permutation(40)[:n].astype(np.int32)
        B, W = int(rng.integers(0, 5)), int(rng.integers(0, 4))
        keep = orc.select_unit(score, pos, B, W)
        assert set(np.nonzero(keep)[0].tolist()) == _brute_keep(score, pos, B, W)


def test_tiny_trajectory_brute_force():
    """A whole evicting trajectory against an independent brute force: torch
    SDPA for the outputs and (with identity values) the probabilities, plain
    lists for the state, subset enumeration for TopB."""
    L, H, G, d, P, B, W, T = 1, 2, 2, 8, 7, 3, 2, 14
    w = inputs.Workload("t", L, H, G, d, "f32", B, W, P, T, sigma=1.5)
    c = orc.OracleCache(1, L, H, G, d, cap=P + 1)
    k, v = inputs.prompt(w, 21, 0, P)
    c.load(0, k, v)
    # brute-force state per head: list of [pos, score, k, v]
    rows = [[[i, 0.0, k[0, h, i].astype(np.float64), v[0, h, i].astype(np.float64)]
             for i in range(P)] for h in range(H)]
    for t in range(T):
        q, kn, vn = inputs.step_inputs(w, 21, t, 1)
        out = c.step(q, kn, vn, B=B, W=W)
        for h in range(H):
            rows[h].append([P + t, 0.0, kn[0, 0, h].astype(np.float64),
                            vn[0, 0, h].astype(np.float64)])
            n = len(rows[h])
            Kh = torch.tensor(np.array([r[2] for r in rows[h]]))
            Vh = torch.tensor(np.array([r[3] for r in rows[h]]))
            qh = torch.tensor(q[0, 0, h * G:(h + 1) * G].astype(np.float64))
            o = F.scaled_dot_product_attention(qh[:, None], Kh[None].expand(G, n, d),
                                               Vh[None].expand(G, n, d))[:, 0]
            prob = F.scaled_dot_product_attention(
                qh[:, None], Kh[None].expand(G, n, d),
                torch.eye(n, dtype=torch.float64)[None].expand(G, n, n))[:, 0]
            np.testing.assert_allclose(out[0, 0, h * G:(h + 1) * G], o.numpy(),
                                       rtol=1e-12, atol=1e-13)
            for i in range(n):
                rows[h][i][1] += float(prob[:, i].mean())
            keep = _brute_keep([r[1] for r in rows[h]], [r[0] for r in rows[h]],
                               B, W)
            rows[h] = [r for i, r in enumerate(rows[h]) if i in keep]
            pos, score, _, _ = c.unit_rows(0, 0, h)
            assert pos.tolist() == sorted(r[0] for r in rows[h])
            np.testing.assert_allclose(
                score, [r[1] for r in sorted(rows[h], key=lambda r: r[0])],
                rtol=1e-12)


def test_layer_range_step_touches_only_its_layers():
    w = inputs.Workload("t", 3, 1, 2, 8, "f32", 2, 1, 6, 0)
    c = orc.OracleCache(1, 3, 1, 2, 8, cap=8)
    k, v = inputs.prompt(w, 1, 0, 6)
    c.load(0, k, v)
    snap = c.copy()
    q, kn, vn = inputs.step_inputs(w, 1, 0, 1, n_layers=1)
    c.step(q, kn, vn, B=2, W=1, layer_begin=1, layer_end=2)
    for l in (0, 2):
        assert (c.K[0, l] == snap.K[0, l]).all() and (c.len[0, l] == 6).all()
    assert (c.len[0, 1] == 3).all()
    # the same layer driven alone in a one-layer cache gives the same state
    one = orc.OracleCache(1, 1, 1, 2, 8, cap=8)
    one.load(0, k[1:2], v[1:2])
    one.step(q, kn, vn, B=2, W=1)
    assert (one.pos[0, 0] == c.pos[0, 1]).all()
    np.testing.assert_allclose(one.score[0, 0], c.score[0, 1], rtol=0, atol=0)


def test_tiny_workload_invariants():
    """The Tiny workload (prompt 128, B=16, W=8) for 256 steps: retained size,
    window and score conservation hold at every step."""
    w = inputs.WORKLOADS["tiny"]
    c = orc.OracleCache(1, w.n_layers, w.n_kv_heads, w.group, w.head_dim,
                        cap=w.prompt + 1)
    k, v = inputs.prompt(w, 0, 0, w.prompt)
    c.load(0, k, v)
    evicted = np.zeros(c.len.shape)

    def live_sum():
        return np.array([c.score[idx][:c.len[idx]].sum()
                         for idx in np.ndindex(*c.len.shape)]).reshape(c.len.shape)

    for t in range(w.steps):
        q, kn, vn = inputs.step_inputs(w, 0, t, 1)
        c.step(q, kn, vn, evict=False)
        before = live_sum()
        c.evict(w.budget, w.window)
        evicted += before - live_sum()
        assert (c.len == min(w.prompt + t + 1, w.budget + w.window)).all()
        newest = w.prompt + t
        for idx in np.ndindex(*c.len.shape):
            live = set(c.pos[idx][:c.len[idx]].tolist())
            assert set(range(newest - w.window + 1, newest + 1)) <= live
    np.testing.assert_allclose(live_sum() + evicted, w.steps, rtol=1e-11)


def test_resized_oracle_steps_identically():
    """OracleCache.resized only moves data: a resized copy takes the same
    next step (outputs, scores, retained rows) as the original."""
    w = inputs.Workload("rs", 2, 2, 3, 16, "f32", 6, 2, 20, 0, sigma=1.0)
    o = orc.OracleCache(1, 2, 2, 3, 16, cap=21)
    k, v = inputs.prompt(w, 5, 0, 20)
    o.load(0, k, v)
    o.step(*inputs.step_inputs(w, 5, 0, 1), B=6, W=2)
    r = o.resized(9)
    q, kn, vn = inputs.step_inputs(w, 5, 1, 1)
    a = o.step(q, kn, vn, B=6, W=2)
    b = r.step(q, kn, vn, B=6, W=2)
    assert np.array_equal(a, b)
    for l in range(2):
        for h in range(2):
            for x, y in zip(o.unit_rows(0, l, h), r.unit_rows(0, l, h)):
                assert np.array_equal(x, y)
    with pytest.raises(ValueError):
        o.resized(5)


# --------------------------------------------------------------------------
# Absorbing a chunk (a token block attended causally in one call)
# --------------------------------------------------------------------------

def _chunk(rng, c, H, G, d):
    q = rng.standard_normal((1, 1, c, H * G, d))
    kn = rng.standard_normal((1, 1, c, H, d))
    vn = rng.standard_normal((1, 1, c, H, d))
    return q, kn, vn


def test_absorb_equals_masked_sdpa_and_column_sums():
    """Against the library: outputs are SDPA with a mask that lets token j
    see every prompt row and chunk rows 0..j; scores are the column sums over
    the chunk's tokens of the head-mean probabilities (SDPA with identity
    values); each token adds exactly 1 per KV head."""
    H, G, d, P, c = 2, 3, 16, 5, 6
    rng = np.random.default_rng(21)
    o = orc.OracleCache(1, 1, H, G, d, cap=P + c)
    kp = rng.standard_normal((1, H, P, d))
    vp = rng.standard_normal((1, H, P, d))
    o.load(0, kp, vp)
    q, kn, vn = _chunk(rng, c, H, G, d)
    out = o.absorb(q, kn, vn, evict=False)
    n = P + c
    mask = torch.zeros(c, n, dtype=torch.bool)
    for j in range(c):
        mask[j, :P + j + 1] = True
    for h in range(H):
        K = torch.from_numpy(np.concatenate([kp[0, h], kn[0, 0, :, h]]))
        V = torch.from_numpy(np.concatenate([vp[0, h], vn[0, 0, :, h]]))
        Q = torch.from_numpy(np.ascontiguousarray(
            q[0, 0, :, h * G:(h + 1) * G].transpose(1, 0, 2)))  # [G, c, d]
        ref = F.scaled_dot_product_attention(Q, K[None].expand(G, n, d),
                                             V[None].expand(G, n, d),
                                             attn_mask=mask)
        np.testing.assert_allclose(out[0, 0, :, h * G:(h + 1) * G],
                                   ref.numpy().transpose(1, 0, 2),
                                   rtol=1e-12, atol=1e-13)
        eye = torch.eye(n, dtype=torch.float64)
        prob = F.scaled_dot_product_attention(Q, K[None].expand(G, n, d),
                                              eye[None].expand(G, n, n),
                                              attn_mask=mask)  # [G, c, n]
        want = prob.mean(0).sum(0).numpy()
        np.testing.assert_allclose(o.score[0, 0, h, :n], want, rtol=1e-12,
                                   atol=1e-14)
        assert abs(o.score[0, 0, h, :n].sum() - c) < 1e-12
    assert (o.len == n).all() and (o.next_pos == n).all()


def test_absorb_then_evict_keeps_the_brute_force_set():
    """After a chunk, the unit is cut to B + W once: the W newest positions
    plus the top B of the rest under (score desc, position asc), found here
    by subset enumeration on the pre-eviction scores."""
    H, G, d, B, W = 2, 2, 8, 3, 2
    rng = np.random.default_rng(22)
    for P, c in ((4, 5), (0, 7), (6, 1), (2, 3)):
        o = orc.OracleCache(1, 1, H, G, d, cap=P + c)
        if P:
            o.load(0, rng.standard_normal((1, H, P, d)),
                   rng.standard_normal((1, H, P, d)))
        q, kn, vn = _chunk(rng, c, H, G, d)
        keep = o.copy()
        keep.absorb(q, kn, vn, evict=False)
        o.absorb(q, kn, vn, B=B, W=W)
        for h in range(H):
            n = P + c
            sc, ps = keep.score[0, 0, h, :n], keep.pos[0, 0, h, :n]
            want = {int(ps[i]) for i in _brute_keep(list(sc), list(ps), B, W)}
            got = set(o.pos[0, 0, h, :o.len[0, 0, h]].tolist())
            assert got == want


def test_copied_sequence_steps_like_its_source():
    """A candidate forked by copy (App. C) and driven with the parent's own
    inputs evolves exactly as the parent does, eviction every token
    included; a copy into a larger capacity changes nothing either."""
    w = inputs.WORKLOADS["tiny"]
    seed, S = 3, 2
    par = orc.OracleCache(S, w.n_layers, w.n_kv_heads, w.group, w.head_dim,
                          cap=w.budget + w.window + 1)
    for s in range(S):
        k, v = inputs.prompt(w, seed, s, 20)
        par.load(s, k, v)
    for t in range(6):
        q, kn, vn = inputs.step_inputs(w, seed, t, S)
        par.step(q, kn, vn, B=w.budget, W=w.window)
    kids = orc.OracleCache(2 * S, w.n_layers, w.n_kv_heads, w.group,
                           w.head_dim, cap=w.budget + w.window + 9)
    kids.copy_sequences(par, [0, 0, 1, 1], [0, 1, 2, 3])
    for t in range(6, 16):
        q, kn, vn = inputs.step_inputs(w, seed, t, S)
        ref = par.step(q, kn, vn, B=w.budget, W=w.window)
        rep = np.repeat(np.arange(S), 2)
        out = kids.step(q[rep], kn[rep], vn[rep], B=w.budget, W=w.window)
        assert np.array_equal(out, ref[rep])
        for c in range(2 * S):
            a = rep[c]
            for l in range(w.n_layers):
                for h in range(w.n_kv_heads):
                    pp, ps, pk, pv = par.unit_rows(a, l, h)
                    cp, cs, ck, cv = kids.unit_rows(c, l, h)
                    assert np.array_equal(pp, cp) and np.array_equal(ps, cs)
                    assert np.array_equal(pk, ck) and np.array_equal(pv, cv)
    # commit: the parent takes a candidate's state back
    par2 = par.copy()
    par2.copy_sequences(kids, [1, 2], [0, 1])
    assert np.array_equal(par2.len, par.len)
    assert np.array_equal(par2.next_pos, par.next_pos)
