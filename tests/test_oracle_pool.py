"""The spawned-process oracle of full-length candidate runs
(tests/oracle_pool.py), driven on the CPU: a device side emulated by the
oracle itself must pass every check, and planted mistakes in what that side
reports (an output, a score) must be caught."""
import numpy as np
import pytest

from oracle import oracle as orc
from oracle import parity
from paper_2608_15797_gb300 import inputs
from tests import oracle_pool

W_ = inputs.Workload("pool", 3, 2, 2, 16, "f32", 4, 2, 12, 0, n_cand=3,
                     cand_step=5, sigma=1.0)


def _emulated_run(plant=None, steps=2):
    w = W_
    B, W, N, T = w.budget, w.window, w.n_cand, w.cand_step
    m = B + W
    par = orc.OracleCache(1, w.n_layers, w.n_kv_heads, w.group, w.head_dim,
                          w.prompt + 1)
    k, v = inputs.prompt(w, 5, 0, w.prompt)
    par.load(0, k, v)
    q, kn, vn = inputs.step_inputs(w, 5, 0, 1)
    par.step(q, kn, vn, B, W)
    par = par.resized(m)
    pool = oracle_pool.CandidateOraclePool(w, N, m, T, seed=5, parts=2)
    try:
        pool.set_parent(par)
        a = pool.a
        for j in range(steps):
            a["gpos"][...] = par.pos[0]
            a["glen"][...] = par.len[0]
            cands = [par.resized(m + T) for _ in range(N)]
            pool.fork()
            for t in range(T):
                pool.token_inputs(100 + j * T + t)
                for c_ in range(N):
                    qq, kk, vv = inputs.step_inputs(w, 5, 100 + j * T + t, 1,
                                                    cand=c_ + 1)
                    assert np.array_equal(a["q"][c_], qq[0])
                    out = cands[c_].step(qq, kk, vv, evict=False)
                    a["out"][c_] = out[0]
                    n_p = par.len[0]
                    a["pscore"][c_] = cands[c_].score[0, :, :, :m]
                    a["tscore"][c_] = 0
                    a["tpos"][c_] = 0
                    for l in range(w.n_layers):
                        for h in range(w.n_kv_heads):
                            p0, n = n_p[l, h], cands[c_].len[0, l, h]
                            a["tscore"][c_, l, h, :n - p0] = \
                                cands[c_].score[0, l, h, p0:n]
                            a["tpos"][c_, l, h, :n - p0] = \
                                cands[c_].pos[0, l, h, p0:n]
                            a["tlen"][c_, l, h] = n - p0
                if plant == "out" and j == 1 and t == 3:
                    a["out"][2, 1, 0, 5] += 0.05
                if plant == "score" and j == 1 and t == 2:
                    a["tscore"][1, 2, 1, 0] *= 1 + 3e-4
                pool.check(t)
            chosen = int(inputs.candidate_pick(5, j, 1, N)[0])
            nxt = cands[chosen].copy()
            nxt.evict(B, W)
            a["gpos"][...] = nxt.pos[0, :, :, :m]
            a["gscore"][...] = nxt.score[0, :, :, :m].astype(np.float32)
            a["glen"][...] = nxt.len[0]
            st = pool.commit(chosen, B, W)
            assert st.units == w.n_layers * w.n_kv_heads
            par = nxt.resized(m)
    finally:
        pool.close()


def test_pool_passes_an_exact_device_side():
    _emulated_run()


@pytest.mark.parametrize("plant", ["out", "score"])
def test_pool_catches_planted_mistakes(plant):
    with pytest.raises(parity.ParityError):
        _emulated_run(plant)
