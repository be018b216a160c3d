"""Pins of the entropy-test oracle (oracle/entropy.py) against what the paper
and the mathematics fix: scipy's entropy of scipy's softmax (library
routines), closed forms (uniform over k tokens gives ln k; a two-level
distribution), invariances (shift, permutation), a hand-derived worked
example of the detector (tests/golden/entropy_detector_worked.json), and the
float32 decision against the fp64 one.  A last test plants plausible mistakes
in copies of the oracle and checks that these pins catch each one.
"""
import json
import math
import os

import numpy as np
import pytest
from scipy import special, stats

from oracle import entropy as ent


def _golden(golden_dir):
    with open(os.path.join(golden_dir, "entropy_detector_worked.json")) as f:
        return json.load(f)


def _uniform_logits(k, vocab):
    row = np.full(vocab, -np.inf)
    row[:k] = 0.0
    return row


def _expand(segments):
    ks = []
    for count, k in segments:
        ks += [k] * count
    return ks


# --------------------------------------------------------------------------
# Checks shared by the pins and the planted-mistake test
# --------------------------------------------------------------------------

def _check_library(token_entropy):
    rng = np.random.default_rng(11)
    for V, sigma, T, shift in [(7, 1.0, 1.0, 0.0), (1000, 3.0, 1.0, 0.0),
                               (4096, 2.0, 2.0, 0.0), (4096, 4.0, 0.8, 0.0),
                               (513, 2.5, 1.0, 900.0)]:
        x = rng.standard_normal((3, V)) * sigma + shift
        want = stats.entropy(special.softmax(x / T, axis=-1), axis=-1)
        got = token_entropy(x, T)
        if not np.allclose(got, want, rtol=1e-12, atol=1e-12):
            return False
    return True


def _check_closed_forms(token_entropy):
    V = 152064
    for k in (1, 2, 7, 1000, 1097, V):
        if abs(token_entropy(_uniform_logits(k, V)) - math.log(k)) > 1e-12:
            return False
    # one token at logit a, the other V - 1 at 0:
    # p1 = e^a / (e^a + V - 1), H = -p1 ln p1 - (1 - p1) ln((1 - p1) / (V - 1))
    V, a = 5000, 9.0
    p1 = math.exp(a) / (math.exp(a) + V - 1)
    want = -p1 * math.log(p1) - (1 - p1) * math.log((1 - p1) / (V - 1))
    row = np.zeros(V)
    row[17] = a
    return abs(token_entropy(row) - want) < 1e-12


def _run_golden(detector_cls, g, token_entropy=ent.token_entropy):
    rows = g["rows"]
    ks = [_expand(r["segments"]) for r in rows]
    E = max(len(k) for k in ks)
    det = detector_cls(len(rows), g["window"], g["guard"], g["tau"])
    for e in range(E):
        H = np.array([token_entropy(_uniform_logits(k[e], g["vocab"]))
                      if e < len(k) else 0.0 for k in ks])
        _, stop = det.step(H)
    return [int(s) for s in stop]


# --------------------------------------------------------------------------
# Pins
# --------------------------------------------------------------------------

def test_entropy_equals_scipy_entropy_of_softmax():
    assert _check_library(ent.token_entropy)


def test_entropy_closed_forms():
    assert _check_closed_forms(ent.token_entropy)


def test_entropy_invariances():
    rng = np.random.default_rng(3)
    x = rng.standard_normal((4, 3000)) * 3.0
    h = ent.token_entropy(x)
    assert np.allclose(ent.token_entropy(x + 123.5), h, rtol=0, atol=1e-12)
    perm = rng.permutation(3000)
    assert np.allclose(ent.token_entropy(x[:, perm]), h, rtol=0, atol=1e-12)
    # bounds: 0 <= H <= ln V
    assert np.all(h >= 0) and np.all(h <= math.log(3000) + 1e-12)


def test_golden_entropy_detector_worked_example(golden_dir):
    g = _golden(golden_dir)
    for r in g["rows"]:
        for _, k in r["segments"]:
            assert abs(ent.token_entropy(_uniform_logits(k, g["vocab"]))
                       - math.log(k)) < 1e-12
    assert _run_golden(ent.EntropyDetector, g) == [r["stop"] for r in g["rows"]]


def test_detector_skips_stopped_rows_and_resets():
    det = ent.EntropyDetector(2, window=3, guard=2, tau=1.0)
    for _ in range(3):
        mean, stop = det.step([2.0, 0.5])
    assert list(stop) == [3, 0]
    mean, stop = det.step([0.0, 0.5])
    assert math.isnan(mean[0]) and list(stop) == [3, 0]
    assert det.hist[0] == [2.0, 2.0, 2.0]
    det.reset(0, 1)
    assert det.hist[0] == [] and det.stop[0] == 0 and det.hist[1] == [0.5] * 4


# --------------------------------------------------------------------------
# Planted mistakes: each must fail at least one of the checks above
# --------------------------------------------------------------------------

def _entropy_log2(x, T=1.0):
    return ent.token_entropy(x, T) / math.log(2.0)


def _entropy_no_temperature(x, T=1.0):
    return ent.token_entropy(x, 1.0)


def _entropy_no_max_shift(x, T=1.0):
    z = np.asarray(x, np.float64) / T
    with np.errstate(all="ignore"):
        p = np.exp(z) / np.exp(z).sum(-1, keepdims=True)
        return -np.nansum(np.where(p > 0, p * np.log(p), 0.0), axis=-1)


def _entropy_top20(x, T=1.0):
    z = np.asarray(x, np.float64) / T
    kth = min(20, z.shape[-1])
    cut = np.sort(z, axis=-1)[..., -kth][..., None]
    return ent.token_entropy(np.where(z >= cut, z, -np.inf), 1.0)


class _Window(ent.EntropyDetector):
    def __init__(self, rows, window, guard, tau, delta=0):
        super().__init__(rows, window + delta, guard, tau)


class _Window11(_Window):
    def __init__(self, rows, window, guard, tau):
        super().__init__(rows, window, guard, tau, -1)


class _Window13(_Window):
    def __init__(self, rows, window, guard, tau):
        super().__init__(rows, window, guard, tau, +1)


class _GuardInclusive(ent.EntropyDetector):
    def __init__(self, rows, window, guard, tau):
        super().__init__(rows, window, guard - 1, tau)


class _CumulativeMean(ent.EntropyDetector):
    def __init__(self, rows, window, guard, tau):
        super().__init__(rows, 1 << 30, guard, tau)


def test_planted_mistakes_are_caught(golden_dir):
    g = _golden(golden_dir)
    want = [r["stop"] for r in g["rows"]]
    for bad in (_entropy_log2, _entropy_no_temperature, _entropy_no_max_shift,
                _entropy_top20):
        caught = not (_check_library(bad) and _check_closed_forms(bad)
                      and _run_golden(ent.EntropyDetector, g, bad) == want)
        assert caught, bad.__name__
    for bad in (_Window11, _Window13, _GuardInclusive, _CumulativeMean):
        assert _run_golden(bad, g) != want, bad.__name__
