"""fp64 oracle of the entropy test of the online degeneration detector.

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` leg of ``bench.py`` may use this module; the product path
never imports it.  It shares no code with the CUDA library.

What it computes (Sec. 3.2, "Incoherent generation"; App. C, "Online
degeneration detection"):

* ``token_entropy`` -- H_e = -sum_v p_e(v) log p_e(v), the predictive
  entropy of the next-token distribution at generated position e, in nats.
  p_e is the softmax of the logits divided by the temperature, over the whole
  vocabulary.
* ``EntropyDetector`` -- the moving mean of H over a recent window of |W_e|
  positions, and termination of a candidate once that mean exceeds
  tau_ent.  App. C fixes tau_ent = 7.0, a window of 12 and a guard of 24
  tokens.

Readings where the paper is silent:

* The window is the last min(e, window) positions, the current one included.
* The guard: no test is made while e <= guard (e counts the candidate's
  generated tokens from 1), so the first position tested is guard + 1.
* A terminated candidate stays terminated: its later positions are not
  scored and do not enter its window.
* The distribution is the full-vocabulary softmax at the given temperature
  (1 unless stated), before any top-k / top-p truncation: with top-k 20 the
  entropy could never exceed ln 20 < 3, so tau_ent = 7 would never fire.

Pins: ``tests/test_entropy_oracle_pins.py`` (scipy's entropy of scipy's softmax,
closed forms, invariances) and ``tests/golden/entropy_detector_worked.json``
(hand-derived stop positions).
"""
from __future__ import annotations

import numpy as np


def token_entropy(logits, temperature: float = 1.0) -> np.ndarray:
    """H of each row of ``logits`` ([..., V]) in nats, fp64.

    p = exp(z - max z) / sum exp(z - max z) with z = logits / temperature;
    H = -sum over p > 0 of p log p (0 log 0 = 0, so -inf logits add nothing).
    """
    z = np.asarray(logits, dtype=np.float64) / float(temperature)
    z = z - z.max(axis=-1, keepdims=True)
    e = np.exp(z)
    p = e / e.sum(axis=-1, keepdims=True)
    with np.errstate(divide="ignore", invalid="ignore"):
        terms = np.where(p > 0, p * np.log(np.where(p > 0, p, 1.0)), 0.0)
    return -terms.sum(axis=-1)


class EntropyDetector:
    """Per-row state of the entropy test: the entropies seen since the row's
    last reset and the position at which it stopped (0 while live)."""

    def __init__(self, rows: int, window: int = 12, guard: int = 24,
                 tau: float = 7.0):
        self.rows, self.window, self.guard, self.tau = rows, window, guard, tau
        self.hist = [[] for _ in range(rows)]
        self.stop = np.zeros(rows, np.int64)

    def reset(self, begin: int = 0, end: int | None = None):
        """A new candidate takes rows [begin, end): empty history, live."""
        end = self.rows if end is None else end
        for r in range(begin, end):
            self.hist[r] = []
            self.stop[r] = 0

    def step(self, H):
        """Feed one generated position's entropies ``H`` [rows] (fp64).

        Returns (mean, stopped): the moving mean H-bar_e of each live row
        (NaN for rows already stopped, which are skipped) and the stop
        positions after this position."""
        H = np.asarray(H, dtype=np.float64)
        mean = np.full(self.rows, np.nan)
        for r in range(self.rows):
            if self.stop[r]:
                continue
            self.hist[r].append(float(H[r]))
            e = len(self.hist[r])
            win = self.hist[r][-self.window:]
            mean[r] = sum(win) / len(win)
            if e > self.guard and mean[r] > self.tau:
                self.stop[r] = e
        return mean, self.stop.copy()
