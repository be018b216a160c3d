"""The lock-step checker (oracle/parity.py) against planted mistakes.

The checker decides what a valid retained set is (Eq. 1 TopB with the
Sec. 4.1 window, ties kept at the lower position), so it is pinned here on
hand-built units: a set that breaks the tie rule, drops a row that is no
near-tie, evicts a window row or returns a wrong score must be rejected,
and the valid alternatives must pass.  CPU only.
"""
import numpy as np
import pytest

from oracle import parity


def _unit():
    # Seven rows; the window (W=2) is positions 5 and 6.  Positions 1 and 3
    # tie exactly at the lowest candidate score; position 4 is a near-tie of
    # position 0 (within 1e-4 relative).
    pos = np.array([0, 1, 2, 3, 4, 5, 6], np.int32)
    score = np.array([0.50, 0.25, 0.90, 0.25, 0.50 * (1 - 5e-5), 0.1, 0.0])
    return pos, score


def _check(keep, B=3, W=2):
    pos, score = _unit()
    g_pos = np.array(sorted(keep), np.int32)
    g_score = score[g_pos]
    return parity.check_unit(pos, score, g_pos, g_score, B, W, evict=True,
                             where="unit")


def test_the_oracle_set_passes_without_adoption():
    # TopB (B=3) over candidates 0..4: 2 (0.9), 0 (0.5), 4 (0.49997).
    adopted, worst, got = _check({2, 0, 4, 5, 6})
    assert not adopted and worst == 0.0 and got == {0, 2, 4, 5, 6}


def test_a_near_tie_swap_is_adopted():
    # Keeping 4 instead of 0 is a near-tie (relative gap 5e-5 <= 1e-4).
    pos, score = _unit()
    # B=2: oracle keeps 2 and 0; a set keeping 2 and 4 is a near-tie swap.
    g_pos = np.array([2, 4, 5, 6], np.int32)
    adopted, _, _ = parity.check_unit(pos, score, g_pos, score[g_pos], 2, 2,
                                      evict=True, where="unit")
    assert adopted


def test_an_exact_tie_must_keep_the_lower_position():
    pos, score = _unit()
    # B=4: the oracle keeps 2, 0, 4 and, of the tie 1/3, position 1.
    ok = np.array([0, 1, 2, 4, 5, 6], np.int32)
    parity.check_unit(pos, score, ok, score[ok], 4, 2, evict=True, where="u")
    bad = np.array([0, 2, 3, 4, 5, 6], np.int32)   # kept 3, evicted 1
    with pytest.raises(parity.ParityError, match="exact tie"):
        parity.check_unit(pos, score, bad, score[bad], 4, 2, evict=True,
                          where="u")


def test_a_dropped_row_above_the_near_tie_band_fails():
    pos, score = _unit()
    bad = np.array([1, 2, 4, 5, 6], np.int32)   # dropped 0 (0.5) for 1 (0.25)
    with pytest.raises(parity.ParityError, match="not a near-tie"):
        parity.check_unit(pos, score, bad, score[bad], 3, 2, evict=True,
                          where="u")


def test_an_evicted_window_row_fails():
    pos, score = _unit()
    bad = np.array([0, 2, 4, 5, 1], np.int32)
    with pytest.raises(parity.ParityError, match="window"):
        parity.check_unit(pos, score, bad, score[bad], 3, 2, evict=True,
                          where="u")


def test_a_wrong_retained_score_fails():
    pos, score = _unit()
    g = np.array([0, 2, 4, 5, 6], np.int32)
    s = score[g].copy()
    s[1] *= 1 + 2e-4
    with pytest.raises(parity.ParityError, match="score of pos"):
        parity.check_unit(pos, score, g, s, 3, 2, evict=True, where="u")


def test_swap_rule_for_absolute_slack_keeps_ties_at_lower_positions():
    # The R-KV form (absolute near-tie slack on z) has the same tie rule.
    kept = [(0.3, 7), (0.1, 9)]
    parity.check_swaps(kept, [(0.1, 12)], 1e-6, "u", "z", relative=False)
    with pytest.raises(parity.ParityError, match="exact tie"):
        parity.check_swaps(kept, [(0.1, 4)], 1e-6, "u", "z", relative=False)
    with pytest.raises(parity.ParityError, match="not a near-tie"):
        parity.check_swaps(kept, [(0.2, 15)], 1e-6, "u", "z", relative=False)
