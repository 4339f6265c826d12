"""Pins of the parity comparator (oracle/compare.py) on hand-computed cases.

Every GPU parity verdict goes through `score_error` (the score tolerance:
2e-2 maximum relative error with a 1e-3 floor on the denominator) and
`best_ok` (the best index of Eq. 1, with near-ties accepted when the oracle
score of the GPU's choice is within tau = 2e-2 * max(|o_best|, 1e-3) of the
oracle maximum; the smallest-index tie rule of Appendix B.1 is what makes
an exact match the normal case).  The expected values below are worked out
by hand from those definitions, not by calling the comparator.  The mutants
at the end are plausible slips of the same functions; each must fail at
least one pin, which shows that the pins can tell them apart.
"""
import math

import numpy as np
import pytest

from oracle import compare

TOL = 2e-2
FLOOR = 1e-3


# ----------------------------------------------------------------------------------------------
# hand-computed cases: (gpu, oracle, expected error)
# ----------------------------------------------------------------------------------------------
SCORE_CASES = [
    # |1.0196 - 1| / 1 = 0.0196: just inside the tolerance
    ([1.0196], [1.0], 0.0196),
    # 0.0204: just outside
    ([1.0204], [1.0], 0.0204),
    # below the floor the denominator is 1e-3: 1.9e-5 / 1e-3 = 0.019
    ([1e-4 + 1.9e-5], [1e-4], 0.019),
    # 2.1e-5 / 1e-3 = 0.021
    ([1e-4 + 2.1e-5], [1e-4], 0.021),
    # an oracle score of exactly zero: the floor alone, 5e-6 / 1e-3 = 5e-3
    ([5e-6], [0.0], 5e-3),
    # the denominator is |o| (negative scores): 0.01 / 0.5 = 0.02
    ([-0.51], [-0.5], 0.02),
    # the denominator is the oracle's score, not the GPU's: |2 - 1| / 1 = 1
    ([2.0], [1.0], 1.0),
    # the maximum over all (b, k), not a mean: the worst element is 0.1 / 1
    ([[1.0, 1.0], [1.0, 1.1]], [[1.0, 1.0], [1.0, 1.0]], 0.1),
    # |o| just above the floor uses |o| itself: 4e-5 / 2e-3 = 0.02
    ([2.04e-3], [2e-3], 0.02),
    # a NaN on one side only can never pass
    ([math.nan, 1.0], [1.0, 1.0], math.inf),
    ([1.0, 1.0], [1.0, math.nan], math.inf),
    # NaN on both sides at the same place (an isolated request) counts as equal;
    # the remaining element decides: 0.005 / 0.5 = 0.01
    ([[math.nan, math.nan], [0.505, 1.0]], [[math.nan, math.nan], [0.5, 1.0]], 0.01),
    # empty input (a batch of zero requests or K = 0)
    (np.zeros((0, 5)), np.zeros((0, 5)), 0.0),
]


@pytest.mark.parametrize("g,o,want", SCORE_CASES)
def test_score_error_hand_cases(g, o, want):
    got = compare.score_error(g, o)
    if math.isinf(want):
        assert math.isinf(got)
    else:
        assert got == pytest.approx(want, rel=1e-9, abs=1e-15)


def test_score_error_threshold_sides():
    # the same cases as verdicts against the tolerance
    assert compare.score_error([1.0196], [1.0]) <= compare.REL_TOL
    assert compare.score_error([1.0204], [1.0]) > compare.REL_TOL
    assert compare.score_error([1e-4 + 1.9e-5], [1e-4]) <= compare.REL_TOL
    assert compare.score_error([1e-4 + 2.1e-5], [1e-4]) > compare.REL_TOL
    assert compare.REL_TOL == TOL and compare.ABS_FLOOR == FLOOR


# ----------------------------------------------------------------------------------------------
# best index: (gpu best, oracle scores, oracle best, expected ok, expected exact fraction)
# ----------------------------------------------------------------------------------------------
BEST_CASES = [
    # exact match
    ([0], [[1.0, 0.985, 0.975]], [0], True, 1.0),
    # near-tie inside tau = 0.02 * 1.0: 0.985 >= 0.98
    ([1], [[1.0, 0.985, 0.975]], [0], True, 0.0),
    # just outside: 0.975 < 0.98
    ([2], [[1.0, 0.985, 0.975]], [0], False, 0.0),
    # negative maximum: tau = 0.02 * |-1| = 0.02; -1.015 >= -1.02
    ([1], [[-1.0, -1.015, -1.025]], [0], True, 0.0),
    ([2], [[-1.0, -1.015, -1.025]], [0], False, 0.0),
    # maximum below the floor: tau = 0.02 * 1e-3 = 2e-5; -0.9e-5 >= 1e-5 - 2e-5
    ([1], [[1e-5, -0.9e-5, -1.1e-5]], [0], True, 0.0),
    ([2], [[1e-5, -0.9e-5, -1.1e-5]], [0], False, 0.0),
    # the GPU's index out of range (3 with K = 3): rejected, not an IndexError
    ([3], [[1.0, 1.0, 1.0]], [0], False, 0.0),
    # -1 (no maximum) against a valid index, and the reverse
    ([-1], [[1.0, 0.5, 0.2]], [0], False, 0.0),
    ([0], [[math.nan, math.nan, math.nan]], [-1], False, 0.0),
    # -1 on both sides: an isolated request
    ([-1], [[math.nan, math.nan, math.nan]], [-1], True, 1.0),
    # two requests, one exact and one near-tie: all ok, exact fraction 1/2
    ([0, 2], [[3.0, 1.0, 2.0], [1.0, 0.5, 0.99]], [0, 0], True, 0.5),
    # one of two requests wrong makes the batch fail
    ([0, 1], [[3.0, 1.0, 2.0], [1.0, 0.5, 0.99]], [0, 0], False, 0.5),
]


@pytest.mark.parametrize("gb,o,ob,want_ok,want_exact", BEST_CASES)
def test_best_ok_hand_cases(gb, o, ob, want_ok, want_exact):
    ok, exact = compare.best_ok(np.array(gb), np.array(o, dtype=np.float64), np.array(ob))
    assert ok is want_ok
    assert exact == pytest.approx(want_exact)


def test_best_ok_reads_oracle_scores_of_the_gpu_choice():
    # tau is measured on the oracle's scores; the GPU's own scores play no part
    o = np.array([[1.0, 0.5]])
    assert compare.best_ok(np.array([1]), o, np.array([0])) == (False, 0.0)


# ----------------------------------------------------------------------------------------------
# plausible slips of the comparator: each one must fail a pin above
# ----------------------------------------------------------------------------------------------
def _score_mutant(kind):
    def f(gpu_scores, oracle_scores):
        g = np.asarray(gpu_scores, dtype=np.float64)
        o = np.asarray(oracle_scores, dtype=np.float64)
        if g.size == 0:
            return 0.0
        both = np.isnan(g) & np.isnan(o)
        if kind != "nan_ignored" and (np.isnan(g) != np.isnan(o)).any():
            return float("inf")
        floor = {"floor_one": 1.0, "no_floor": 0.0}.get(kind, FLOOR)
        den = {"signed_den": np.maximum(o, floor), "gpu_den": np.maximum(np.abs(g), floor),
               "min_den": np.minimum(np.abs(o), 1.0)}.get(kind, np.maximum(np.abs(o), floor))
        with np.errstate(divide="ignore", invalid="ignore"):
            e = np.abs(g - o) / den
        e[both] = 0.0
        e = np.where(np.isnan(e), 0.0, e) if kind == "nan_ignored" else e
        return float(e.mean() if kind == "mean" else e.max())
    return f


def _best_mutant(kind):
    def f(gpu_best, oracle_scores, oracle_best):
        gb, ob = np.asarray(gpu_best), np.asarray(oracle_best)
        o = np.asarray(oracle_scores, dtype=np.float64)
        ok = []
        for b in range(len(ob)):
            if ob[b] < 0 or gb[b] < 0:
                ok.append(gb[b] == ob[b])
                continue
            top = o[b, ob[b]]
            tau = {"signed_tau": TOL * max(top, FLOOR), "no_floor": TOL * abs(top),
                   "tau_10x": 10 * TOL * max(abs(top), FLOOR)}.get(kind, TOL * max(abs(top), FLOOR))
            if kind == "no_range_check":
                ok.append(gb[b] == ob[b] or o[b, gb[b] % o.shape[1]] >= top - tau)
            else:
                ok.append(gb[b] == ob[b] or (0 <= gb[b] < o.shape[1] and o[b, gb[b]] >= top - tau))
        return bool(all(ok)), float(np.mean(gb == ob)) if len(ob) else 1.0
    return f


def _score_pins_pass(fn):
    for g, o, want in SCORE_CASES:
        got = fn(g, o)
        if math.isinf(want):
            if not math.isinf(got):
                return False
        elif not (abs(got - want) <= 1e-9 * abs(want) + 1e-15):
            return False
    return True


def _best_pins_pass(fn):
    for gb, o, ob, want_ok, want_exact in BEST_CASES:
        ok, exact = fn(np.array(gb), np.array(o, dtype=np.float64), np.array(ob))
        if ok is not want_ok or abs(exact - want_exact) > 1e-12:
            return False
    return True


def test_pins_accept_the_comparator():
    assert _score_pins_pass(compare.score_error)
    assert _best_pins_pass(compare.best_ok)


@pytest.mark.parametrize("kind", ["floor_one", "no_floor", "signed_den", "gpu_den", "min_den", "mean", "nan_ignored"])
def test_pins_reject_score_error_slips(kind):
    assert not _score_pins_pass(_score_mutant(kind))


@pytest.mark.parametrize("kind", ["signed_tau", "no_floor", "tau_10x", "no_range_check"])
def test_pins_reject_best_ok_slips(kind):
    assert not _best_pins_pass(_best_mutant(kind))
