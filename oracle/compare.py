"""Parity criteria between the CUDA path and the oracle (test infrastructure).

Scores: err = max over (b, k) of |g - o| / max(|o|, 1e-3) must be <= 2e-2
(relative error with an absolute floor of 1e-3 on the denominator).

Best index: exact match, or -- for near-ties -- the oracle score of the GPU's
choice is within tau_b = 2e-2 * max(|o_best|, 1e-3) of the oracle maximum.
"""
from __future__ import annotations

import numpy as np

REL_TOL = 2e-2
ABS_FLOOR = 1e-3


def score_error(gpu_scores, oracle_scores) -> float:
    g = np.asarray(gpu_scores, dtype=np.float64)
    o = np.asarray(oracle_scores, dtype=np.float64)
    if g.size == 0:
        return 0.0
    both_nan = np.isnan(g) & np.isnan(o)
    if (np.isnan(g) != np.isnan(o)).any():
        return float("inf")
    e = np.abs(g - o) / np.maximum(np.abs(o), ABS_FLOOR)
    e[both_nan] = 0.0
    return float(e.max())


def best_ok(gpu_best, oracle_scores, oracle_best):
    """(all_ok, exact_fraction)."""
    gb = np.asarray(gpu_best)
    ob = np.asarray(oracle_best)
    o = np.asarray(oracle_scores, dtype=np.float64)
    ok = []
    for b in range(len(ob)):
        if ob[b] < 0 or gb[b] < 0:
            ok.append(gb[b] == ob[b])
            continue
        top = o[b, ob[b]]
        tau = REL_TOL * max(abs(top), ABS_FLOOR)
        ok.append(gb[b] == ob[b] or (0 <= gb[b] < o.shape[1] and o[b, gb[b]] >= top - tau))
    exact = float(np.mean(gb == ob)) if len(ob) else 1.0
    return bool(all(ok)), exact
