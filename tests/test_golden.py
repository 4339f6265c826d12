"""The oracle still reproduces its stored output for the seeded tiny workload."""
import os

import numpy as np

import oracle.fe_oracle as O
from paper_2603_02565_gb300 import workloads as wl

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "tiny_oracle.txt")


def read_golden():
    out = {}
    for line in open(GOLDEN):
        if line.startswith("#"):
            continue
        k, *v = line.split()
        out[k] = v
    return out


def test_tiny_golden():
    g = read_golden()
    w = wl.make_workload("tiny")
    assert [int(x) for x in g["cand_idx"]] == w.cand_idx[0].ravel().tolist()
    s, best, U, slots = O.evaluate(w.context, w.pool, w.cand_idx, w.weights, w.cfg)
    np.testing.assert_allclose(s[0], [float(x) for x in g["scores"]], rtol=1e-12, atol=1e-15)
    assert int(g["best"][0]) == best[0] and int(g["U"][0]) == U[0]
    assert [int(x) for x in g["slots"]] == slots[0].ravel().tolist()
