"""Writes tiny_oracle.txt: the oracle's scores, best index and distinct-element
layout for the seeded tiny workload (B=1, C=16, d=32, 1 head, 1 layer, M=20,
K=4, L=5).  Calls only the oracle and the workload generator; rerun it only
when the oracle's arithmetic changes for a reason stated in the commit."""
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import oracle.fe_oracle as O  # noqa: E402
from paper_2603_02565_gb300 import workloads as wl  # noqa: E402


def main():
    w = wl.make_workload("tiny")
    s, best, U, slots = O.evaluate(w.context, w.pool, w.cand_idx, w.weights, w.cfg)
    out = os.path.join(os.path.dirname(os.path.abspath(__file__)), "tiny_oracle.txt")
    with open(out, "w") as f:
        f.write("# oracle output for the seeded tiny workload (tests/golden/make_golden.py)\n")
        f.write("scores " + " ".join(repr(float(x)) for x in s[0]) + "\n")
        f.write(f"best {int(best[0])}\n")
        f.write(f"U {int(U[0])}\n")
        f.write("cand_idx " + " ".join(str(int(x)) for x in w.cand_idx[0].ravel()) + "\n")
        f.write("slots " + " ".join(str(int(x)) for x in slots[0].ravel()) + "\n")


if __name__ == "__main__":
    main()
