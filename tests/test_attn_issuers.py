"""The two issuer forms of the flash-attention kernel (fe_attn.cu) against the
oracle.  A launch whose CTAs each walk many key chunks issues S = Q K^T and
PV = P V from two threads; a short launch keeps one issuer.  The choice is made
per launch from the chunk count, so the default runs of the small test shapes
take one form only; FE_ATTN_SPLIT=0 / 1 forces one or the other for d_h = 32
(read once per process, hence one child process per case).  The shapes cover
element -> context attention over fixed-length contexts (Section 4.2) and the
cross-sequence attention over K sequences (Section 4.4) with a partial last
chunk (K = 1000 and K = 200 are not multiples of the 64-key chunk), whose V
rows past the key count the PV issuer zeroes.  The stress batch of 24 requests
gives each CTA several units, some of them query tiles past their request's
distinct elements (skipped), so the unit cursor's stride arithmetic and the
role-warp rotation of the second CTA on an SM run in both forms; three of its
requests are checked."""
import os
import subprocess
import sys

import numpy as np
import pytest

import oracle.fe_oracle as O
from oracle import compare
from paper_2603_02565_gb300 import workloads as wl

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r"""
import sys
import numpy as np
import torch
from paper_2603_02565_gb300 import workloads as wl
from paper_2603_02565_gb300.binding import Evaluator
kind, B, K, out = sys.argv[1], int(sys.argv[2]), int(sys.argv[3]), sys.argv[4]
w = wl.make_workload(kind, B=B, K=K) if K > 0 else wl.make_workload(kind, B=B)
ev = Evaluator(w.cfg, w.weights)
dev = torch.device("cuda:0")
dt = torch.bfloat16 if w.cfg.io_bf16 else torch.float32
ctx = torch.from_numpy(w.context).to(dev, dt)
pool = torch.from_numpy(w.pool).to(dev, dt)
idx = torch.from_numpy(np.ascontiguousarray(w.cand_idx)).to(dev)
s, b = ev.evaluate(ctx, pool, idx)
np.savez(out, s=s.cpu().numpy(), b=b.cpu().numpy())
"""

# name: (workload, B, K (0: the workload's own), requests checked (None: all))
CASES = {"serving": ("serving", 4, 0, None), "ksweep_K1000": ("ksweep", 2, 1000, None),
         "stress": ("stress", 3, 0, None), "stress24": ("stress", 24, 0, [0, 11, 23])}


@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2603_02565_gb300 import build
    build.build()
    return torch.device("cuda:0")


_oracle = {}


def oracle_scores(case):
    if case not in _oracle:
        kind, B, K, rq = CASES[case]
        w = wl.make_workload(kind, B=B, K=K) if K > 0 else wl.make_workload(kind, B=B)
        o_s, o_b, _, _ = O.evaluate(w.context, w.pool, w.cand_idx, w.weights, w.cfg, requests=rq)
        _oracle[case] = (o_s, o_b)
    return _oracle[case]


@pytest.mark.parametrize("split", [0, 1])
@pytest.mark.parametrize("case", sorted(CASES))
def test_attention_issuer_forms(dev, case, split, tmp_path):
    kind, B, K, rq = CASES[case]
    env = dict(os.environ)
    env["FE_ATTN_SPLIT"] = str(split)
    out = str(tmp_path / f"{case}_{split}.npz")
    r = subprocess.run([sys.executable, "-c", CHILD, kind, str(B), str(K), out], cwd=ROOT, env=env,
                       capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    g = np.load(out)
    o_s, o_b = oracle_scores(case)
    rq = list(range(B)) if rq is None else rq
    err = compare.score_error(g["s"][rq], o_s[rq])
    ok, _ = compare.best_ok(g["b"][rq], o_s[rq], o_b[rq])
    assert err <= compare.REL_TOL, f"max rel err {err:.3e}"
    assert ok
