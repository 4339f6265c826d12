"""The LayerNorm GEMM epilogue over thread-block clusters (fe_gemm.cu) against the
oracle.  Rows wider than 128 columns (d = 512 for the summarisation shape,
d = 256 for the stress shape) with fewer row tiles than SMs are split over a
cluster of 2 to 8 CTAs that exchange the row sums through distributed shared
memory (the residual + LayerNorm steps of Sections 4.2-4.4).  Each case runs in
a child process, since the cluster setting is read once per process:
FE_GEMM_CLUSTERS=0 takes the single-CTA wide-row path, 1 and 2 cap a launch at
one or two resident clusters so that every cluster walks several row tiles
(both accumulators and both phases of the exchange barriers), and unset is the
default sizing."""
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
import json, sys
import numpy as np
import torch
from paper_2603_02565_gb300 import workloads as wl
from paper_2603_02565_gb300.binding import Evaluator
kind, B, out = sys.argv[1], int(sys.argv[2]), sys.argv[3]
w = wl.summarisation(B=B) if kind == "summarisation" else wl.make_workload(kind, B=B)
ev = Evaluator(w.cfg, w.weights)
ev.keep_intermediates(True)
dev = torch.device("cuda:0")
dt = torch.bfloat16 if w.cfg.io_bf16 else torch.float32
ctx = torch.from_numpy(w.context).to(dev, dt)
pool = torch.from_numpy(w.pool).to(dev, dt)
idx = torch.from_numpy(np.ascontiguousarray(w.cand_idx)).to(dev)
s, b = ev.evaluate(ctx, pool, idx)
np.savez(out, s=s.cpu().numpy(), b=b.cpu().numpy(), elem=ev.fetch("elem"), seq=ev.fetch("seq"))
"""


@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2603_02565_gb300 import build
    build.build()
    return torch.device("cuda:0")


def run_child(kind, B, clusters, tmp_path):
    env = dict(os.environ)
    env.pop("FE_GEMM_CLUSTERS", None)
    if clusters is not None:
        env["FE_GEMM_CLUSTERS"] = str(clusters)
    out = str(tmp_path / f"{kind}_{B}_{clusters}.npz")
    r = subprocess.run([sys.executable, "-c", CHILD, kind, str(B), out], cwd=ROOT, env=env,
                       capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    return np.load(out)


def oracle_intermediates(w):
    cfg, W = w.cfg, w.weights
    eps = cfg.ln_eps
    elem, seq = [], []
    for b in range(w.shape[0]):
        kv = O.context_kv(w.context[b], W, cfg.n_layers, eps)
        uniq, slots = O.distinct_layout(w.cand_idx[b])
        Hb = O.encode_elements(w.pool[b][uniq], kv, W, cfg.n_heads, eps)
        elem.append(Hb)
        seq.append(np.vstack([O.seq_encode(Hb[slots[k]], W, cfg.n_heads, eps) for k in range(w.shape[3])]))
    return np.vstack(elem), np.vstack(seq)


@pytest.fixture(scope="module")
def summ():
    """Three requests: ten element row tiles (clusters of 4 x 128 columns), one
    SeqEnc / cross-sequence row tile (8 x 64); the oracle runs once."""
    w = wl.summarisation(B=3)
    o_s, o_b, _, _ = O.evaluate(w.context, w.pool, w.cand_idx, w.weights, w.cfg)
    elem, seq = oracle_intermediates(w)
    return w, o_s, o_b, elem, seq


@pytest.mark.parametrize("clusters", [None, 0, 1, 2])
def test_summarisation_clusters(dev, summ, clusters, tmp_path):
    """d = 512: element, SeqEnc and cross-sequence LayerNorm GEMMs."""
    w, o_s, o_b, elem, seq = summ
    g = run_child("summarisation", 3, clusters, tmp_path)
    err = compare.score_error(g["s"], o_s)
    ok, _ = compare.best_ok(g["b"], o_s, o_b)
    assert err <= compare.REL_TOL, f"max rel err {err:.3e}"
    assert ok
    np.testing.assert_allclose(g["elem"], elem, rtol=0, atol=5e-4)
    np.testing.assert_allclose(g["seq"], seq, rtol=1e-3, atol=2e-4)


@pytest.mark.parametrize("clusters", [0, 1])
def test_stress_clusters(dev, clusters, tmp_path):
    """d = 256: the cross-sequence LayerNorm GEMM, one CTA of 256 columns or
    clusters of 4 x 64 per row tile."""
    w = wl.make_workload("stress", B=3)
    g = run_child("stress", 3, clusters, tmp_path)
    o_s, o_b, _, _ = O.evaluate(w.context, w.pool, w.cand_idx, w.weights, w.cfg)
    err = compare.score_error(g["s"], o_s)
    ok, _ = compare.best_ok(g["b"], o_s, o_b)
    assert err <= compare.REL_TOL, f"max rel err {err:.3e}"
    assert ok
