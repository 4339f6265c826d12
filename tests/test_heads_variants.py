"""Multi-objective task heads with fusion, and the variant without
cross-sequence interaction (end of Section 4.4; "- CrossSeq" of Appendix B.4).

CPU part: the oracle's new paths are pinned by reducing them to the already
pinned single-head, full model (closed forms that hold exactly in exact
arithmetic), and by the defining property of the "- CrossSeq" variant: a
sequence's score does not depend on the other sequences of its request.
GPU part (marked gpu): the CUDA path against the oracle for these variants.
"""
import dataclasses

import numpy as np
import pytest

import oracle.fe_oracle as O
from oracle import compare
from paper_2603_02565_gb300 import workloads as wl


def _small(n_tasks=1, cross_seq=True, seed=11, B=3, C=12, d=32, H=1, Ly=1, M=14, K=5, L=4):
    return wl.make_workload("serving", seed=seed, B=B, C=C, d=d, H=H, Ly=Ly, M=M, K=K, L=L,
                            n_tasks=n_tasks, cross_seq=cross_seq)


def _single_head_from(w, t):
    """The single-head model whose head is task t's head of w."""
    cfg1 = dataclasses.replace(w.cfg, n_tasks=1)
    W = {k: v for k, v in w.weights.items() if not (k.startswith(("W1h.", "b1h.", "w2h.", "b2h.")) or
                                                  k.startswith("fuse_"))}
    for n in ("W1h", "b1h", "w2h", "b2h"):
        W[n] = w.weights[f"{n}.{t}"]
    return cfg1, W


def test_identical_heads_averaged_equal_the_single_head():
    w1 = _small(n_tasks=1)
    cfg2 = dataclasses.replace(w1.cfg, n_tasks=2)
    W2 = {k: v for k, v in w1.weights.items() if k not in ("W1h", "b1h", "w2h", "b2h")}
    for t in range(2):
        for n in ("W1h", "b1h", "w2h", "b2h"):
            W2[f"{n}.{t}"] = w1.weights[n]
    W2["fuse_w"] = np.array([0.5, 0.5], np.float32)
    W2["fuse_b"] = np.zeros(1, np.float32)
    s1, b1, _, _ = O.evaluate(w1.context, w1.pool, w1.cand_idx, w1.weights, w1.cfg)
    s2, b2, _, _, st = O.evaluate(w1.context, w1.pool, w1.cand_idx, W2, cfg2, with_tasks=True)
    np.testing.assert_allclose(s2, s1, rtol=1e-12, atol=0)
    np.testing.assert_array_equal(st[..., 0], s1)
    np.testing.assert_array_equal(st[..., 1], s1)
    np.testing.assert_array_equal(b2, b1)


@pytest.mark.parametrize("t", [0, 1, 2])
def test_one_hot_fusion_selects_one_task_head(t):
    w = _small(n_tasks=3)
    W = dict(w.weights)
    W["fuse_w"] = np.eye(3, dtype=np.float32)[t]
    W["fuse_b"] = np.zeros(1, np.float32)
    s, b, _, _, st = O.evaluate(w.context, w.pool, w.cand_idx, W, w.cfg, with_tasks=True)
    cfg1, W1 = _single_head_from(w, t)
    s1, b1, _, _ = O.evaluate(w.context, w.pool, w.cand_idx, W1, cfg1)
    np.testing.assert_array_equal(s, s1)
    np.testing.assert_array_equal(st[..., t], s1)
    np.testing.assert_array_equal(b, b1)


def test_fusion_bias_shifts_every_score():
    w = _small(n_tasks=2)
    W = dict(w.weights)
    s0, _, _, _ = O.evaluate(w.context, w.pool, w.cand_idx, W, w.cfg)
    W["fuse_b"] = W["fuse_b"] + np.float32(0.25)
    s1, _, _, _ = O.evaluate(w.context, w.pool, w.cand_idx, W, w.cfg)
    np.testing.assert_allclose(s1 - s0, 0.25, rtol=0, atol=1e-12)


def test_zero_output_projection_equals_no_cross_block():
    full = _small(cross_seq=True)
    W = dict(full.weights)
    W["WOx"] = np.zeros_like(W["WOx"])
    nocross_cfg = dataclasses.replace(full.cfg, cross_seq=False)
    Wn = {k: v for k, v in W.items() if k not in ("WQx", "WKx", "WVx", "WOx")}
    s_full, b_full, _, _ = O.evaluate(full.context, full.pool, full.cand_idx, W, full.cfg)
    s_nc, b_nc, _, _ = O.evaluate(full.context, full.pool, full.cand_idx, Wn, nocross_cfg)
    np.testing.assert_array_equal(s_full, s_nc)
    np.testing.assert_array_equal(b_full, b_nc)


def test_no_cross_scores_are_independent_of_the_other_sequences():
    w = _small(cross_seq=False, B=2, K=6)
    s, _, _, _ = O.evaluate(w.context, w.pool, w.cand_idx, w.weights, w.cfg)
    for b in range(2):
        for k in range(6):
            alone = w.cand_idx[b:b + 1, k:k + 1]
            s1, _, _, _ = O.evaluate(w.context[b:b + 1], w.pool[b:b + 1], alone, w.weights, w.cfg)
            np.testing.assert_allclose(s1[0, 0], s[b, k], rtol=1e-12, atol=1e-15)


def test_with_cross_scores_do_depend_on_the_other_sequences():
    """The check above has teeth: with the cross-sequence block, scoring a
    sequence alone changes its score."""
    w = _small(cross_seq=True, B=1, K=6)
    s, _, _, _ = O.evaluate(w.context, w.pool, w.cand_idx, w.weights, w.cfg)
    s1, _, _, _ = O.evaluate(w.context, w.pool, w.cand_idx[:, :1], w.weights, w.cfg)
    assert abs(s1[0, 0] - s[0, 0]) > 1e-9


@pytest.mark.parametrize("n_tasks,cross_seq", [(3, True), (2, False)])
def test_reuse_equals_no_reuse_for_the_variants(n_tasks, cross_seq):
    w = _small(n_tasks=n_tasks, cross_seq=cross_seq, B=2)
    a = O.evaluate(w.context, w.pool, w.cand_idx, w.weights, w.cfg, mode="reuse", with_tasks=True)
    b = O.evaluate(w.context, w.pool, w.cand_idx, w.weights, w.cfg, mode="no_reuse", with_tasks=True)
    np.testing.assert_allclose(a[0], b[0], rtol=1e-9, atol=1e-12)
    np.testing.assert_allclose(a[4], b[4], rtol=1e-9, atol=1e-12)


@pytest.mark.parametrize("n_tasks,cross_seq", [(1, True), (3, True), (4, False), (1, False)])
def test_weight_count_matches_the_parameter_list(n_tasks, cross_seq):
    from paper_2603_02565_gb300 import binding
    try:
        L = binding.load_library()
    except ImportError:
        pytest.skip("library not built")
    cfg = wl.ModelConfig(d=128, n_heads=4, n_layers=2, max_L=6, n_tasks=n_tasks, cross_seq=cross_seq)
    c = binding.make_config(cfg)
    import ctypes
    n = L.fe_weight_count(ctypes.byref(c))
    assert n == sum(int(np.prod(s)) for _, s in wl.param_shapes(cfg))


def test_unsupported_head_widths_are_rejected():
    from paper_2603_02565_gb300 import binding
    try:
        L = binding.load_library()
    except ImportError:
        pytest.skip("library not built")
    import ctypes
    for n_tasks, d in ((5, 64), (3, 256), (2, 512)):
        c = binding.make_config(wl.ModelConfig(d=d, n_heads=d // 64, n_layers=1, n_tasks=n_tasks))
        assert L.fe_weight_count(ctypes.byref(c)) == 0


# ---------------------------------------------------------------- GPU parity
try:
    import torch
except ImportError:  # the CPU part above does not need it
    torch = None


@pytest.fixture(scope="module")
def dev():
    if torch is None or not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2603_02565_gb300 import build
    build.build()
    return torch.device("cuda:0")


def _gpu(w, dev):
    from paper_2603_02565_gb300.binding import Evaluator
    ev = Evaluator(w.cfg, w.weights)
    dt = torch.bfloat16 if w.cfg.io_bf16 else torch.float32
    ctx = torch.from_numpy(w.context).to(dev, dt)
    pool = torch.from_numpy(w.pool).to(dev, dt)
    idx = torch.from_numpy(np.ascontiguousarray(w.cand_idx)).to(dev)
    s, b = ev.evaluate(ctx, pool, idx)
    return ev, s.cpu().numpy(), b.cpu().numpy()


@pytest.mark.gpu
@pytest.mark.parametrize("n_tasks,cross_seq,kw", [
    (3, True, dict(B=5)),                      # 3 heads: 384 head columns padded to 512
    (4, True, dict(B=3)),                      # 4 heads: 512 columns
    (1, False, dict(B=5)),                     # single head without cross-sequence block
    (2, False, dict(B=4, K=40, L=10)),         # both
    (3, True, dict(B=2, d=64, H=2, M=60, K=33, L=7, C=100)),
])
def test_variants_match_the_oracle(dev, n_tasks, cross_seq, kw):
    p = dict(seed=21, B=4, C=256, d=128, H=4, Ly=2, M=100, K=50, L=6)
    p.update(kw)
    w = wl.make_workload("serving", n_tasks=n_tasks, cross_seq=cross_seq, **p)
    ev, gs, gb = _gpu(w, dev)
    o_s, o_b, _, _, o_t = O.evaluate(w.context, w.pool, w.cand_idx, w.weights, w.cfg, with_tasks=True)
    err = compare.score_error(gs, o_s)
    assert err <= compare.REL_TOL, f"fused scores: max rel err {err:.3e}"
    ok, exact = compare.best_ok(gb, o_s, o_b)
    assert ok, f"best index mismatch beyond near-ties (exact {exact:.3f})"
    B, K = gs.shape
    gt = ev.fetch("task_scores", cols=n_tasks).reshape(B, K, n_tasks)
    terr = compare.score_error(gt, o_t)
    assert terr <= compare.REL_TOL, f"task scores: max rel err {terr:.3e}"
    if not cross_seq:
        from paper_2603_02565_gb300.binding import FeError
        with pytest.raises(FeError):
            ev.fetch("cross", cols=w.cfg.d)
