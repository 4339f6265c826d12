"""Linear-attention context module (the online deployment's linear attention,
Appendix B.3; feature map elu(x) + 1 of Katharopoulos et al.).

CPU part: the oracle's linear attention is pinned by worked values of its
feature map, a brute-force kernel smoother on tiny inputs (explicit
normalised weights, no context state), its properties (positive weights
summing to one, so outputs are convex combinations of the values; linear in
the values; indifferent to the order of the context rows), and by a case
where it must agree with the pinned softmax model: a request whose context
rows are all equal, where both attentions return that row's value.
GPU part (marked gpu): the CUDA path against the oracle.
"""
import dataclasses
import math

import numpy as np
import pytest

import oracle.fe_oracle as O
from oracle import compare
from paper_2603_02565_gb300 import workloads as wl


def _small(seed=17, B=2, C=9, d=32, H=2, Ly=2, M=10, K=4, L=3, **kw):
    return wl.make_workload("serving", seed=seed, B=B, C=C, d=d, H=H, Ly=Ly, M=M, K=K, L=L,
                            linear_context_attn=True, **kw)


def test_feature_map_worked_values():
    x = np.array([0.0, 1.0, 2.5, math.log(0.5), math.log(0.25), -50.0])
    want = np.array([1.0, 2.0, 3.5, 0.5, 0.25, math.exp(-50.0)])
    np.testing.assert_allclose(O.elu_feature(x), want, rtol=1e-15, atol=0)


def test_matches_a_brute_force_kernel_smoother():
    """out_i = sum_c w_ic v_c with w_ic proportional to phi(q_i) . phi(k_c),
    written with explicit loops and its own feature map."""
    rng = np.random.default_rng(3)
    n, m, d, H = 3, 5, 8, 2
    q, k, v = rng.normal(size=(n, d)), rng.normal(size=(m, d)), rng.normal(size=(m, d))

    def feat(x):
        return [xx + 1.0 if xx > 0 else math.exp(xx) for xx in x]

    dh = d // H
    want = np.zeros((n, d))
    for h in range(H):
        c0 = h * dh
        for i in range(n):
            fq = feat(q[i, c0:c0 + dh])
            w = [sum(a * b for a, b in zip(fq, feat(k[c, c0:c0 + dh]))) for c in range(m)]
            tot = sum(w)
            for j in range(dh):
                want[i, c0 + j] = sum(w[c] * v[c, c0 + j] for c in range(m)) / tot
    np.testing.assert_allclose(O.linear_attention(q, k, v, H), want, rtol=1e-12, atol=1e-14)


def test_outputs_are_convex_combinations_linear_in_the_values():
    rng = np.random.default_rng(4)
    q, k, v = rng.normal(size=(6, 16)), rng.normal(size=(9, 16)), rng.normal(size=(9, 16))
    out = O.linear_attention(q, k, v, 2)
    assert (out <= v.max(axis=0) + 1e-12).all() and (out >= v.min(axis=0) - 1e-12).all()
    np.testing.assert_allclose(O.linear_attention(q, k, 3.0 * v - 1.0, 2), 3.0 * out - 1.0, rtol=1e-12, atol=1e-12)
    perm = rng.permutation(9)
    np.testing.assert_allclose(O.linear_attention(q, k[perm], v[perm], 2), out, rtol=1e-12, atol=1e-14)


def test_equal_context_rows_make_it_the_softmax_model():
    """All context rows of a request equal: both attentions return that
    row's value, so the linear model's scores are the pinned softmax model's."""
    w = _small()
    ctx = np.repeat(w.context[:, :1], w.context.shape[1], axis=1)
    soft = dataclasses.replace(w.cfg, linear_context_attn=False)
    s_lin, b_lin, _, _ = O.evaluate(ctx, w.pool, w.cand_idx, w.weights, w.cfg)
    s_soft, b_soft, _, _ = O.evaluate(ctx, w.pool, w.cand_idx, w.weights, soft)
    np.testing.assert_allclose(s_lin, s_soft, rtol=1e-10, atol=1e-13)
    np.testing.assert_array_equal(b_lin, b_soft)
    s_gen, _, _, _ = O.evaluate(w.context, w.pool, w.cand_idx, w.weights, w.cfg)
    s_gen_soft, _, _, _ = O.evaluate(w.context, w.pool, w.cand_idx, w.weights, soft)
    assert np.abs(s_gen - s_gen_soft).max() > 1e-9  # with distinct rows they differ


def test_context_row_order_does_not_matter():
    w = _small(C=11)
    perm = np.random.default_rng(8).permutation(11)
    s0, _, _, _ = O.evaluate(w.context, w.pool, w.cand_idx, w.weights, w.cfg)
    s1, _, _, _ = O.evaluate(w.context[:, perm], w.pool, w.cand_idx, w.weights, w.cfg)
    np.testing.assert_allclose(s1, s0, rtol=1e-11, atol=1e-14)


def test_reuse_equals_no_reuse_with_linear_attention():
    w = _small(B=2, K=3, L=3, M=8)
    a, _, _, _ = O.evaluate(w.context, w.pool, w.cand_idx, w.weights, w.cfg, mode="reuse")
    b, _, _, _ = O.evaluate(w.context, w.pool, w.cand_idx, w.weights, w.cfg, mode="no_reuse")
    np.testing.assert_allclose(a, b, rtol=1e-9, atol=1e-12)


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


def _gpu(w, dev, factorized=False):
    from paper_2603_02565_gb300.binding import Evaluator
    ev = Evaluator(w.cfg, w.weights)
    dt = torch.bfloat16 if w.cfg.io_bf16 else torch.float32
    ctx = torch.from_numpy(w.context).to(dev, dt)
    pool = torch.from_numpy(w.pool).to(dev, dt)
    idx = torch.from_numpy(np.ascontiguousarray(w.cand_idx)).to(dev)
    s, b = ev.evaluate(ctx, pool, idx, factorized=factorized)
    return ev, s.cpu().numpy(), b.cpu().numpy()


def _check(w, gs, gb):
    o_s, o_b, _, _ = O.evaluate(w.context, w.pool, w.cand_idx, w.weights, w.cfg)
    err = compare.score_error(gs, o_s)
    assert err <= compare.REL_TOL, f"max rel err {err:.3e}"
    ok, exact = compare.best_ok(gb, o_s, o_b)
    assert ok, f"best index mismatch beyond near-ties (exact {exact:.3f})"


@pytest.mark.gpu
@pytest.mark.parametrize("kw", [
    dict(),                                                   # serving shape, d_h = 32
    dict(d=128, H=2, C=200),                                  # d_h = 64
    dict(d=64, H=2, C=1000, M=60, K=50, L=6),                 # the online setting: 1,000 interactions, pool 60
    dict(elem_self_attn=True, n_tasks=2),
])
def test_linear_context_attention_matches_the_oracle(dev, kw):
    p = dict(seed=41, B=3, C=256, d=128, H=4, Ly=2, M=100, K=50, L=6)
    p.update(kw)
    w = wl.make_workload("serving", linear_context_attn=True, **p)
    ev, gs, gb = _gpu(w, dev)
    _check(w, gs, gb)


@pytest.mark.gpu
def test_linear_context_attention_unfused_context_path(dev):
    """fp32 inputs take the unfused context path (row-major K/V)."""
    w = wl.make_workload("tiny", seed=5)
    w.cfg = dataclasses.replace(w.cfg, linear_context_attn=True)
    ev, gs, gb = _gpu(w, dev)
    _check(w, gs, gb)


@pytest.mark.gpu
def test_linear_factorized_matches_joint(dev):
    w = wl.make_workload("serving", seed=42, B=2, C=256, M=40, K=12, L=5, linear_context_attn=True)
    _, gs, gb = _gpu(w, dev)
    _, fs, fb = _gpu(w, dev, factorized=True)
    np.testing.assert_allclose(fs, gs, rtol=1e-4, atol=1e-6)
    np.testing.assert_array_equal(fb, gb)
