"""Pins for the CPU oracle: library routines, closed forms, invariants of
Sections 4.1-4.4 and brute force on tiny inputs.  No GPU needed."""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle.fe_oracle as O
from paper_2603_02565_gb300 import workloads as wl
from tests.torch_modules_model import TorchEvaluator


def micro_case(seed, d=8, H=2, Ly=1, C=5, M=7, K=4, L=3, std=0.3, io_bf16=False):
    """Small random case with weights large enough that every term matters."""
    rng = np.random.default_rng(seed)
    cfg = wl.ModelConfig(d=d, n_heads=H, n_layers=Ly, max_L=L, io_bf16=io_bf16)
    W = wl.make_weights(cfg, rng, std=std)
    ctx = rng.normal(size=(1, C, d)).astype(np.float32)
    pool = rng.normal(size=(1, M, d)).astype(np.float32)
    cand = wl.sample_sequences(rng, 1, M, K, L)
    return cfg, W, ctx, pool, cand


# -- LayerNorm ---------------------------------------------------------------

def test_layer_norm_matches_library():
    x = np.random.default_rng(0).normal(size=(6, 13)) * 3 + 1
    ref = F.layer_norm(torch.as_tensor(x), (13,), eps=1e-5).numpy()
    np.testing.assert_allclose(O.layer_norm(x, 1e-5), ref, rtol=1e-12, atol=1e-12)


def test_layer_norm_two_values_closed_form():
    # x = [a, b]: mean (a+b)/2, biased var ((a-b)/2)^2
    a, b, eps = 3.0, -1.0, 1e-5
    half = (a - b) / 2
    v = half / math.sqrt(half * half + eps)
    np.testing.assert_allclose(O.layer_norm(np.array([a, b]), eps), [v, -v], rtol=1e-14)


def test_layer_norm_shift_and_scale_invariant():
    x = np.random.default_rng(1).normal(size=(4, 32))
    np.testing.assert_allclose(O.layer_norm(x * 7.0 + 5.0, 0.0), O.layer_norm(x, 0.0), atol=1e-12)
    y = O.layer_norm(x, 0.0)
    np.testing.assert_allclose(y.mean(-1), 0, atol=1e-13)
    np.testing.assert_allclose((y ** 2).mean(-1), 1, atol=1e-12)


# -- softmax / multi-head attention ------------------------------------------

def test_softmax_two_logits_is_logistic():
    a, b = 0.7, -1.9
    p = O.softmax(np.array([a, b]))
    s = 1.0 / (1.0 + math.exp(-(a - b)))
    np.testing.assert_allclose(p, [s, 1 - s], rtol=1e-12, atol=1e-15)
    # invariant to a common shift, including huge values (max subtraction)
    np.testing.assert_allclose(O.softmax(np.array([a, b]) + 1000.0), p, rtol=1e-12)


def test_mha_hand_example():
    # one head, d = 2, scale 1/sqrt(2): logits [1/sqrt 2, 0]
    q = np.array([[1.0, 0.0]])
    k = np.array([[1.0, 0.0], [0.0, 1.0]])
    v = np.array([[1.0, 2.0], [3.0, 4.0]])
    p = 1.0 / (1.0 + math.exp(-1.0 / math.sqrt(2.0)))  # 0.66976...
    assert abs(p - 0.6697615493266569) < 1e-15
    np.testing.assert_allclose(O.mha(q, k, v, 1), [[p * 1 + (1 - p) * 3, p * 2 + (1 - p) * 4]],
                               rtol=1e-14)


def test_mha_two_heads_use_separate_column_blocks():
    # head 0 sees columns 0-1, head 1 columns 2-3; a key that only differs in
    # head-1 columns must not change head-0 output
    rng = np.random.default_rng(3)
    q, k, v = rng.normal(size=(3, 4)), rng.normal(size=(5, 4)), rng.normal(size=(5, 4))
    k2 = k.copy()
    k2[:, 2:] += rng.normal(size=(5, 2))
    a, b = O.mha(q, k, v, 2), O.mha(q, k2, v, 2)
    np.testing.assert_allclose(a[:, :2], b[:, :2], rtol=1e-14)
    assert np.abs(a[:, 2:] - b[:, 2:]).max() > 1e-3


def test_mha_identical_keys_average_values():
    rng = np.random.default_rng(2)
    q = rng.normal(size=(3, 8))
    k = np.tile(rng.normal(size=(1, 8)), (6, 1))
    v = rng.normal(size=(6, 8))
    np.testing.assert_allclose(O.mha(q, k, v, 2), np.tile(v.mean(0), (3, 1)), rtol=1e-13)


@pytest.mark.parametrize("H", [1, 2, 4])
def test_mha_matches_library(H):
    rng = np.random.default_rng(10 + H)
    d = 8
    xq, xk = rng.normal(size=(5, d)), rng.normal(size=(7, d))
    WQ, WK, WV, WO = (rng.normal(size=(d, d)) * 0.5 for _ in range(4))
    mod = torch.nn.MultiheadAttention(d, H, bias=False, batch_first=True, dtype=torch.float64)
    with torch.no_grad():
        mod.in_proj_weight.copy_(torch.as_tensor(np.concatenate([WQ.T, WK.T, WV.T], 0)))
        mod.out_proj.weight.copy_(torch.as_tensor(WO.T))
    ref = mod(torch.as_tensor(xq)[None], torch.as_tensor(xk)[None], torch.as_tensor(xk)[None],
              need_weights=False)[0][0].detach().numpy()
    got = O.mha(xq @ WQ, xk @ WK, xk @ WV, H) @ WO
    np.testing.assert_allclose(got, ref, rtol=1e-11, atol=1e-12)


# -- element encoder (Section 4.2) --------------------------------------------

def test_zero_query_attention_is_context_mean():
    """W_Q = 0 makes every logit 0, so cross-attention returns the mean of V;
    with W1 = 0 and b1 = 0 the FFN adds only b2."""
    cfg, W, ctx, pool, cand = micro_case(5, Ly=1)
    W = dict(W)
    W["WQ.0"] = np.zeros_like(W["WQ.0"])
    W["W1.0"] = np.zeros_like(W["W1.0"])
    W["b1.0"] = np.zeros_like(W["b1.0"])
    kv = O.context_kv(ctx[0], W, 1, cfg.ln_eps)
    h0 = pool[0, :3].astype(np.float64)
    got = O.encode_elements(h0, kv, W, cfg.n_heads, cfg.ln_eps)
    X = O.layer_norm(ctx[0], cfg.ln_eps)
    h1 = h0 + (X.mean(0) @ W["WV.0"]) @ W["WO.0"] + W["b2.0"]
    np.testing.assert_allclose(got, O.layer_norm(h1, cfg.ln_eps), rtol=1e-11, atol=1e-12)


def test_context_rows_are_a_set():
    cfg, W, ctx, pool, cand = micro_case(6, Ly=2)
    perm = np.random.default_rng(0).permutation(ctx.shape[1])
    a = O.evaluate(ctx, pool, cand, W, cfg)[0]
    b = O.evaluate(ctx[:, perm], pool, cand, W, cfg)[0]
    np.testing.assert_allclose(a, b, rtol=1e-11)


def test_element_encoding_is_row_independent():
    cfg, W, ctx, pool, cand = micro_case(7, Ly=2)
    kv = O.context_kv(ctx[0], W, 2, cfg.ln_eps)
    allrows = O.encode_elements(pool[0], kv, W, cfg.n_heads, cfg.ln_eps)
    for m in range(pool.shape[1]):
        one = O.encode_elements(pool[0, [m]], kv, W, cfg.n_heads, cfg.ln_eps)
        np.testing.assert_allclose(one[0], allrows[m], rtol=1e-12, atol=1e-13)


# -- reuse (Sections 4.2, 5.2) -------------------------------------------------

@pytest.mark.parametrize("seed", range(4))
def test_reuse_equals_no_reuse(seed):
    cfg, W, ctx, pool, cand = micro_case(20 + seed, Ly=2, K=5, L=3, M=6)
    a = O.evaluate(ctx, pool, cand, W, cfg, mode="reuse")
    b = O.evaluate(ctx, pool, cand, W, cfg, mode="no_reuse")
    np.testing.assert_allclose(a[0], b[0], rtol=1e-11, atol=1e-13)
    assert (a[1] == b[1]).all()


def test_reuse_equals_no_reuse_tiny_workload():
    w = wl.make_workload("tiny")
    a = O.evaluate(w.context, w.pool, w.cand_idx, w.weights, w.cfg, mode="reuse")
    b = O.evaluate(w.context, w.pool, w.cand_idx, w.weights, w.cfg, mode="no_reuse")
    np.testing.assert_allclose(a[0], b[0], rtol=1e-11, atol=1e-14)


def test_duplicated_occurrence_keeps_element_representation():
    """Overwriting one occurrence with an element already present elsewhere
    leaves every element representation unchanged (it is computed once per
    distinct element and only conditioned on the request context)."""
    cfg, W, ctx, pool, cand = micro_case(8, Ly=2, K=4, L=3, M=9)
    kv = O.context_kv(ctx[0], W, 2, cfg.ln_eps)
    uniq, _ = O.distinct_layout(cand[0])
    before = O.encode_elements(pool[0][uniq], kv, W, cfg.n_heads, cfg.ln_eps)
    cand2 = cand.copy()
    cand2[0, 0, 0] = cand[0, 1, 1]
    uniq2, _ = O.distinct_layout(cand2[0])
    after = O.encode_elements(pool[0][uniq2], kv, W, cfg.n_heads, cfg.ln_eps)
    for i, m in enumerate(uniq2):
        np.testing.assert_allclose(after[i], before[list(uniq).index(m)], rtol=1e-12, atol=1e-13)


# -- assembly / SeqEnc (Section 4.3) -------------------------------------------

def test_without_positions_sequence_order_does_not_matter():
    cfg, W, ctx, pool, cand = micro_case(9, K=3, L=4, M=8)
    W = dict(W)
    W["P"] = np.zeros_like(W["P"])
    cand2 = cand[:, :, ::-1].copy()
    np.testing.assert_allclose(O.evaluate(ctx, pool, cand, W, cfg)[0],
                               O.evaluate(ctx, pool, cand2, W, cfg)[0], rtol=1e-11)


def test_positions_are_added_after_indexing():
    """With positions, reversing a sequence changes its representation; the
    reversed sequence equals the original one scored with a reversed table."""
    cfg, W, ctx, pool, cand = micro_case(11, K=3, L=4, M=8)
    a = O.evaluate(ctx, pool, cand, W, cfg)[0]
    cand2 = cand[:, :, ::-1].copy()
    b = O.evaluate(ctx, pool, cand2, W, cfg)[0]
    assert np.abs(a - b).max() > 1e-6
    W2 = dict(W)
    W2["P"] = W["P"][:4][::-1].copy()
    np.testing.assert_allclose(O.evaluate(ctx, pool, cand2, W2, cfg)[0], a, rtol=1e-11)


def test_seqenc_single_element_closed_form():
    """L = 1: the [CLS] query sees two keys, so each head's weight on the
    element is the logistic function of the logit difference."""
    rng = np.random.default_rng(12)
    d, H = 8, 2
    cfg = wl.ModelConfig(d=d, n_heads=H, n_layers=1, max_L=1, io_bf16=False)
    W = wl.make_weights(cfg, rng, std=0.4)
    r = rng.normal(size=(1, d))
    got = O.seq_encode(r, W, H, cfg.ln_eps)
    cls, x1 = W["cls"].astype(np.float64), r[0] + W["P"][0]
    q, k0, k1 = cls @ W["WQs"], cls @ W["WKs"], x1 @ W["WKs"]
    v0, v1 = cls @ W["WVs"], x1 @ W["WVs"]
    dh = d // H
    o = np.empty(d)
    for h in range(H):
        s = slice(h * dh, (h + 1) * dh)
        w1 = 1.0 / (1.0 + math.exp(-(q[s] @ k1[s] - q[s] @ k0[s]) / math.sqrt(dh)))
        o[s] = (1 - w1) * v0[s] + w1 * v1[s]
    c = cls + o @ W["WOs"]
    mu, var = c.mean(), c.var()
    z = (c - mu) / math.sqrt(var + cfg.ln_eps)
    c = c + np.maximum(z @ W["W1s"] + W["b1s"], 0) @ W["W2s"] + W["b2s"]
    np.testing.assert_allclose(got, c, rtol=1e-12, atol=1e-13)


# -- cross-sequence interaction and head (Section 4.4, Eq. 1) --------------------

def test_permuting_candidates_permutes_scores():
    cfg, W, ctx, pool, cand = micro_case(13, K=6, L=3, M=8)
    perm = np.random.default_rng(1).permutation(6)
    s, best = O.evaluate(ctx, pool, cand, W, cfg)[:2]
    s2, best2 = O.evaluate(ctx, pool, cand[:, perm], W, cfg)[:2]
    np.testing.assert_allclose(s2[0], s[0][perm], rtol=1e-11)
    assert perm[best2[0]] == best[0]


def test_single_candidate_cross_attention_closed_form():
    """K = 1: softmax over one key is 1, so C' = C + LN(C) W_Vx W_Ox."""
    rng = np.random.default_rng(14)
    cfg = wl.ModelConfig(d=8, n_heads=2, n_layers=1, max_L=2, io_bf16=False)
    W = wl.make_weights(cfg, rng, std=0.4)
    Cm = rng.normal(size=(1, 8))
    Z = O.layer_norm(Cm, cfg.ln_eps)
    np.testing.assert_allclose(O.cross_sequence(Cm, W, 2, cfg.ln_eps),
                               Cm + Z @ W["WVx"] @ W["WOx"], rtol=1e-12)


def test_zero_parameters_give_constant_scores_and_first_index():
    cfg, W, ctx, pool, cand = micro_case(15, K=5)
    Z = {k: np.zeros_like(v) for k, v in W.items()}
    Z["b2h"] = np.array([0.375], dtype=np.float32)
    s, best = O.evaluate(ctx, pool, cand, Z, cfg)[:2]
    np.testing.assert_array_equal(s, np.full_like(s, 0.375))
    assert best[0] == 0


def test_head_bias_shifts_every_score():
    cfg, W, ctx, pool, cand = micro_case(16)
    s = O.evaluate(ctx, pool, cand, W, cfg)[0]
    W2 = dict(W)
    W2["b2h"] = W["b2h"].astype(np.float64) + 2.0
    np.testing.assert_allclose(O.evaluate(ctx, pool, cand, W2, cfg)[0], s + 2.0, rtol=1e-12)


def test_select_best_brute_force():
    rng = np.random.default_rng(17)
    for _ in range(200):
        s = rng.integers(0, 4, size=rng.integers(1, 9)).astype(np.float64)
        m = max(s)
        assert O.select_best(s) == min(i for i in range(len(s)) if s[i] == m)
    assert O.select_best(np.array([1.0, np.nan])) == -1


# -- layout -----------------------------------------------------------------------

def test_distinct_layout_brute_force():
    rng = np.random.default_rng(18)
    for _ in range(50):
        K, L, M = rng.integers(1, 8), rng.integers(1, 6), rng.integers(6, 30)
        cand = np.stack([rng.choice(M, L, replace=False) for _ in range(K)])
        uniq, slots = O.distinct_layout(cand)
        ref = sorted(set(int(x) for x in cand.ravel()))
        assert list(uniq) == ref
        for k in range(K):
            for j in range(L):
                assert ref[slots[k, j]] == cand[k, j]


def test_bad_index_isolates_request():
    cfg, W, ctx, pool, cand = micro_case(19, K=3, L=2, M=5)
    ctx2, pool2, cand2 = (np.concatenate([a, a]) for a in (ctx, pool, cand))
    cand2[1, 2, 1] = 5   # == M: out of range
    s, best, U, slots = O.evaluate(ctx2, pool2, cand2, W, cfg)
    assert np.isnan(s[1]).all() and best[1] == -1 and U[1] == 0
    np.testing.assert_allclose(s[0], O.evaluate(ctx, pool, cand, W, cfg)[0][0], rtol=1e-13)


def test_nan_input_isolates_request():
    """A NaN in one request's pool row or context row: that request's scores are
    NaN (the cross-sequence attention mixes every candidate) and Eq. 1 selects
    nothing (-1); the other request is untouched."""
    cfg, W, ctx, pool, cand = micro_case(23, K=3, L=2, M=5)
    for where in ("pool", "context"):
        ctx2, pool2, cand2 = (np.concatenate([a, a]) for a in (ctx, pool, cand))
        if where == "pool":
            pool2[1, cand2[1, 0, 0], 0] = np.nan
        else:
            ctx2[1, 0, 0] = np.nan
        s, best, U, slots = O.evaluate(ctx2, pool2, cand2, W, cfg)
        assert np.isnan(s[1]).all() and best[1] == -1 and U[1] == U[0]
        np.testing.assert_allclose(s[0], O.evaluate(ctx, pool, cand, W, cfg)[0][0], rtol=1e-13)


# -- the whole evaluator against stock torch.nn layers -----------------------------

@pytest.mark.parametrize("seed", range(40))
def test_oracle_matches_torch_modules(seed):
    rng = np.random.default_rng(1000 + seed)
    H = int(rng.choice([1, 2]))
    d = int(rng.choice([8, 16]))
    cfg, W, ctx, pool, cand = micro_case(
        2000 + seed, d=d, H=H, Ly=int(rng.integers(1, 3)), C=int(rng.integers(1, 9)),
        M=int(rng.integers(4, 11)), K=int(rng.integers(1, 6)), L=int(rng.integers(1, 5)))
    ref = TorchEvaluator(W, cfg)
    s, best = O.evaluate(ctx, pool, cand, W, cfg)[:2]
    rs = ref.scores(ctx[0], pool[0], cand[0])
    np.testing.assert_allclose(s[0], rs, rtol=1e-9, atol=1e-12)
    assert best[0] == ref.best(rs)


def test_oracle_matches_torch_modules_tiny_workload():
    w = wl.make_workload("tiny")
    s = O.evaluate(w.context, w.pool, w.cand_idx, w.weights, w.cfg)[0]
    rs = TorchEvaluator(w.weights, w.cfg).scores(w.context[0], w.pool[0], w.cand_idx[0])
    np.testing.assert_allclose(s[0], rs, rtol=1e-9, atol=1e-15)
