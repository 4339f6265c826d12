"""Element self-attention H^(1) over the request's element set (Section 4.2),
and the whole-pool element set U(z) = C(x), U = M (Section 4.1).

CPU part: the oracle's H^(1) block is pinned by a zero output projection
(reduces to the pinned model), a closed form (identical elements attend to
identical keys and values), invariance to the order of the pool rows, and
the set semantics (with U(z) the set couples the sequences of a request; with
the whole pool and no cross-sequence block it does not).  GPU part (marked
gpu): the CUDA path against the oracle.
"""
import dataclasses

import numpy as np
import pytest

import oracle.fe_oracle as O
from oracle import compare
from paper_2603_02565_gb300 import workloads as wl


def _small(seed=13, B=2, C=10, d=32, H=2, Ly=1, M=12, K=4, L=3, **kw):
    return wl.make_workload("serving", seed=seed, B=B, C=C, d=d, H=H, Ly=Ly, M=M, K=K, L=L, **kw)


def _ev(w, cfg=None, W=None, cand=None, pool=None, **kw):
    return O.evaluate(w.context, w.pool if pool is None else pool, w.cand_idx if cand is None else cand,
                      w.weights if W is None else W, w.cfg if cfg is None else cfg, **kw)


def test_zero_output_projection_is_the_model_without_it():
    w = _small(elem_self_attn=True)
    W = dict(w.weights)
    W["WOe"] = np.zeros_like(W["WOe"])
    plain = dataclasses.replace(w.cfg, elem_self_attn=False)
    s0, b0, _, _ = _ev(w, cfg=plain, W={k: v for k, v in W.items() if not k.endswith("e")
                                        or k in ("b1h", "b2h", "cls")})
    s1, b1, _, _ = _ev(w, W=W)
    np.testing.assert_array_equal(s1, s0)
    np.testing.assert_array_equal(b1, b0)


def test_identical_elements_attend_to_their_common_value():
    """Attention over identical keys and values returns that value, so for a
    set of identical rows h: H^(1) = h + (LN(h) W_Ve) W_Oe, row by row."""
    w = _small(elem_self_attn=True)
    h = np.tile(w.pool[0, :1].astype(np.float64), (7, 1))
    got = O.elem_self_attention(h, w.weights, w.cfg.n_heads, w.cfg.ln_eps)
    z = O.layer_norm(h[:1], w.cfg.ln_eps)
    want = h + (z @ w.weights["WVe"].astype(np.float64)) @ w.weights["WOe"].astype(np.float64)
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-15)


@pytest.mark.parametrize("encode_pool", [False, True])
def test_scores_do_not_depend_on_the_order_of_the_pool_rows(encode_pool):
    w = _small(elem_self_attn=True, encode_pool=encode_pool, M=12)
    rng = np.random.default_rng(5)
    perm = rng.permutation(w.pool.shape[1])          # new row i holds old row perm[i]
    inv = np.argsort(perm)
    pool2 = w.pool[:, perm]
    cand2 = inv[w.cand_idx].astype(np.int32)
    s0, b0, _, _ = _ev(w)
    s1, b1, _, _ = _ev(w, pool=pool2, cand=cand2)
    np.testing.assert_allclose(s1, s0, rtol=1e-11, atol=1e-14)
    np.testing.assert_array_equal(b1, b0)


def test_whole_pool_without_self_attention_equals_distinct_elements():
    w = _small(encode_pool=False)
    wp = dataclasses.replace(w.cfg, encode_pool=True)
    s0, b0, U0, _ = _ev(w)
    s1, b1, U1, sl1 = _ev(w, cfg=wp)
    np.testing.assert_allclose(s1, s0, rtol=1e-11, atol=1e-14)
    np.testing.assert_array_equal(b1, b0)
    assert (U1 == w.pool.shape[1]).all() and (U0 < U1).all()
    np.testing.assert_array_equal(sl1, w.cand_idx)


def test_distinct_set_couples_the_sequences_of_a_request():
    """With H^(1) over U(z) and no cross-sequence block, a sequence's score
    still changes when another sequence brings new elements into the set."""
    w = _small(elem_self_attn=True, cross_seq=False, B=1, K=4, M=12)
    s_all, _, _, _ = _ev(w)
    s_one, _, _, _ = _ev(w, cand=w.cand_idx[:, :1])
    assert abs(s_one[0, 0] - s_all[0, 0]) > 1e-9


def test_whole_pool_set_does_not_couple_the_sequences():
    w = _small(elem_self_attn=True, encode_pool=True, cross_seq=False, B=1, K=4, M=12)
    s_all, _, _, _ = _ev(w)
    for k in range(4):
        s_one, _, _, _ = _ev(w, cand=w.cand_idx[:, k:k + 1])
        np.testing.assert_allclose(s_one[0, 0], s_all[0, k], rtol=1e-11, atol=1e-14)


@pytest.mark.parametrize("encode_pool", [False, True])
def test_reuse_equals_no_reuse_with_self_attention(encode_pool):
    w = _small(elem_self_attn=True, encode_pool=encode_pool, M=9, K=3, L=3)
    a, _, _, _ = _ev(w, mode="reuse")
    b, _, _, _ = _ev(w, mode="no_reuse")
    np.testing.assert_allclose(a, b, rtol=1e-9, atol=1e-12)


def test_weight_count_with_self_attention():
    from paper_2603_02565_gb300 import binding
    try:
        L = binding.load_library()
    except ImportError:
        pytest.skip("library not built")
    import ctypes
    for kw in (dict(elem_self_attn=True), dict(elem_self_attn=True, n_tasks=2, cross_seq=False),
               dict(encode_pool=True)):
        cfg = wl.ModelConfig(d=64, n_heads=2, n_layers=2, max_L=5, **kw)
        n = L.fe_weight_count(ctypes.byref(binding.make_config(cfg)))
        assert n == sum(int(np.prod(s)) for _, s in wl.param_shapes(cfg))


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


@pytest.mark.gpu
@pytest.mark.parametrize("kw", [
    dict(elem_self_attn=True),                                        # H^(1) over U(z)
    dict(elem_self_attn=True, encode_pool=True),                      # H^(1) over the pool
    dict(encode_pool=True),                                           # the pool, no H^(1)
    dict(elem_self_attn=True, d=128, H=2, C=200),                     # d_h = 64
    dict(elem_self_attn=True, encode_pool=True, M=300, K=20, L=10, C=128),  # 3 query tiles, 5 key chunks
    dict(elem_self_attn=True, n_tasks=2, cross_seq=False),
])
def test_self_attention_variants_match_the_oracle(dev, kw):
    p = dict(seed=31, B=3, C=256, d=128, H=4, Ly=2, M=100, K=50, L=6)
    p.update(kw)
    w = wl.make_workload("serving", **p)
    ev, gs, gb = _gpu(w, dev)
    o_s, o_b, o_U, o_sl = O.evaluate(w.context, w.pool, w.cand_idx, w.weights, w.cfg)
    err = compare.score_error(gs, o_s)
    assert err <= compare.REL_TOL, f"max rel err {err:.3e}"
    ok, exact = compare.best_ok(gb, o_s, o_b)
    assert ok, f"best index mismatch beyond near-ties (exact {exact:.3f})"
    B, C, M, K, L = w.shape
    sl, U = ev.layout(B, K, L)
    np.testing.assert_array_equal(U, o_U)
    np.testing.assert_array_equal(sl, o_sl)


@pytest.mark.gpu
def test_self_attention_bad_index_isolated(dev):
    w = wl.make_workload("serving", seed=32, B=4, C=128, M=60, K=20, L=5, elem_self_attn=True, encode_pool=True)
    w.cand_idx[2, 3, 1] = 60
    ev, gs, gb = _gpu(w, dev)
    assert np.isnan(gs[2]).all() and gb[2] == -1
    o_s, o_b, _, _ = O.evaluate(w.context, w.pool, w.cand_idx, w.weights, w.cfg)
    keep = [0, 1, 3]
    assert compare.score_error(gs[keep], o_s[keep]) <= compare.REL_TOL


@pytest.mark.gpu
def test_factorized_refuses_set_encodings(dev):
    from paper_2603_02565_gb300.binding import FeError
    w = wl.make_workload("serving", seed=33, B=2, C=128, M=40, K=8, L=4, elem_self_attn=True)
    with pytest.raises(FeError):
        _gpu(w, dev, factorized=True)
