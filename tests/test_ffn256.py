"""The d = 256 output projection + FFN kernel (fe_ffn256.cu) against the oracle:
one block's x0 + A W_O, LayerNorm, FFN (Section 4.2 for the element layers,
Section 4.3 for SeqEnc), LN(x_out) and the next layer's Q as a tail product.
These cases cover a single element row (one partial tile), several partial
tiles, one layer (no Q tail) and three layers (two tails), the element
encodings and the SeqEnc output against the oracle's intermediates, a rejected
request and a NaN pool row next to valid requests, and the element
self-attention with two task heads on the same kernel."""
import numpy as np
import pytest

import oracle.fe_oracle as O
from oracle import compare
from paper_2603_02565_gb300 import workloads as wl

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2603_02565_gb300 import build
    build.build()
    return torch.device("cuda:0")


def run(w, dev, keep=False, cand=None):
    from paper_2603_02565_gb300.binding import Evaluator
    ev = Evaluator(w.cfg, w.weights)
    if keep:
        ev.keep_intermediates(True)
    dt = torch.bfloat16
    ctx = torch.from_numpy(w.context).to(dev, dt)
    pool = torch.from_numpy(w.pool).to(dev, dt)
    idx = w.cand_idx if cand is None else cand
    s, b = ev.evaluate(ctx, pool, torch.from_numpy(np.ascontiguousarray(idx)).to(dev))
    return ev, s.cpu().numpy(), b.cpu().numpy()


def check(w, gs, gb, requests):
    o_s, o_b, _, _ = O.evaluate(w.context, w.pool, w.cand_idx, w.weights, w.cfg, requests=requests)
    rq = list(requests)
    err = compare.score_error(gs[rq], o_s[rq])
    ok, _ = compare.best_ok(gb[rq], o_s[rq], o_b[rq])
    assert err <= compare.REL_TOL, f"max rel err {err:.3e}"
    assert ok
    return o_s, o_b


# the stress width (d = 256, 8 heads) at small sizes
def small(**kw):
    p = dict(B=2, C=128, M=40, K=6, L=4)
    p.update(kw)
    return wl.stress(**p)


@pytest.mark.parametrize("kw", [
    dict(B=1, K=1, L=1, M=1),        # one element row: a single partial tile
    dict(B=3, K=40, L=5, M=200),     # several tiles, the last one partial
    dict(Ly=1),                      # one layer: no Q tail, LN(x_out) stored
    dict(Ly=3),                      # three layers: two Q tails
])
def test_shapes(dev, kw):
    w = small(**kw)
    _, gs, gb = run(w, dev)
    check(w, gs, gb, range(w.shape[0]))


def test_intermediates(dev):
    """The element encodings (LN of the last layer's x_out) and the SeqEnc output c."""
    w = small(B=2, K=5, L=3, M=30)
    ev, gs, gb = run(w, dev, keep=True)
    cfg, W = w.cfg, w.weights
    eps = cfg.ln_eps
    elem, seq = [], []
    for b in range(2):
        kv = O.context_kv(w.context[b], W, cfg.n_layers, eps)
        uniq, slots = O.distinct_layout(w.cand_idx[b])
        Hb = O.encode_elements(w.pool[b][uniq], kv, W, cfg.n_heads, eps)
        elem.append(Hb)
        seq.append(np.vstack([O.seq_encode(Hb[slots[k]], W, cfg.n_heads, eps) for k in range(w.shape[3])]))
    np.testing.assert_allclose(ev.fetch("elem"), np.vstack(elem), rtol=0, atol=2e-4)
    np.testing.assert_allclose(ev.fetch("seq"), np.vstack(seq), rtol=1e-3, atol=1e-4)
    check(w, gs, gb, range(2))


def test_bad_index_and_nan_isolated(dev):
    """An out-of-range index rejects its request (NaN scores, best -1, FE_ERR_INDEX);
    a NaN element row makes its request's scores NaN (FE_ERR_NUMERIC); the
    other requests of the batch are unaffected."""
    from paper_2603_02565_gb300 import binding
    w = small(B=4, K=8, L=4, M=40)
    bad = w.cand_idx.copy()
    bad[1, 2, 1] = w.shape[2]                      # == M
    ev, gs, gb = run(w, dev, cand=bad)
    assert ev.last_status == binding.FE_ERR_INDEX
    assert np.isnan(gs[1]).all() and gb[1] == -1
    check(w, gs, gb, [0, 2, 3])
    w.pool = w.pool.copy()
    w.pool[3, int(w.cand_idx[3, 0, 0]), 7] = np.nan   # one value of one element of request 3
    ev, gs, gb = run(w, dev)
    assert ev.last_status == binding.FE_ERR_NUMERIC
    assert np.isnan(gs[3]).all() and gb[3] == -1
    check(w, gs, gb, [0, 1, 2])


def test_elem_self_attn_two_heads(dev):
    """H^(1) before the element layers and two task heads, on the same kernel."""
    w = small(B=2, K=5, L=3, M=20, elem_self_attn=True, n_tasks=2)
    _, gs, gb = run(w, dev)
    check(w, gs, gb, range(2))
