"""The sequence stage (index-based assembly and SeqEnc of Section 4.3, the
cross-sequence block and head of Section 4.4, the argmax of Eq. 1) as one
kernel, for d = 128, K <= 128, L <= 31 and one score head: G whole requests
share a 128-row tile, so the cross-sequence attention runs with a
block-diagonal request mask and the argmax inside the tile.  These cases
cover tiles of one, two and twelve requests, the largest K and L, d_h = 64,
rejected and NaN requests next to valid ones in the same tile, and the
intermediates."""
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


def run(w, dev, keep=False, idx=None):
    from paper_2603_02565_gb300.binding import Evaluator
    ev = Evaluator(w.cfg, w.weights)
    if keep:
        ev.keep_intermediates(True)
    dt = torch.bfloat16
    ctx = torch.from_numpy(w.context).to(dev, dt)
    pool = torch.from_numpy(w.pool).to(dev, dt)
    cand = w.cand_idx if idx is None else idx
    s, b = ev.evaluate(ctx, pool, torch.from_numpy(np.ascontiguousarray(cand)).to(dev))
    return ev, s.cpu().numpy(), b.cpu().numpy()


def check(w, gs, gb, requests):
    o_s, o_b, _, _ = O.evaluate(w.context, w.pool, w.cand_idx, w.weights, w.cfg, requests=requests)
    rq = list(requests)
    err = compare.score_error(gs[rq], o_s[rq])
    ok, _ = compare.best_ok(gb[rq], o_s[rq], o_b[rq])
    assert err <= compare.REL_TOL, f"max rel err {err:.3e}"
    assert ok
    return o_s, o_b


@pytest.mark.parametrize("K,L,B", [(1, 6, 5), (128, 6, 3), (50, 31, 3), (20, 1, 4), (64, 2, 3)])
def test_edge_K_L(dev, K, L, B):
    # K = 1: one sequence per request (cross-sequence attention over itself); K = 128: a
    # full tile; L = 31: the longest sequences; L = 1
    w = wl.serving(B=B, K=K, L=L, M=max(40, L))
    _, gs, gb = run(w, dev)
    check(w, gs, gb, range(B))


def test_dh64(dev):
    w = wl.serving(B=4, H=2)
    _, gs, gb = run(w, dev)
    check(w, gs, gb, range(4))


def test_packed_tiles_sampled(dev):
    # B = 1900 requests of K = 10 fill the GPU with twelve requests per tile:
    # requests at tile edges and in the middle against the oracle
    w = wl.ksweep(10, B=1900, C=128)
    _, gs, gb = run(w, dev)
    rq = [0, 1, 11, 12, 13, 23, 24, 950, 1139, 1140, 1887, 1888, 1899]
    check(w, gs, gb, rq)


def test_rejected_and_nan_requests_in_a_packed_tile(dev):
    w = wl.ksweep(10, B=1900, C=128)
    idx = np.array(w.cand_idx)
    idx[37, 2, 3] = w.shape[2]                            # request 37: index == M, rejected
    w.pool[38, int(idx[38, 4, 1]), 7] = np.nan            # request 38: a NaN element
    w.context[40, 9, 0] = np.inf                          # request 40: an infinite context value
    w = wl.Workload(w.name, w.cfg, w.context, w.pool, idx, w.weights)
    from paper_2603_02565_gb300.binding import FE_ERR_INDEX
    _, gs, gb = run(w, dev)
    for b in (37, 38, 40):
        assert np.isnan(gs[b]).all() and gb[b] == -1, b
    # the other requests of the same tile (36..47) and the tiles around it are untouched
    check(w, gs, gb, [36, 39, 41, 42, 47, 48, 35])


def test_nan_in_packed_serving_tile(dev):
    # two requests per tile: a NaN in one must not reach its neighbour through the
    # cross-sequence attention's masked keys (P = 0 times a NaN value row)
    w = wl.serving(B=8)
    w.pool[2, int(w.cand_idx[2, 7, 0]), 5] = np.nan
    _, gs, gb = run(w, dev)
    assert np.isnan(gs[2]).all() and gb[2] == -1
    check(w, gs, gb, [0, 1, 3, 4, 5, 6, 7])


def test_intermediates_only_when_kept(dev):
    from paper_2603_02565_gb300.binding import FeError
    w = wl.serving(B=2)
    ev, gs, gb = run(w, dev)
    with pytest.raises(FeError):
        ev.fetch("seq")
    with pytest.raises(FeError):
        ev.fetch("cross")
    ev2, gs2, gb2 = run(w, dev, keep=True)
    # storing the intermediates changes nothing else
    assert np.array_equal(gs, gs2) and np.array_equal(gb, gb2)
    cfg, W = w.cfg, w.weights
    seq, cross = [], []
    for b in range(2):
        kv = O.context_kv(w.context[b], W, cfg.n_layers, cfg.ln_eps)
        uniq, slots = O.distinct_layout(w.cand_idx[b])
        Hb = O.encode_elements(w.pool[b][uniq], kv, W, cfg.n_heads, cfg.ln_eps)
        Cm = np.vstack([O.seq_encode(Hb[slots[k]], W, cfg.n_heads, cfg.ln_eps) for k in range(w.shape[3])])
        seq.append(Cm)
        cross.append(O.cross_sequence(Cm, W, cfg.n_heads, cfg.ln_eps))
    # c and C' come from the [CLS] attention, whose value rows are single f16 planes
    # like every attention operand (unit roundoff 2^-11 on values of magnitude up to
    # ~0.2): an absolute error of up to ~1e-4 on c, rtol 1e-3 elsewhere
    np.testing.assert_allclose(ev2.fetch("seq"), np.vstack(seq), rtol=1e-3, atol=1e-4)
    np.testing.assert_allclose(ev2.fetch("cross"), np.vstack(cross), rtol=1e-3, atol=1e-4)
    ev2.keep_intermediates(False)


def test_one_launch_for_the_sequence_stage(dev):
    w = wl.serving(B=4)
    ev, _, _ = run(w, dev)
    ev.profile(True)
    dt = torch.bfloat16
    ctx = torch.from_numpy(w.context).to(dev, dt)
    pool = torch.from_numpy(w.pool).to(dev, dt)
    idx = torch.from_numpy(w.cand_idx).to(dev)
    ev.evaluate(ctx, pool, idx)
    sites = [s[0] for s in ev.profile_read()]
    ev.profile(False)
    assert "seq_stage" in sites
    for old in ("seq_cls_attn", "ffn_seq", "gemm_cross_qkv", "attn_cross_seq", "gemm_cross_o_ln", "gemm_head"):
        assert old not in sites
