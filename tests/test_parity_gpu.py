"""CUDA path vs the CPU oracle, through the C-ABI (needs a GB300)."""
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


def to_dev(w, dev):
    dt = torch.bfloat16 if w.cfg.io_bf16 else torch.float32
    return (torch.from_numpy(w.context).to(dev, dt), torch.from_numpy(w.pool).to(dev, dt),
            torch.from_numpy(np.ascontiguousarray(w.cand_idx)).to(dev))


def run_gpu(w, dev, ev=None):
    from paper_2603_02565_gb300.binding import Evaluator
    ev = ev or Evaluator(w.cfg, w.weights)
    ctx, pool, idx = to_dev(w, dev)
    s, b = ev.evaluate(ctx, pool, idx)
    return ev, s.cpu().numpy(), b.cpu().numpy()


def check(w, gs, gb, requests=None):
    o_s, o_b, o_U, o_sl = O.evaluate(w.context, w.pool, w.cand_idx, w.weights, w.cfg, requests=requests)
    rq = list(range(w.shape[0])) if requests is None else list(requests)
    err = compare.score_error(gs[rq], o_s[rq])
    ok, exact = compare.best_ok(gb[rq], o_s[rq], o_b[rq])
    assert err <= compare.REL_TOL, f"{w.name}: max rel err {err:.3e}"
    assert ok, f"{w.name}: best index mismatch beyond near-ties (exact {exact:.3f})"
    return o_s, o_b, o_U, o_sl, err


def check_layout(ev, w, o_U, o_sl, requests=None):
    B, C, M, K, L = w.shape
    sl, U = ev.layout(B, K, L)
    rq = list(range(B)) if requests is None else list(requests)
    np.testing.assert_array_equal(U[rq], o_U[rq])
    np.testing.assert_array_equal(sl[rq], o_sl[rq])


def test_tiny(dev):
    w = wl.make_workload("tiny")
    ev, gs, gb = run_gpu(w, dev)
    o_s, o_b, o_U, o_sl, err = check(w, gs, gb)
    check_layout(ev, w, o_U, o_sl)
    assert gb[0] == o_b[0]
    # fp32 inputs take the unfused context path: LN(context) and K/V both visible
    X = O.layer_norm(w.context[0], w.cfg.ln_eps)
    np.testing.assert_allclose(ev.fetch("ctx_ln"), X, rtol=0, atol=2e-5)
    np.testing.assert_allclose(ev.fetch("ctx_kv", cols=2 * w.cfg.n_layers * w.cfg.d), context_kv_rows(w, 1),
                               rtol=KV_RTOL, atol=KV_ATOL)


@pytest.mark.parametrize("B", [3, 8])
def test_serving_small_batches(dev, B):
    w = wl.make_workload("serving", B=B)
    ev, gs, gb = run_gpu(w, dev)
    o_s, o_b, o_U, o_sl, err = check(w, gs, gb)
    check_layout(ev, w, o_U, o_sl)


@pytest.mark.parametrize("d,H", [(32, 1), (64, 2)])
def test_serving_narrow(dev, d, H):
    """Narrow bf16 rows: the fused embedding and FFN kernels with one 64-column
    k block (d = 32 leaves half of it as zero padding), the FFN tails, and at
    d = 32 the unfused context path (N = 2 Ly d = 128 < 256)."""
    w = wl.make_workload("serving", B=5, d=d, H=H)
    ev, gs, gb = run_gpu(w, dev)
    o_s, o_b, o_U, o_sl, err = check(w, gs, gb)
    check_layout(ev, w, o_U, o_sl)


def context_kv_rows(w, nreq):
    """Oracle [K_0 | V_0 | K_1 | V_1 ...] rows of the first nreq requests."""
    cfg = w.cfg
    rows = []
    for b in range(nreq):
        kv = O.context_kv(w.context[b], w.weights, cfg.n_layers, cfg.ln_eps)
        rows.append(np.hstack([m for pair in kv for m in pair]))
    return np.vstack(rows)


# The context K/V are held as f16 (unit roundoff 2^-11 = 4.9e-4 relative) after a
# split-bf16 product (relative error ~2^-16): rtol 1e-3 bounds both, atol covers
# values near zero where the f16 subnormal spacing (6e-8) and the products'
# absolute error (~1e-6 at these weight scales) dominate.
KV_RTOL, KV_ATOL = 1e-3, 1e-5


@pytest.mark.parametrize("kind,B", [("stress", 2), ("summarisation", 2)])
def test_context_kv_ln_folded(dev, kind, B):
    """d = 256 and d = 512 with bf16 inputs: the K/V product multiplies the raw
    context rows and applies the row statistics in its epilogue,
    rstd (x W) - mu rstd colsum(W); LN(context) is not materialised."""
    from paper_2603_02565_gb300.binding import Evaluator, FeError
    w = wl.summarisation(B=B) if kind == "summarisation" else wl.make_workload(kind, B=B)
    ev = Evaluator(w.cfg, w.weights)
    ev, gs, gb = run_gpu(w, dev, ev)
    np.testing.assert_allclose(ev.fetch("ctx_kv", cols=2 * w.cfg.n_layers * w.cfg.d), context_kv_rows(w, B),
                               rtol=KV_RTOL, atol=KV_ATOL)
    with pytest.raises(FeError):
        ev.fetch("ctx_ln")
    if kind == "stress":  # (the summarisation scores: test_summarisation_small)
        check(w, gs, gb)


def test_stagewise_serving(dev):
    """Intermediates: context K/V, element cache, SeqEnc and cross-sequence outputs
    (serving runs the fused context kernel, so LN(context) is not materialised)."""
    from paper_2603_02565_gb300.binding import Evaluator, FeError
    w = wl.make_workload("serving", B=2)
    ev = Evaluator(w.cfg, w.weights)
    ev.keep_intermediates(True)  # c and C' are otherwise kept on chip by the sequence-stage kernel
    ev, gs, gb = run_gpu(w, dev, ev)
    cfg, W = w.cfg, w.weights
    eps = cfg.ln_eps
    np.testing.assert_allclose(ev.fetch("ctx_kv", cols=2 * cfg.n_layers * cfg.d), context_kv_rows(w, 2),
                               rtol=KV_RTOL, atol=KV_ATOL)
    with pytest.raises(FeError):
        ev.fetch("ctx_ln")
    elem, seq, cross = [], [], []
    for b in range(2):
        kv = O.context_kv(w.context[b], W, cfg.n_layers, eps)
        uniq, slots = O.distinct_layout(w.cand_idx[b])
        Hb = O.encode_elements(w.pool[b][uniq], kv, W, cfg.n_heads, eps)
        elem.append(Hb)
        Cm = np.vstack([O.seq_encode(Hb[slots[k]], W, cfg.n_heads, eps) for k in range(w.shape[3])])
        seq.append(Cm)
        cross.append(O.cross_sequence(Cm, W, cfg.n_heads, eps))
    np.testing.assert_allclose(ev.fetch("elem"), np.vstack(elem), rtol=0, atol=2e-4)
    # c and C' come from the [CLS] attention, whose value rows are single f16 planes
    # like every attention operand (unit roundoff 2^-11 on values of magnitude up to
    # ~0.2): an absolute error of up to ~1e-4 on c, rtol 1e-3 elsewhere
    np.testing.assert_allclose(ev.fetch("seq"), np.vstack(seq), rtol=1e-3, atol=1e-4)
    np.testing.assert_allclose(ev.fetch("cross"), np.vstack(cross), rtol=1e-3, atol=1e-4)


@pytest.mark.parametrize("K", [1, 10, 50, 100, 129, 400, 1000])
def test_ksweep_small(dev, K):
    w = wl.make_workload("ksweep", K=K, B=3)
    ev, gs, gb = run_gpu(w, dev)
    o_s, o_b, o_U, o_sl, err = check(w, gs, gb)
    check_layout(ev, w, o_U, o_sl)


def test_summarisation_small(dev):
    w = wl.summarisation(B=2)
    ev, gs, gb = run_gpu(w, dev)
    o_s, o_b, o_U, o_sl, err = check(w, gs, gb)
    check_layout(ev, w, o_U, o_sl)


def test_stress_small(dev):
    w = wl.make_workload("stress", B=3)
    ev, gs, gb = run_gpu(w, dev)
    check(w, gs, gb)


def test_bad_index_isolated(dev):
    from paper_2603_02565_gb300 import binding
    w = wl.make_workload("serving", B=4)
    w.cand_idx = w.cand_idx.copy()
    w.cand_idx[2, 7, 3] = w.shape[2]          # == M
    w.cand_idx[3, 0, 0] = -1
    ev, gs, gb = run_gpu(w, dev)
    assert ev.last_status == binding.FE_ERR_INDEX
    assert np.isnan(gs[2:]).all() and (gb[2:] == -1).all()
    check(w, gs, gb, requests=[0, 1])


def test_nan_request_isolated(dev):
    """A NaN input value leaves Eq. 1 without a maximum for its request: that
    request's scores are NaN and its best index -1 (FE_ERR_NUMERIC, the NaN
    flags of the fused argmax), the other requests are unaffected, and the next
    batch starts clean, through the device entry and the pipelined host entry."""
    from paper_2603_02565_gb300 import binding
    w = wl.make_workload("serving", B=4)
    clean = wl.make_workload("serving", B=4)   # the same weights and inputs, without the NaNs
    w.pool, w.context = w.pool.copy(), w.context.copy()
    w.pool[1, int(w.cand_idx[1, 0, 0]), 3] = np.nan   # one element of request 1
    w.context[3, 5, 0] = np.nan                        # one context row of request 3
    ev, gs, gb = run_gpu(w, dev)
    for b in (1, 3):
        assert np.isnan(gs[b]).all() and gb[b] == -1
    assert ev.last_status == binding.FE_ERR_NUMERIC
    check(w, gs, gb, requests=[0, 2])
    _, cs, cb = run_gpu(clean, dev, ev)
    assert ev.last_status == binding.FE_OK
    check(clean, cs, cb)
    dt = torch.bfloat16
    host = [(torch.from_numpy(x.context).to(dt).pin_memory(), torch.from_numpy(x.pool).to(dt).pin_memory(),
             torch.from_numpy(np.ascontiguousarray(x.cand_idx)).pin_memory()) for x in (w, clean)]
    outs = [(np.zeros((4, w.shape[3]), np.float32), np.zeros(4, np.int32)) for _ in range(2)]
    ev.submit_host(*host[0], *outs[0])
    ev.submit_host(*host[1], *outs[1])
    assert ev.wait_host() == binding.FE_ERR_NUMERIC
    assert ev.wait_host() == binding.FE_OK
    np.testing.assert_array_equal(outs[0][0], gs)
    np.testing.assert_array_equal(outs[0][1], gb)
    np.testing.assert_array_equal(outs[1][0], cs)
    np.testing.assert_array_equal(outs[1][1], cb)


@pytest.mark.parametrize("kw,where", [
    (dict(B=3, C=100), "context"),
    (dict(B=3, C=128, M=60, K=20, L=5, elem_self_attn=True, encode_pool=True, seed=32), "pool")])
def test_nan_isolated_across_partial_chunks(dev, kw, where):
    """Request 0's last key chunk reaches into request 1's rows: context rows
    100-127 of a 100-row context, element rows 60-63 of the element
    self-attention over 60 elements. A NaN there stays in request 1."""
    from paper_2603_02565_gb300 import binding
    w = wl.make_workload("serving", **kw)
    w.pool, w.context = w.pool.copy(), w.context.copy()
    if where == "context":
        w.context[1, 3, 0] = np.nan   # key row 103 of request 0's second chunk
    else:
        w.pool[1, 2, 0] = np.nan      # element row 62 of request 0's only chunk
    ev, gs, gb = run_gpu(w, dev)
    assert np.isnan(gs[1]).all() and gb[1] == -1
    assert ev.last_status == binding.FE_ERR_NUMERIC
    check(w, gs, gb, requests=[0, 2])


def test_empty_batches(dev):
    """K = 0 leaves Eq. 1 without candidates: best -1 for every request with
    status FE_OK, as in the oracle; B = 0 does nothing; a normal batch on the
    same context afterwards is unaffected."""
    from paper_2603_02565_gb300 import binding
    w = wl.make_workload("serving", B=3, K=0)
    ev, gs, gb = run_gpu(w, dev)
    assert gs.shape == (3, 0) and ev.last_status == binding.FE_OK
    np.testing.assert_array_equal(gb, O.evaluate(w.context, w.pool, w.cand_idx, w.weights, w.cfg)[1])
    _, gs0, gb0 = run_gpu(wl.make_workload("serving", B=0), dev, ev)
    assert gs0.shape == (0, 50) and gb0.shape == (0,) and ev.last_status == binding.FE_OK
    w1 = wl.make_workload("serving", B=2)
    _, gs1, gb1 = run_gpu(w1, dev, ev)
    check(w1, gs1, gb1)


def test_edge_shapes(dev):
    """K = 1, L = 1, M = 1, and a sequence repeating one element."""
    for kw in [dict(K=1), dict(L=1), dict(M=1, L=1, K=3), dict(K=2, L=3, M=3)]:
        w = wl.make_workload("serving", B=2, **kw)
        ev, gs, gb = run_gpu(w, dev)
        check(w, gs, gb)
    w = wl.make_workload("serving", B=2, K=3, L=4)
    w.cand_idx = w.cand_idx.copy()
    w.cand_idx[0, 1, :] = w.cand_idx[0, 1, 0]  # one element four times
    ev, gs, gb = run_gpu(w, dev)
    check(w, gs, gb)


def test_repeat_calls_and_host_entry_agree(dev):
    w = wl.make_workload("serving", B=5)
    ev, gs1, gb1 = run_gpu(w, dev)
    _, gs2, gb2 = run_gpu(w, dev, ev)
    np.testing.assert_array_equal(gs1, gs2)
    ctx = torch.from_numpy(w.context).to(torch.bfloat16).pin_memory()
    pool = torch.from_numpy(w.pool).to(torch.bfloat16).pin_memory()
    idx = torch.from_numpy(w.cand_idx).pin_memory()
    hs, hb = ev.evaluate_host(ctx, pool, idx)
    np.testing.assert_array_equal(hs, gs1)
    np.testing.assert_array_equal(hb, gb1)


def test_serving_full_batch(dev):
    """The benchmark's serving batch (B=256, K=50), every request checked."""
    w = wl.make_workload("serving")
    ev, gs, gb = run_gpu(w, dev)
    o_s, o_b, o_U, o_sl, err = check(w, gs, gb)
    check_layout(ev, w, o_U, o_sl)


def test_stress_full_batch_sampled(dev):
    """Throughput-stress batch at full size (B=1024), 6 sampled requests checked."""
    w = wl.make_workload("stress")
    ev, gs, gb = run_gpu(w, dev)
    rq = [0, 1, 511, 777, 1022, 1023]
    o_s, o_b, o_U, o_sl, err = check(w, gs, gb, requests=rq)
    check_layout(ev, w, o_U, o_sl, requests=rq)


def test_stress_mid_batch_sampled(dev):
    """Stress width at B=24: the cross-sequence LayerNorm GEMM and the score head
    (4800 sequence rows, 38 row tiles) over clusters of two CTAs of 128 columns;
    three sampled requests checked."""
    w = wl.make_workload("stress", B=24)
    ev, gs, gb = run_gpu(w, dev)
    rq = [0, 11, 23]
    o_s, o_b, o_U, o_sl, err = check(w, gs, gb, requests=rq)
    check_layout(ev, w, o_U, o_sl, requests=rq)


def test_summarisation_full_batch_sampled(dev):
    """The summarisation batch at the benchmark's size (B=32, C=1024, d=512, K=16,
    L=64): clustered LayerNorm GEMMs and score head, the folded context K/V and the
    several-warps [CLS] attention at their launch sizes; the first and last
    requests checked."""
    w = wl.summarisation()
    ev, gs, gb = run_gpu(w, dev)
    rq = [0, w.shape[0] - 1]
    o_s, o_b, o_U, o_sl, err = check(w, gs, gb, requests=rq)
    check_layout(ev, w, o_U, o_sl, requests=rq)


def test_pipelined_host_entry(dev):
    """fe_submit_host / fe_wait_host: three different batches in flight give the
    same results as the synchronous entry; other calls are refused meanwhile."""
    from paper_2603_02565_gb300.binding import Evaluator, FeError
    w1 = wl.make_workload("serving", B=4)
    w2 = wl.make_workload("serving", B=4, seed=11)
    w3 = wl.make_workload("serving", B=4, seed=12)
    ev = Evaluator(w1.cfg, w1.weights)
    dt = torch.bfloat16
    host = []
    for w in (w1, w2, w3):
        host.append((torch.from_numpy(w.context).to(dt).pin_memory(), torch.from_numpy(w.pool).to(dt).pin_memory(),
                     torch.from_numpy(np.ascontiguousarray(w.cand_idx)).pin_memory()))
    ref = [ev.evaluate_host(*h) for h in host]
    outs = [(np.full((4, w1.shape[3]), -1.0, np.float32), np.full(4, -7, np.int32)) for _ in range(3)]
    for rep in range(2):
        ev.submit_host(*host[0], *outs[0])
        ev.submit_host(*host[1], *outs[1])
        ev.submit_host(*host[2], *outs[2])
        with pytest.raises(FeError):
            ev.submit_host(*host[0], *outs[0])  # a fourth outstanding submission
        with pytest.raises(FeError):
            ev.evaluate_host(*host[0])          # the workspace is in use
        ev.wait_host()
        ev.wait_host()
        ev.wait_host()
        for (s_ref, b_ref), (s, b) in zip(ref, outs):
            np.testing.assert_array_equal(s, s_ref)
            np.testing.assert_array_equal(b, b_ref)
    with pytest.raises(FeError):
        ev.wait_host()                          # nothing outstanding
    check(w1, outs[0][0], outs[0][1])


@pytest.mark.parametrize("name,kw", [("ksweep", dict(K=10, B=3)), ("ksweep", dict(K=100, B=2)),
                                     ("serving", dict(B=3))])
def test_factorized_matches_joint(dev, name, kw):
    """fe_evaluate_factorized (context K/V per sequence, every occurrence encoded on
    its own) gives the joint evaluation's scores: the same per-row arithmetic, only
    more of it; against the oracle as well."""
    w = wl.make_workload(name, **kw)
    ev, gs, gb = run_gpu(w, dev)
    ctx, pool, idx = to_dev(w, dev)
    fs, fb = ev.evaluate(ctx, pool, idx, factorized=True)
    fs, fb = fs.cpu().numpy(), fb.cpu().numpy()
    np.testing.assert_allclose(fs, gs, rtol=1e-5, atol=1e-7)
    np.testing.assert_array_equal(fb, gb)
    check(w, fs, fb)
    B, C, M, K, L = w.shape
    sl, U = ev.layout(B, K, L)
    np.testing.assert_array_equal(U, np.full(B, K * L))
    np.testing.assert_array_equal(sl.reshape(B, -1), np.tile(np.arange(K * L), (B, 1)))
    # the joint evaluation still works on the same context afterwards
    gs2, gb2 = ev.evaluate(ctx, pool, idx)
    np.testing.assert_array_equal(gs2.cpu().numpy(), gs)


def test_factorized_bad_index(dev):
    w = wl.make_workload("serving", B=4)
    idx_bad = np.array(w.cand_idx)
    idx_bad[1, 3, 2] = w.shape[2]  # == M: out of range
    from paper_2603_02565_gb300.binding import Evaluator
    ev = Evaluator(w.cfg, w.weights)
    ctx, pool, _ = to_dev(w, dev)
    idx = torch.from_numpy(np.ascontiguousarray(idx_bad)).to(dev)
    fs, fb = ev.evaluate(ctx, pool, idx, factorized=True)
    fs, fb = fs.cpu().numpy(), fb.cpu().numpy()
    assert np.isnan(fs[1]).all() and fb[1] == -1
    js, jb = ev.evaluate(ctx, pool, idx)
    ok = [0, 2, 3]
    np.testing.assert_allclose(fs[ok], js.cpu().numpy()[ok], rtol=1e-5, atol=1e-7)
    np.testing.assert_array_equal(fb[ok], jb.cpu().numpy()[ok])
