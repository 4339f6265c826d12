"""Failure paths of the boundary, exercised without faulting the GPU.

* Allocation failure: the library's allocation hook (fe_debug_alloc_hook)
  makes a chosen device or page-locked allocation fail as if the device were
  out of memory.  fe_init and a workspace grow must return FE_ERR_OOM, leave no
  allocation behind, and the context must keep working after a failed grow.
* Bounded waits: fe_debug_wait_probe runs one thread that waits, through the
  batch kernels' own bounded mbarrier wait, on a barrier nothing arrives on
  (limit 1 ms, nothing else in flight).  The status must reach the host as
  FE_ERR_TIMEOUT and the next batch on the same context must be correct.
* A weight blob gives the same context as the raw weight array.
"""
import ctypes

import numpy as np
import pytest

from oracle import compare
from oracle import fe_oracle as O
from paper_2603_02565_gb300 import binding
from paper_2603_02565_gb300 import workloads as wl

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def _lib():
    from paper_2603_02565_gb300 import build
    build.build()
    return binding.load_library()


def _live(L):
    n = ctypes.c_int64()
    assert L.fe_debug_alloc_hook(-1, ctypes.byref(n)) == binding.FE_OK
    return n.value


def _arm(L, n):
    assert L.fe_debug_alloc_hook(n, None) == binding.FE_OK


def _inputs(w, dev):
    dt = torch.bfloat16 if w.cfg.io_bf16 else torch.float32
    return (torch.from_numpy(w.context).to(dev, dt), torch.from_numpy(w.pool).to(dev, dt),
            torch.from_numpy(w.cand_idx).to(dev))


def _check_parity(w, scores, best):
    o_s, o_b, _, _ = O.evaluate(w.context, w.pool, w.cand_idx, w.weights, w.cfg)
    assert compare.score_error(scores.cpu().numpy(), o_s) <= compare.REL_TOL
    assert compare.best_ok(best.cpu().numpy(), o_s, o_b)[0]


def test_init_allocation_failures_leak_nothing():
    L = _lib()
    w = wl.make_workload("serving", B=2)
    c = binding.make_config(w.cfg)
    flat = binding.pack_weights(w.cfg, w.weights)
    ptr = flat.ctypes.data_as(ctypes.POINTER(ctypes.c_float))
    live0 = _live(L)
    h = ctypes.c_void_p()
    assert L.fe_init(ctypes.byref(c), ptr, flat.size, ctypes.byref(h)) == binding.FE_OK
    n_init = _live(L) - live0
    assert n_init > 0
    assert L.fe_destroy(h) == binding.FE_OK
    assert _live(L) == live0
    for n in range(1, n_init + 1):
        _arm(L, n)
        h = ctypes.c_void_p()
        rc = L.fe_init(ctypes.byref(c), ptr, flat.size, ctypes.byref(h))
        _arm(L, 0)
        assert rc == binding.FE_ERR_OOM, (n, rc)
        assert not h.value
        assert _live(L) == live0, n
    # disarmed: a normal context again
    h = ctypes.c_void_p()
    assert L.fe_init(ctypes.byref(c), ptr, flat.size, ctypes.byref(h)) == binding.FE_OK
    L.fe_destroy(h)
    assert _live(L) == live0


def test_failed_workspace_grow_leaves_a_usable_context():
    L = _lib()
    dev = torch.device("cuda:0")
    w = wl.make_workload("serving", B=4)
    live0 = _live(L)
    ev = binding.Evaluator(w.cfg, w.weights)
    live_w = _live(L)
    ctx, pool, idx = _inputs(w, dev)
    s0, b0 = ev.evaluate(ctx, pool, idx)
    _check_parity(w, s0, b0)
    s0, b0 = s0.clone(), b0.clone()
    n_ws = _live(L) - live_w
    assert n_ws > 0
    B2 = 16
    big = wl.make_workload("serving", B=B2)
    bctx, bpool, bidx = _inputs(big, dev)
    for n in sorted({1, 2, n_ws // 2, n_ws}):
        # a grow through fe_reserve
        _arm(L, n)
        with pytest.raises(binding.FeError) as e:
            ev.reserve(B2, 256, 100, 50, 6)
        _arm(L, 0)
        assert e.value.code == binding.FE_ERR_OOM
        assert _live(L) == live_w  # the old workspace and the partial new one are released
        # the context still evaluates, and gives the same result as before
        s1, b1 = ev.evaluate(ctx, pool, idx)
        assert torch.equal(s1, s0) and torch.equal(b1, b0)
        # a grow inside an evaluation
        _arm(L, n)
        with pytest.raises(binding.FeError) as e:
            ev.evaluate(bctx, bpool, bidx)
        _arm(L, 0)
        assert e.value.code == binding.FE_ERR_OOM
        assert _live(L) == live_w
    s2, b2 = ev.evaluate(bctx, bpool, bidx)
    _check_parity(big, s2, b2)
    ev.close()
    assert _live(L) == live0  # fe_destroy released everything the context owned


def test_bounded_wait_reports_timeout_and_the_context_recovers():
    L = _lib()
    dev = torch.device("cuda:0")
    stream = torch.cuda.current_stream(dev).cuda_stream
    w = wl.make_workload("serving", B=4)
    # a context with no workspace yet: the probe reserves a minimal one
    ev = binding.Evaluator(w.cfg, w.weights)
    assert L.fe_debug_wait_probe(ev._h, 1000, ctypes.c_void_p(stream)) == binding.FE_ERR_TIMEOUT
    ctx, pool, idx = _inputs(w, dev)
    s0, b0 = ev.evaluate(ctx, pool, idx)
    assert ev.last_status == binding.FE_OK
    _check_parity(w, s0, b0)
    s0, b0 = s0.clone(), b0.clone()
    # again between two batches on the same workspace
    assert L.fe_debug_wait_probe(ev._h, 1000, ctypes.c_void_p(stream)) == binding.FE_ERR_TIMEOUT
    s1, b1 = ev.evaluate(ctx, pool, idx)
    assert ev.last_status == binding.FE_OK
    assert torch.equal(s1, s0) and torch.equal(b1, b0)
    assert L.fe_debug_wait_probe(ev._h, 0, None) == binding.FE_ERR_INVALID_ARG
    ev.close()


def test_blob_context_matches_raw_weights():
    _lib()
    dev = torch.device("cuda:0")
    for w in (wl.make_workload("tiny"), wl.make_workload("serving", B=3)):
        ctx, pool, idx = _inputs(w, dev)
        a = binding.Evaluator(w.cfg, w.weights)
        b = binding.Evaluator.from_blob(binding.weights_blob(w.cfg, w.weights))
        sa, ba = a.evaluate(ctx, pool, idx)
        sb, bb = b.evaluate(ctx, pool, idx)
        assert torch.equal(sa, sb) and torch.equal(ba, bb)
        _check_parity(w, sb, bb)
        a.close()
        b.close()
