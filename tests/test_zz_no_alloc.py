"""The allocation-free layout entry point, for callers that may not allocate
GPU memory (a serving runtime whose pool owns the device, code that must not
risk an allocation's implicit synchronisation).  Its output must equal the
layout the regular evaluation computes, call after call, although every call
reuses the same fixed device scratch.

Collected last on purpose (file name), so that a failure here cannot stop a
run before the other tests have executed."""
import ctypes

import numpy as np
import pytest

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


def regular_layout(w, dev):
    """Layout from the existing entry point: fe_evaluate, then fe_debug_layout."""
    from paper_2603_02565_gb300.binding import Evaluator
    ev = Evaluator(w.cfg, w.weights)
    dt = torch.bfloat16 if w.cfg.io_bf16 else torch.float32
    ev.evaluate(torch.from_numpy(w.context).to(dev, dt), torch.from_numpy(w.pool).to(dev, dt),
                torch.from_numpy(np.ascontiguousarray(w.cand_idx)).to(dev))
    B, C, M, K, L = w.shape
    slots, U = ev.layout(B, K, L)
    ev.close()
    return slots, U


def noalloc_layout(cand_idx, M, dev):
    """Calls fe_distinct_layout_noalloc through the C-ABI.  The output buffers
    are allocated here, by the caller, before the call."""
    from paper_2603_02565_gb300.binding import FE_OK, load_library
    lib = load_library()
    B, K, L = cand_idx.shape
    idx = torch.from_numpy(np.ascontiguousarray(cand_idx)).to(dev)
    U = torch.full((B,), -7, dtype=torch.int32, device=dev)
    slots = torch.full((B, K, L), -7, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream(dev)
    rc = lib.fe_distinct_layout_noalloc(ctypes.c_void_p(idx.data_ptr()), B, M, K, L,
                                        ctypes.c_void_p(U.data_ptr()), ctypes.c_void_p(slots.data_ptr()),
                                        ctypes.c_void_p(stream.cuda_stream))
    assert rc == FE_OK
    stream.synchronize()
    return slots.cpu().numpy(), U.cpu().numpy()


def test_noalloc_layout_matches_evaluate_twice_in_a_row(dev):
    # two different batches back to back: the second call must not see the
    # first call's leftovers in the shared scratch
    wa = wl.make_workload("serving", B=9)
    wb = wl.make_workload("ksweep", K=100, B=5)
    ref_a = regular_layout(wa, dev)
    ref_b = regular_layout(wb, dev)
    for w, ref in ((wa, ref_a), (wb, ref_b)):
        slots, U = noalloc_layout(w.cand_idx, w.shape[2], dev)
        np.testing.assert_array_equal(U, ref[1])
        np.testing.assert_array_equal(slots, ref[0])
    # and the first batch once more, after the larger second one
    slots, U = noalloc_layout(wa.cand_idx, wa.shape[2], dev)
    np.testing.assert_array_equal(U, ref_a[1])
    np.testing.assert_array_equal(slots, ref_a[0])


def test_noalloc_marks_bad_requests(dev):
    w = wl.make_workload("serving", B=4)
    cand = w.cand_idx.copy()
    cand[1, 3, 2] = w.shape[2]
    slots, U = noalloc_layout(cand, w.shape[2], dev)
    assert U[1] == 0 and (slots[1] == -1).all()
    ref_slots, ref_U = regular_layout(w, dev)
    np.testing.assert_array_equal(U[[0, 2, 3]], ref_U[[0, 2, 3]])
    np.testing.assert_array_equal(slots[[0, 2, 3]], ref_slots[[0, 2, 3]])


def test_noalloc_rejects_batches_beyond_the_fixed_scratch(dev):
    from paper_2603_02565_gb300.binding import FE_ERR_UNSUPPORTED, load_library
    lib = load_library()
    # B * min(M, K*L) = 2048 * 600 > 1048576: refused before anything is enqueued
    rc = lib.fe_distinct_layout_noalloc(None, 2048, 600, 100, 10, None, None, None)
    assert rc == FE_ERR_UNSUPPORTED
    rc = lib.fe_distinct_layout_noalloc(None, 70000, 10, 1, 1, None, None, None)
    assert rc == FE_ERR_UNSUPPORTED
