"""The C-ABI library builds for sm_103a, loads, and exports every entry point
that include/fe.h declares.  Host-only calls; no GPU needed."""
import ctypes
import os
import re

import pytest

from paper_2603_02565_gb300 import binding, build as fe_build
from paper_2603_02565_gb300 import workloads as wl

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    text = open(os.path.join(ROOT, "include", "fe.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(fe_[a-z_]+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    fe_build.build()
    return binding.load_library()


def test_header_and_binding_agree():
    assert declared_functions() == sorted(binding.EXPORTS)


def test_every_declared_symbol_is_exported(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_weight_count_matches_parameter_inventory(lib):
    for name, kw in [("tiny", {}), ("serving", dict(B=1)), ("stress", dict(B=1))]:
        w = wl.make_workload(name, **kw)
        c = binding.make_config(w.cfg)
        n = sum(a.size for a in w.weights.values())
        assert lib.fe_weight_count(ctypes.byref(c)) == n
        assert binding.pack_weights(w.cfg, w.weights).size == n


def test_unsupported_configs_are_rejected(lib):
    for bad in [dict(d=96), dict(d=128, n_heads=8), dict(d=128, n_heads=4, n_layers=0),
                dict(d=128, n_heads=4, max_L=0)]:
        cfg = dict(d=128, n_heads=4, n_layers=2, ffn_mult=4, max_L=8, io_dtype=0, ln_eps=1e-5)
        cfg.update(bad)
        c = binding.FeConfig(**cfg)
        assert lib.fe_weight_count(ctypes.byref(c)) == 0


def test_errors_have_names(lib):
    for code in range(9):
        assert lib.fe_strerror(code).decode() not in ("", "unknown error")
    assert lib.fe_strerror(99).decode() == "unknown error"


def test_init_argument_errors_fail_loudly(lib):
    w = wl.make_workload("tiny")
    c = binding.make_config(w.cfg)
    h = ctypes.c_void_p()
    flat = binding.pack_weights(w.cfg, w.weights)
    ptr = flat.ctypes.data_as(ctypes.POINTER(ctypes.c_float))
    assert lib.fe_init(ctypes.byref(c), ptr, flat.size - 1, ctypes.byref(h)) == binding.FE_ERR_INVALID_ARG
    assert lib.fe_init(None, ptr, flat.size, ctypes.byref(h)) == binding.FE_ERR_INVALID_ARG
