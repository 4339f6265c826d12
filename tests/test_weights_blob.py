"""The weight blob (magic FEW1, version, configuration, count, fp32 weights):
the package's writer, the library's parser (host only, fe_blob_parse) and
the oracle's own reader agree, and malformed blobs are refused.  CPU only."""
import ctypes
import dataclasses
import struct

import numpy as np
import pytest

from oracle import fe_oracle as O
from oracle.weights_blob import read_blob
from paper_2603_02565_gb300 import binding, build as fe_build
from paper_2603_02565_gb300 import workloads as wl

CASES = [("tiny", {}), ("serving", dict(B=2)), ("serving", dict(B=2, n_tasks=3, cross_seq=False)),
         ("serving", dict(B=2, elem_self_attn=True, encode_pool=True)),
         ("serving", dict(B=2, linear_context_attn=True))]


@pytest.fixture(scope="module")
def lib():
    fe_build.build()
    return binding.load_library()


def _cfg_fields(cfg):
    return (cfg.d, cfg.n_heads, cfg.n_layers, cfg.ffn_mult, cfg.max_L, bool(cfg.io_bf16), np.float32(cfg.ln_eps),
            max(int(getattr(cfg, "n_tasks", 1)), 1), bool(getattr(cfg, "cross_seq", True)),
            bool(getattr(cfg, "elem_self_attn", False)), bool(getattr(cfg, "encode_pool", False)),
            bool(getattr(cfg, "linear_context_attn", False)))


@pytest.mark.parametrize("name,kw", CASES)
def test_oracle_reads_what_the_package_writes(name, kw, tmp_path):
    w = wl.make_workload(name, **kw)
    path = tmp_path / "w.few1"
    binding.save_blob(str(path), w.cfg, w.weights)
    data = path.read_bytes()
    cfg, weights = read_blob(data)
    assert _cfg_fields(cfg) == _cfg_fields(w.cfg)
    assert weights.keys() == w.weights.keys()
    for k in weights:
        assert weights[k].shape == w.weights[k].shape
        assert np.array_equal(weights[k].view(np.uint32), np.asarray(w.weights[k], np.float32).view(np.uint32))
    # the oracle gives bitwise the same scores from the blob's weights and configuration
    # (the blob holds ln_eps as the library's float32)
    cfg32 = dataclasses.replace(w.cfg, ln_eps=float(np.float32(w.cfg.ln_eps)))
    s0, b0, _, _ = O.evaluate(w.context[:1], w.pool[:1], w.cand_idx[:1], w.weights, cfg32)
    s1, b1, _, _ = O.evaluate(w.context[:1], w.pool[:1], w.cand_idx[:1], weights, cfg)
    assert np.array_equal(s0, s1, equal_nan=True) and np.array_equal(b0, b1)


@pytest.mark.parametrize("name,kw", CASES)
def test_library_parser_agrees(name, kw, lib):
    w = wl.make_workload(name, **kw)
    blob = binding.weights_blob(w.cfg, w.weights)
    cfg, n = binding.parse_blob(blob)
    assert _cfg_fields(cfg) == _cfg_fields(w.cfg)
    assert n == sum(a.size for a in w.weights.values())
    assert len(blob) == 64 + 4 * n
    # the weights start at byte 64, in fe_init's order
    flat = np.frombuffer(blob, dtype="<f4", offset=64)
    assert np.array_equal(flat, binding.pack_weights(w.cfg, w.weights))


def _parse_rc(lib, blob):
    c = binding.FeConfig()
    n = ctypes.c_size_t()
    buf = ctypes.create_string_buffer(bytes(blob), max(len(blob), 1))
    return lib.fe_blob_parse(buf, len(blob), ctypes.byref(c), ctypes.byref(n))


def test_malformed_blobs_are_refused(lib):
    w = wl.make_workload("tiny")
    good = binding.weights_blob(w.cfg, w.weights)
    assert _parse_rc(lib, good) == binding.FE_OK
    bad_magic = b"FEW0" + good[4:]
    v2 = good[:4] + struct.pack("<I", 2) + good[8:]
    truncated = good[:-4]
    extra = good + b"\0\0\0\0"
    short = good[:60]
    count_off = good[:56] + struct.pack("<Q", (len(good) - 64) // 4 + 1) + good[64:]
    d96 = good[:8] + struct.pack("<i", 96) + good[12:]
    heads3 = good[:12] + struct.pack("<i", 3) + good[16:]
    assert _parse_rc(lib, bad_magic) == binding.FE_ERR_INVALID_ARG
    assert _parse_rc(lib, v2) == binding.FE_ERR_UNSUPPORTED
    assert _parse_rc(lib, truncated) == binding.FE_ERR_INVALID_ARG
    assert _parse_rc(lib, extra) == binding.FE_ERR_INVALID_ARG
    assert _parse_rc(lib, short) == binding.FE_ERR_INVALID_ARG
    assert _parse_rc(lib, count_off) == binding.FE_ERR_INVALID_ARG
    assert _parse_rc(lib, d96) == binding.FE_ERR_UNSUPPORTED
    assert _parse_rc(lib, heads3) == binding.FE_ERR_UNSUPPORTED
    assert lib.fe_blob_parse(None, 64, None, None) == binding.FE_ERR_INVALID_ARG
    for blob in (bad_magic, v2, truncated):
        with pytest.raises(ValueError):
            read_blob(blob)
    h = ctypes.c_void_p()
    buf = ctypes.create_string_buffer(bad_magic, len(bad_magic))
    assert lib.fe_init_blob(buf, len(bad_magic), ctypes.byref(h)) == binding.FE_ERR_INVALID_ARG
    assert not h.value
