"""Reader of the library's weight blob, for the oracle (test infrastructure).

The blob carries the parameters theta of E_theta (Section 3) with the
configuration they belong to.  The paper defines no storage format; this
reader follows the library's (magic "FEW1", a version, the configuration
fields, the weight count, then the fp32 weights in a fixed tensor order, all
little-endian) and is written separately from the library's writer and
parser, so that a test can check the three against each other.  Only the
test suite may use it.
"""
from __future__ import annotations

import struct
import types

import numpy as np

HEADER_BYTES = 64


def tensor_list(d, F, n_layers, max_L, n_tasks, cross_seq, elem_self_attn):
    """(name, shape) of every parameter in blob order: the element stack per
    layer (Section 4.2), SeqEnc with positions and [CLS] (Section 4.3), the
    cross-sequence block and the head(s) with the fusion (Section 4.4), and
    the element self-attention H^(1) last."""
    out = []
    for l in range(n_layers):
        out += [(f"WQ.{l}", (d, d)), (f"WK.{l}", (d, d)), (f"WV.{l}", (d, d)), (f"WO.{l}", (d, d)),
                (f"W1.{l}", (d, F)), (f"b1.{l}", (F,)), (f"W2.{l}", (F, d)), (f"b2.{l}", (d,))]
    out += [("P", (max_L, d)), ("cls", (d,))]
    out += [(n, (d, d)) for n in ("WQs", "WKs", "WVs", "WOs")]
    out += [("W1s", (d, F)), ("b1s", (F,)), ("W2s", (F, d)), ("b2s", (d,))]
    if cross_seq:
        out += [(n, (d, d)) for n in ("WQx", "WKx", "WVx", "WOx")]
    if n_tasks <= 1:
        out += [("W1h", (d, d)), ("b1h", (d,)), ("w2h", (d,)), ("b2h", (1,))]
    else:
        for t in range(n_tasks):
            out += [(f"W1h.{t}", (d, d)), (f"b1h.{t}", (d,)), (f"w2h.{t}", (d,)), (f"b2h.{t}", (1,))]
        out += [("fuse_w", (n_tasks,)), ("fuse_b", (1,))]
    if elem_self_attn:
        out += [(n, (d, d)) for n in ("WQe", "WKe", "WVe", "WOe")]
    return out


def read_blob(data: bytes):
    """(cfg, weights) from a blob: cfg has the attributes the oracle reads
    (d, n_heads, n_layers, ffn_mult, max_L, io_bf16, ln_eps, n_tasks,
    cross_seq, elem_self_attn, encode_pool, linear_context_attn); weights maps
    every tensor name to a float32 array.  Raises ValueError on a malformed blob."""
    if len(data) < HEADER_BYTES or data[:4] != b"FEW1":
        raise ValueError("not a FEW1 weight blob")
    (version,) = struct.unpack_from("<I", data, 4)
    if version != 1:
        raise ValueError(f"blob version {version}")
    d, H, Ly, fm, max_L, io = struct.unpack_from("<6i", data, 8)
    (eps,) = struct.unpack_from("<f", data, 32)
    T, no_cross, esa, pool_set, lin = struct.unpack_from("<5i", data, 36)
    (n,) = struct.unpack_from("<Q", data, 56)
    if len(data) != HEADER_BYTES + 4 * n:
        raise ValueError("blob size does not match its weight count")
    cfg = types.SimpleNamespace(d=d, n_heads=H, n_layers=Ly, ffn_mult=fm, max_L=max_L, io_bf16=(io == 0),
                                ln_eps=float(eps), n_tasks=max(T, 1), cross_seq=(no_cross == 0),
                                elem_self_attn=bool(esa), encode_pool=bool(pool_set),
                                linear_context_attn=bool(lin), F=fm * d)
    flat = np.frombuffer(data, dtype="<f4", count=n, offset=HEADER_BYTES)
    names = tensor_list(d, fm * d, Ly, max_L, cfg.n_tasks, cfg.cross_seq, cfg.elem_self_attn)
    if sum(int(np.prod(s)) for _, s in names) != n:
        raise ValueError("weight count does not match the configuration")
    weights, o = {}, 0
    for name, shape in names:
        k = int(np.prod(shape))
        weights[name] = flat[o:o + k].reshape(shape).astype(np.float32)
        o += k
    return cfg, weights
