"""Python binding of libfe.so: argument marshalling only.

Every step of the evaluation runs in the library's CUDA kernels; this module
packs the weights in the order fe.h documents, passes device pointers of torch
tensors (or host buffers) through ctypes and turns return codes into
exceptions.  It never computes anything itself and has no fallback: without
the built library every call raises.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libfe.so")

FE_OK = 0
FE_ERR_INVALID_ARG = 1
FE_ERR_UNSUPPORTED = 2
FE_ERR_INDEX = 3
FE_ERR_WORKSPACE = 4
FE_ERR_OOM = 5
FE_ERR_CUDA = 6
FE_ERR_NUMERIC = 7
FE_ERR_TIMEOUT = 8
FE_IO_BF16 = 0
FE_IO_F32 = 1

EXPORTS = ["fe_weight_count", "fe_init", "fe_reserve", "fe_evaluate", "fe_evaluate_async", "fe_last_status",
           "fe_evaluate_host", "fe_evaluate_factorized", "fe_submit_host", "fe_wait_host", "fe_debug_layout",
           "fe_debug_fetch", "fe_profile",
           "fe_profile_read",
           "fe_kernels_per_batch", "fe_distinct_layout_noalloc", "fe_destroy", "fe_strerror",
           "fe_last_error_message", "fe_blob_parse", "fe_init_blob", "fe_debug_alloc_hook",
           "fe_debug_wait_probe", "fe_debug_keep_intermediates"]


class FeConfig(ctypes.Structure):
    _fields_ = [("d", ctypes.c_int32), ("n_heads", ctypes.c_int32), ("n_layers", ctypes.c_int32),
                ("ffn_mult", ctypes.c_int32), ("max_L", ctypes.c_int32), ("io_dtype", ctypes.c_int32),
                ("ln_eps", ctypes.c_float), ("n_tasks", ctypes.c_int32), ("no_cross_seq", ctypes.c_int32),
                ("elem_self_attn", ctypes.c_int32), ("encode_pool", ctypes.c_int32),
                ("linear_context_attn", ctypes.c_int32)]


class FeError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__(f"fe error {code}: {msg}")
        self.code = code


_lib = None


def load_library(path: str = LIB_PATH):
    """Load libfe.so and declare every entry point of fe.h."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise ImportError(f"{path} is not built; run paper_2603_02565_gb300.build.build()")
    L = ctypes.CDLL(path)
    vp, i32, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t
    L.fe_weight_count.argtypes = [ctypes.POINTER(FeConfig)]
    L.fe_weight_count.restype = sz
    L.fe_init.argtypes = [ctypes.POINTER(FeConfig), ctypes.POINTER(ctypes.c_float), sz, ctypes.POINTER(vp)]
    L.fe_init.restype = i32
    L.fe_blob_parse.argtypes = [vp, sz, ctypes.POINTER(FeConfig), ctypes.POINTER(sz)]
    L.fe_blob_parse.restype = i32
    L.fe_init_blob.argtypes = [vp, sz, ctypes.POINTER(vp)]
    L.fe_init_blob.restype = i32
    L.fe_debug_alloc_hook.argtypes = [i32, ctypes.POINTER(ctypes.c_int64)]
    L.fe_debug_alloc_hook.restype = i32
    L.fe_debug_wait_probe.argtypes = [vp, ctypes.c_uint32, vp]
    L.fe_debug_wait_probe.restype = i32
    L.fe_debug_keep_intermediates.argtypes = [vp, i32]
    L.fe_debug_keep_intermediates.restype = i32
    L.fe_reserve.argtypes = [vp, i32, i32, i32, i32, i32]
    L.fe_reserve.restype = i32
    for name in ("fe_evaluate", "fe_evaluate_async", "fe_evaluate_host", "fe_evaluate_factorized"):
        f = getattr(L, name)
        f.argtypes = [vp, i32, i32, i32, i32, i32, vp, vp, vp, vp, vp, vp]
        f.restype = i32
    L.fe_last_status.argtypes = [vp]
    L.fe_last_status.restype = i32
    L.fe_submit_host.argtypes = [vp, i32, i32, i32, i32, i32, vp, vp, vp, vp, vp]
    L.fe_submit_host.restype = i32
    L.fe_wait_host.argtypes = [vp]
    L.fe_wait_host.restype = i32
    L.fe_debug_layout.argtypes = [vp, vp, vp]
    L.fe_debug_layout.restype = i32
    L.fe_debug_fetch.argtypes = [vp, ctypes.c_char_p, vp, sz, ctypes.POINTER(sz)]
    L.fe_debug_fetch.restype = i32
    L.fe_profile.argtypes = [vp, i32]
    L.fe_profile.restype = i32
    L.fe_profile_read.argtypes = [vp, i32, vp, vp, vp, ctypes.POINTER(i32)]
    L.fe_profile_read.restype = i32
    L.fe_kernels_per_batch.argtypes = [vp]
    L.fe_kernels_per_batch.restype = i32
    L.fe_distinct_layout_noalloc.argtypes = [vp, i32, i32, i32, i32, vp, vp, vp]
    L.fe_distinct_layout_noalloc.restype = i32
    L.fe_destroy.argtypes = [vp]
    L.fe_destroy.restype = i32
    L.fe_strerror.argtypes = [i32]
    L.fe_strerror.restype = ctypes.c_char_p
    L.fe_last_error_message.argtypes = []
    L.fe_last_error_message.restype = ctypes.c_char_p
    _lib = L
    return L


def _check(rc, allowed=(FE_OK,)):
    if rc not in allowed:
        L = load_library()
        raise FeError(rc, f"{L.fe_strerror(rc).decode()} ({L.fe_last_error_message().decode()})")
    return rc


def weight_order(n_layers: int, n_tasks: int = 1, cross_seq: bool = True, elem_self_attn: bool = False):
    """Tensor names in the order fe.h documents for fe_init."""
    names = []
    for l in range(n_layers):
        names += [f"WQ.{l}", f"WK.{l}", f"WV.{l}", f"WO.{l}", f"W1.{l}", f"b1.{l}", f"W2.{l}", f"b2.{l}"]
    names += ["P", "cls", "WQs", "WKs", "WVs", "WOs", "W1s", "b1s", "W2s", "b2s"]
    if cross_seq:
        names += ["WQx", "WKx", "WVx", "WOx"]
    if n_tasks == 1:
        names += ["W1h", "b1h", "w2h", "b2h"]
    else:
        for t in range(n_tasks):
            names += [f"W1h.{t}", f"b1h.{t}", f"w2h.{t}", f"b2h.{t}"]
        names += ["fuse_w", "fuse_b"]
    if elem_self_attn:
        names += ["WQe", "WKe", "WVe", "WOe"]
    return names


def _tasks(cfg):
    return int(getattr(cfg, "n_tasks", 1))


def _cross(cfg):
    return bool(getattr(cfg, "cross_seq", True))


def _flag(cfg, name):
    return 1 if getattr(cfg, name, False) else 0


def make_config(cfg) -> FeConfig:
    """fe_config from any object with d, n_heads, n_layers, ffn_mult, max_L, io_bf16, ln_eps
    (and optionally n_tasks, cross_seq, elem_self_attn, encode_pool, linear_context_attn)."""
    return FeConfig(cfg.d, cfg.n_heads, cfg.n_layers, cfg.ffn_mult, cfg.max_L,
                    FE_IO_BF16 if cfg.io_bf16 else FE_IO_F32, cfg.ln_eps, _tasks(cfg), 0 if _cross(cfg) else 1,
                    _flag(cfg, "elem_self_attn"), _flag(cfg, "encode_pool"), _flag(cfg, "linear_context_attn"))


def pack_weights(cfg, weights: dict) -> np.ndarray:
    parts = [np.ascontiguousarray(weights[n], dtype=np.float32).ravel()
             for n in weight_order(cfg.n_layers, _tasks(cfg), _cross(cfg), bool(_flag(cfg, "elem_self_attn")))]
    return np.concatenate(parts)


BLOB_MAGIC = b"FEW1"
BLOB_VERSION = 1


def weights_blob(cfg, weights: dict) -> bytes:
    """The weight blob of fe.h (magic, version, the fe_config fields, the
    weight count, then the fp32 weights in fe_init's order), little-endian."""
    import struct
    c = make_config(cfg)
    flat = pack_weights(cfg, weights).astype("<f4", copy=False)
    head = BLOB_MAGIC + struct.pack("<I", BLOB_VERSION)
    head += struct.pack("<6if5i", c.d, c.n_heads, c.n_layers, c.ffn_mult, c.max_L, c.io_dtype, c.ln_eps, c.n_tasks,
                        c.no_cross_seq, c.elem_self_attn, c.encode_pool, c.linear_context_attn)
    head += struct.pack("<Q", flat.size)
    return head + flat.tobytes()


def save_blob(path: str, cfg, weights: dict) -> None:
    with open(path, "wb") as f:
        f.write(weights_blob(cfg, weights))


class BlobConfig:
    """The configuration read from a weight blob by fe_blob_parse, with the
    attribute names the rest of this module uses."""

    def __init__(self, c: FeConfig):
        self.d, self.n_heads, self.n_layers = c.d, c.n_heads, c.n_layers
        self.ffn_mult, self.max_L, self.ln_eps = c.ffn_mult, c.max_L, c.ln_eps
        self.io_bf16 = c.io_dtype == FE_IO_BF16
        self.n_tasks = max(c.n_tasks, 1)
        self.cross_seq = c.no_cross_seq == 0
        self.elem_self_attn = bool(c.elem_self_attn)
        self.encode_pool = bool(c.encode_pool)
        self.linear_context_attn = bool(c.linear_context_attn)
        self.F = c.ffn_mult * c.d


def parse_blob(blob: bytes):
    """(BlobConfig, weight count) of a blob, checked by the library's parser."""
    L = load_library()
    c = FeConfig()
    n = ctypes.c_size_t()
    buf = ctypes.create_string_buffer(bytes(blob), len(blob))
    _check(L.fe_blob_parse(buf, len(blob), ctypes.byref(c), ctypes.byref(n)))
    return BlobConfig(c), n.value


def _ptr(t):
    return ctypes.c_void_p(0 if t is None else t.data_ptr())


class Evaluator:
    """One library context: weights on the device plus a reusable workspace."""

    @classmethod
    def from_blob(cls, blob: bytes):
        """A context from a weight blob (fe_init_blob); the configuration is the blob's."""
        L = load_library()
        cfg, _ = parse_blob(blob)
        self = cls.__new__(cls)
        self.cfg = cfg
        buf = ctypes.create_string_buffer(bytes(blob), len(blob))
        h = ctypes.c_void_p()
        _check(L.fe_init_blob(buf, len(blob), ctypes.byref(h)))
        self._h = h
        self.last_status = FE_OK
        return self

    def __init__(self, cfg, weights: dict):
        L = load_library()
        self.cfg = cfg
        self._c = make_config(cfg)
        flat = pack_weights(cfg, weights)
        need = L.fe_weight_count(ctypes.byref(self._c))
        if need != flat.size:
            raise FeError(FE_ERR_INVALID_ARG, f"weights have {flat.size} floats, library expects {need}")
        h = ctypes.c_void_p()
        _check(L.fe_init(ctypes.byref(self._c), flat.ctypes.data_as(ctypes.POINTER(ctypes.c_float)),
                         flat.size, ctypes.byref(h)))
        self._h = h
        self.last_status = FE_OK

    # -- lifetime -------------------------------------------------------------
    def close(self):
        if getattr(self, "_h", None):
            load_library().fe_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def reserve(self, B, C, M, K, L):
        _check(load_library().fe_reserve(self._h, B, C, M, K, L))

    # -- evaluation -------------------------------------------------------------
    def evaluate(self, context, pool, cand_idx, scores=None, best=None, stream=None, sync=True,
                 allowed=(FE_OK, FE_ERR_INDEX, FE_ERR_NUMERIC), factorized=False):
        """context [B,C,d], pool [B,M,d] (bf16 or fp32 per the config), cand_idx [B,K,L]
        int32, all CUDA tensors.  Returns (scores [B,K] fp32, best [B] int32).
        factorized=True runs the candidate-factorized evaluation E^ind
        (fe_evaluate_factorized): same outputs, per-sequence cost structure."""
        import torch
        B, C, _ = context.shape
        M = pool.shape[1]
        K, L = cand_idx.shape[1], cand_idx.shape[2]
        dev = context.device
        if scores is None:
            scores = torch.empty((B, K), dtype=torch.float32, device=dev)
        if best is None:
            best = torch.empty((B,), dtype=torch.int32, device=dev)
        for t in (context, pool, cand_idx, scores, best):
            if not t.is_cuda or not t.is_contiguous():
                raise ValueError("evaluate expects contiguous CUDA tensors")
        if cand_idx.dtype != torch.int32:
            raise ValueError("cand_idx must be int32")
        want = torch.bfloat16 if self.cfg.io_bf16 else torch.float32
        if context.dtype != want or pool.dtype != want:
            raise ValueError(f"context and pool must be {want}")
        if stream is None:
            stream = torch.cuda.current_stream(dev).cuda_stream
        Lb = load_library()
        fn = Lb.fe_evaluate_factorized if factorized else (Lb.fe_evaluate if sync else Lb.fe_evaluate_async)
        rc = fn(self._h, B, C, M, K, L, _ptr(context), _ptr(pool), _ptr(cand_idx), _ptr(scores), _ptr(best),
                ctypes.c_void_p(stream))
        if factorized and sync and rc == FE_OK:
            rc = Lb.fe_last_status(self._h)
        self.last_status = _check(rc, allowed)
        return scores, best

    def wait(self, allowed=(FE_OK, FE_ERR_INDEX, FE_ERR_NUMERIC)):
        """Status of the last evaluate(..., sync=False), after waiting for it."""
        self.last_status = _check(load_library().fe_last_status(self._h), allowed)
        return self.last_status

    def evaluate_host(self, context, pool, cand_idx, scores=None, best=None, stream=0,
                      allowed=(FE_OK, FE_ERR_INDEX, FE_ERR_NUMERIC)):
        """Same as evaluate for host buffers (numpy arrays or CPU tensors, pinned or
        not); the library copies in and out.  context/pool must already hold the
        config's element type (uint16 bf16 bits, a bfloat16 tensor, or float32)."""
        B, C, _ = context.shape
        M = pool.shape[1]
        K, L = cand_idx.shape[1], cand_idx.shape[2]
        if scores is None:
            scores = np.empty((B, K), dtype=np.float32)
        if best is None:
            best = np.empty((B,), dtype=np.int32)

        def hp(a):
            if hasattr(a, "data_ptr"):
                return ctypes.c_void_p(a.data_ptr())
            return ctypes.c_void_p(a.ctypes.data)

        rc = load_library().fe_evaluate_host(self._h, B, C, M, K, L, hp(context), hp(pool), hp(cand_idx),
                                             hp(scores), hp(best), ctypes.c_void_p(stream))
        self.last_status = _check(rc, allowed)
        return scores, best

    def submit_host(self, context, pool, cand_idx, scores, best):
        """Pipelined host entry: enqueue one batch whose buffers live in host memory
        and return at once (fe_submit_host).  scores [B, K] float32 and best [B]
        int32 are host buffers the results are copied into; every buffer must stay
        alive and unchanged until the matching wait_host() returns."""
        B, C, _ = context.shape
        M = pool.shape[1]
        K, L = cand_idx.shape[1], cand_idx.shape[2]

        def hp(a):
            if hasattr(a, "data_ptr"):
                return ctypes.c_void_p(a.data_ptr())
            return ctypes.c_void_p(a.ctypes.data)

        _check(load_library().fe_submit_host(self._h, B, C, M, K, L, hp(context), hp(pool), hp(cand_idx),
                                             hp(scores), hp(best)))

    def wait_host(self, allowed=(FE_OK, FE_ERR_INDEX, FE_ERR_NUMERIC)):
        """Wait for the oldest outstanding submit_host batch; returns its status."""
        self.last_status = _check(load_library().fe_wait_host(self._h), allowed)
        return self.last_status

    # -- tracing ----------------------------------------------------------------------
    def profile(self, enable: bool):
        _check(load_library().fe_profile(self._h, 1 if enable else 0))

    def profile_read(self, max_sites: int = 64):
        """[(site, launches, total_ms)] since the last read, in launch order."""
        names = ctypes.create_string_buffer(32 * max_sites)
        launches = np.zeros(max_sites, dtype=np.int32)
        total = np.zeros(max_sites, dtype=np.float64)
        n = ctypes.c_int()
        _check(load_library().fe_profile_read(self._h, max_sites, names, ctypes.c_void_p(launches.ctypes.data),
                                              ctypes.c_void_p(total.ctypes.data), ctypes.byref(n)))
        raw = names.raw
        out = []
        for i in range(min(n.value, max_sites)):
            nm = raw[32 * i:32 * (i + 1)].split(b"\0", 1)[0].decode()
            out.append((nm, int(launches[i]), float(total[i])))
        return out

    def keep_intermediates(self, on: bool = True):
        """Store c and C' for fetch("seq") / fetch("cross") in later batches even
        where the sequence-stage kernel keeps them on chip (a test hook)."""
        _check(load_library().fe_debug_keep_intermediates(self._h, 1 if on else 0))

    def kernels_per_batch(self) -> int:
        return int(load_library().fe_kernels_per_batch(self._h))

    # -- test hooks ---------------------------------------------------------------
    def layout(self, B, K, L):
        slots = np.empty((B, K, L), dtype=np.int32)
        U = np.empty((B,), dtype=np.int32)
        _check(load_library().fe_debug_layout(self._h, ctypes.c_void_p(slots.ctypes.data),
                                              ctypes.c_void_p(U.ctypes.data)))
        return slots, U

    def fetch(self, name: str, cols: int | None = None):
        Lb = load_library()
        n = ctypes.c_size_t()
        _check(Lb.fe_debug_fetch(self._h, name.encode(), None, 0, ctypes.byref(n)))
        out = np.empty(n.value, dtype=np.float32)
        _check(Lb.fe_debug_fetch(self._h, name.encode(), ctypes.c_void_p(out.ctypes.data), out.size,
                                 ctypes.byref(n)))
        c = cols or self.cfg.d
        return out.reshape(-1, c) if out.size else out.reshape(0, c)
