"""Seeded synthetic workloads for the joint evaluator.

This module only draws numbers: request contexts, candidate pools, candidate
index tensors and model parameters, shaped like the paper's workloads (Table 1
dataset shapes; the online setting of Appendix B.3 with K=50 sequences; the
CNN/DailyMail reranking setting of Appendix B.1).  It holds none of the
evaluator's arithmetic, so both the CPU oracle and the CUDA path consume its
output without sharing any computation.

Conventions
-----------
* Every floating-point array is float32.  For the bf16 workloads every value
  is first rounded (round-to-nearest-even) to a bf16-representable number, so
  the CUDA path ingests exactly the values the oracle sees.
* Parameters follow y = x @ W with W stored [in, out].
* ``cand_idx[b, k, j]`` indexes row ``pool[b, cand_idx[b, k, j]]``.
"""
from __future__ import annotations

import dataclasses
import numpy as np

__all__ = ["ModelConfig", "Workload", "round_to_bf16", "make_weights",
           "make_workload", "WORKLOADS", "param_shapes"]


@dataclasses.dataclass(frozen=True)
class ModelConfig:
    d: int            # model width
    n_heads: int      # attention heads (d_h = d / n_heads)
    n_layers: int     # depth of the item cross-attention stack
    ffn_mult: int = 4  # FFN width F = ffn_mult * d
    max_L: int = 64   # rows of the position-embedding table
    io_bf16: bool = True  # inputs are bf16-valued (False: plain fp32 inputs)
    ln_eps: float = 1e-5
    n_tasks: int = 1      # task-specific prediction heads; > 1 adds the fusion module
    cross_seq: bool = True  # False: the variant without cross-sequence interaction
    elem_self_attn: bool = False  # self-attention H^(1) over the element set
    encode_pool: bool = False     # the element set is the whole pool (U = M)
    linear_context_attn: bool = False  # linear attention in the element -> context attention

    @property
    def F(self) -> int:
        return self.ffn_mult * self.d


@dataclasses.dataclass
class Workload:
    name: str
    cfg: ModelConfig
    context: np.ndarray   # [B, C, d] float32
    pool: np.ndarray      # [B, M, d] float32
    cand_idx: np.ndarray  # [B, K, L] int32
    weights: dict         # name -> float32 array

    @property
    def shape(self):
        B, C, _ = self.context.shape
        M = self.pool.shape[1]
        K, L = self.cand_idx.shape[1:]
        return B, C, M, K, L


def round_to_bf16(x: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bf16 value (ties to even), kept as float32."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    lsb = (u >> 16) & 1
    u = (u + 0x7FFF + lsb) >> 16 << 16
    return (u & 0xFFFFFFFF).astype(np.uint32).view(np.float32)


def param_shapes(cfg: ModelConfig):
    """(name, shape) of every parameter, in a fixed draw order."""
    d, F = cfg.d, cfg.F
    out = []
    for l in range(cfg.n_layers):
        out += [(f"WQ.{l}", (d, d)), (f"WK.{l}", (d, d)), (f"WV.{l}", (d, d)),
                (f"WO.{l}", (d, d)), (f"W1.{l}", (d, F)), (f"b1.{l}", (F,)),
                (f"W2.{l}", (F, d)), (f"b2.{l}", (d,))]
    out += [("P", (cfg.max_L, d)), ("cls", (d,)),
            ("WQs", (d, d)), ("WKs", (d, d)), ("WVs", (d, d)), ("WOs", (d, d)),
            ("W1s", (d, F)), ("b1s", (F,)), ("W2s", (F, d)), ("b2s", (d,))]
    if cfg.cross_seq:
        out += [("WQx", (d, d)), ("WKx", (d, d)), ("WVx", (d, d)), ("WOx", (d, d))]
    if cfg.n_tasks == 1:
        out += [("W1h", (d, d)), ("b1h", (d,)), ("w2h", (d,)), ("b2h", (1,))]
    else:
        for t in range(cfg.n_tasks):
            out += [(f"W1h.{t}", (d, d)), (f"b1h.{t}", (d,)), (f"w2h.{t}", (d,)), (f"b2h.{t}", (1,))]
        out += [("fuse_w", (cfg.n_tasks,)), ("fuse_b", (1,))]
    if cfg.elem_self_attn:
        out += [("WQe", (d, d)), ("WKe", (d, d)), ("WVe", (d, d)), ("WOe", (d, d))]
    return out


def make_weights(cfg: ModelConfig, rng: np.random.Generator, std: float = 0.02) -> dict:
    """Every parameter (biases, position table and [CLS] included) ~ N(0, std),
    except the fusion weights of a multi-task head, which are positive task
    importances ~ U(0.5, 1.5)."""
    w = {}
    for name, shape in param_shapes(cfg):
        if name == "fuse_w":
            a = rng.uniform(0.5, 1.5, size=shape).astype(np.float32)
        else:
            a = rng.normal(0.0, std, size=shape).astype(np.float32)
        w[name] = round_to_bf16(a) if cfg.io_bf16 else a
    return w


def _plackett_luce_rows(rng, logp, n_rows, L):
    """Draw n_rows sequences of L distinct indices, each drawn in turn with
    probability proportional to exp(logp) over the indices not yet drawn.
    Uses the Gumbel-top-L construction, which gives exactly that sequential
    without-replacement distribution, in draw order."""
    g = rng.gumbel(size=(n_rows, logp.shape[-1]))
    keys = logp + g
    top = np.argpartition(-keys, L - 1, axis=1)[:, :L]
    order = np.argsort(-np.take_along_axis(keys, top, axis=1), axis=1, kind="stable")
    return np.take_along_axis(top, order, axis=1)


def sample_sequences(rng, B, M, K, L, zipf_s=None):
    """cand_idx [B, K, L]: per sequence, L distinct pool rows.  zipf_s=None is
    uniform; otherwise rank r (1-based) has weight r**-zipf_s and ranks map to
    pool rows through a per-request random permutation."""
    if L > M:
        raise ValueError("L > M: cannot sample without replacement")
    if zipf_s is None:
        logp = np.zeros(M)
    else:
        logp = -zipf_s * np.log(np.arange(1, M + 1, dtype=np.float64))
    out = np.empty((B, K, L), dtype=np.int32)
    for b in range(B):
        ranks = _plackett_luce_rows(rng, logp, K, L)
        perm = rng.permutation(M)
        out[b] = perm[ranks]
    return out


def _normal(rng, shape, std, bf16):
    a = rng.normal(0.0, std, size=shape).astype(np.float32)
    return round_to_bf16(a) if bf16 else a


def _rec_workload(name, seed, B, C, d, H, Ly, M, K, L, zipf_s, ctx_std, pool_std,
                  io_bf16=True, idx_seed=None, max_L=None, n_tasks=1, cross_seq=True,
                  elem_self_attn=False, encode_pool=False, linear_context_attn=False):
    cfg = ModelConfig(d=d, n_heads=H, n_layers=Ly, max_L=max_L or L, io_bf16=io_bf16,
                      n_tasks=n_tasks, cross_seq=cross_seq, elem_self_attn=elem_self_attn,
                      encode_pool=encode_pool, linear_context_attn=linear_context_attn)
    rng = np.random.default_rng(seed)
    weights = make_weights(cfg, rng)
    context = _normal(rng, (B, C, d), ctx_std, io_bf16)
    pool = _normal(rng, (B, M, d), pool_std, io_bf16)
    irng = rng if idx_seed is None else np.random.default_rng(idx_seed)
    cand = sample_sequences(irng, B, M, K, L, zipf_s)
    return Workload(name, cfg, context, pool, cand, weights)


def tiny(seed=0, **kw):
    """Tiny fp32 case: B=1, C=16, d=32, 1 head, 1 layer, M=20, K=4, L=5,
    uniform sampling; all embeddings and parameters ~ N(0, 0.02)."""
    p = dict(B=1, C=16, d=32, H=1, Ly=1, M=20, K=4, L=5)
    p.update(kw)
    return _rec_workload("tiny", seed, zipf_s=None, ctx_std=0.02, pool_std=0.02,
                         io_bf16=False, **p)


def serving(seed=1, **kw):
    """Serving shape (K=50, as in the online deployment of Appendix B.3):
    B=256, C=256, d=128, 4 heads, 2 layers, M=100, L=6, Zipf(1.1) popularity."""
    p = dict(B=256, C=256, d=128, H=4, Ly=2, M=100, K=50, L=6)
    p.update(kw)
    d = p["d"]
    return _rec_workload("serving", seed, zipf_s=1.1, ctx_std=1 / np.sqrt(d),
                         pool_std=1 / np.sqrt(d), **p)


def ksweep(K, seed=2, **kw):
    """K sweep: B=64, C=256, d=128, 4 heads, 2 layers, M=200, L=10, uniform;
    the same context, pool and parameters for every K, sequences drawn per K."""
    p = dict(B=64, C=256, d=128, H=4, Ly=2, M=200, L=10)
    p.update(kw)
    d = p["d"]
    return _rec_workload(f"ksweep_K{K}", seed, K=K, zipf_s=None, ctx_std=1 / np.sqrt(d),
                         pool_std=1 / np.sqrt(d), idx_seed=[seed, K], **p)


def stress(seed=4, **kw):
    """Throughput stress: B=1024, C=512, d=256, 8 heads, 2 layers, M=500, K=200,
    L=10, Zipf(1.3) for heavy recurrence."""
    p = dict(B=1024, C=512, d=256, H=8, Ly=2, M=500, K=200, L=10)
    p.update(kw)
    d = p["d"]
    return _rec_workload("stress", seed, zipf_s=1.3, ctx_std=1 / np.sqrt(d),
                         pool_std=1 / np.sqrt(d), **p)


def summarisation(seed=3, B=32, C=1024, d=512, H=8, Ly=2, K=16, L=64, vocab=32768,
                  p_sub=0.3):
    """Summarisation-shaped rerank (CNN/DailyMail-like, Appendix B.1): each
    request has one base hypothesis of L uniform tokens; each of the K
    hypotheses copies it and replaces every position with probability p_sub by
    a uniform token.  The pool of a request is the embedding rows of its
    distinct hypothesis tokens in ascending token id, zero-padded to
    M = max_b U_b; the context is the embedding rows of C uniform source
    tokens.  Token embeddings ~ N(0, 0.02)."""
    cfg = ModelConfig(d=d, n_heads=H, n_layers=Ly, max_L=L, io_bf16=True)
    rng = np.random.default_rng(seed)
    weights = make_weights(cfg, rng)
    table = _normal(rng, (vocab, d), 0.02, True)
    hyps = np.empty((B, K, L), dtype=np.int64)
    for b in range(B):
        base = rng.integers(0, vocab, size=L)
        h = np.tile(base, (K, 1))
        sub = rng.random((K, L)) < p_sub
        h[sub] = rng.integers(0, vocab, size=int(sub.sum()))
        hyps[b] = h
    src = rng.integers(0, vocab, size=(B, C))
    context = table[src]
    toks = [np.unique(hyps[b]) for b in range(B)]
    M = max(len(t) for t in toks)
    pool = np.zeros((B, M, d), dtype=np.float32)
    cand = np.empty((B, K, L), dtype=np.int32)
    for b in range(B):
        pool[b, :len(toks[b])] = table[toks[b]]
        cand[b] = np.searchsorted(toks[b], hyps[b])
    return Workload("summarisation", cfg, np.ascontiguousarray(context), pool, cand, weights)


WORKLOADS = {
    "tiny": tiny,
    "serving": serving,
    "ksweep": ksweep,
    "summarisation": summarisation,
    "stress": stress,
}


def make_workload(name: str, **kw) -> Workload:
    return WORKLOADS[name](**kw)
