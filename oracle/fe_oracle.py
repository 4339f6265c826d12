"""CPU oracle for FlashEvaluator joint evaluation (test infrastructure only).

This is a plain, slow restatement in float64 numpy of what the evaluator of
Section 4 computes.  It exists to check the CUDA path: only the test suite,
the smoke check and the benchmark's CPU-baseline leg may import it, and it
shares no code with the CUDA path.

Model, in the paper's order (Section 4.1: H = Enc(x, U(z)) -> c = Idx(H, L) ->
s = Inter(c), then Eq. 1's argmax):

* Query Context Module (Section 4.2): X = LN(context); per layer l the
  context keys/values K_l = X W_K^l, V_l = X W_V^l, computed once per request
  (the K/V half of the QKV-Cache).
* Distinct-element encoding (Section 4.2): for each element of
  U(z) = union of the K sequences (Section 4.1), h = pool row; per layer
  h += MHA(LN(h) W_Q^l, K_l, V_l) W_O^l;  h += FFN^l(LN(h)); output LN(h).
  Each distinct element is encoded once (the Q-Cache).
* Index-based assembly (Section 4.3): x_0 = [CLS], x_j = H[i_{k,j}] + P[j-1];
  one CLS-pooled SeqEnc block gives c_k.
* Cross-sequence interaction (Section 4.4): C' = C + MHA(LN(C)W_Qx,
  LN(C)W_Kx, LN(C)W_Vx) W_Ox over the K sequences; score head
  s_k = ReLU(LN(C'_k) W1h + b1h) . w2h + b2h.
* Selection (Eq. 1): the smallest k attaining max_k s_k (the smallest-index
  rule the paper uses for its listwise labels, Appendix B.1).
* Multi-objective variant (end of Section 4.4): T task-specific heads of the
  same shape read the shared C'_k, and a fusion module combines their scores.
  The paper does not define the fusion module; the reading taken here is a
  learned linear combination s_k = sum_t alpha_t s_{k,t} + beta.
* Variant without cross-sequence interaction ("- CrossSeq", ablation of
  Appendix B.4): C' = C, each sequence scored on its own representation.
* Element self-attention H^(1) (Section 4.2), optional: before the
  cross-attention stack, h += MHA(LN(h) W_Qe, LN(h) W_Ke, LN(h) W_Ve) W_Oe
  over the request's element set (a pre-LN block with residual, like the
  cross-sequence block).  The element set is U(z), or with encode_pool the
  whole pool (U(z) = C(x), U = M, Section 4.1).
* Linear-attention context module, optional (the online deployment of
  Appendix B.3 uses linear attention for its 1,000-interaction contexts):
  the element -> context cross-attention becomes kernelized attention with
  the feature map phi(x) = elu(x) + 1 of Katharopoulos et al. (2020), non-causal
  over the context; per request, layer and head the context reduces to the
  state S = phi(K)^T V and z = sum_c phi(K_c), and an element query reads
  phi(q) S / (phi(q) . z).

The paper leaves the block internals open (norm placement, FFN, pooling, head
shape).  The readings taken here: pre-LN blocks with LayerNorm without affine
parameters, eps 1e-5, biased variance; FFN width 4d with ReLU; projections
without bias, FFN and head with bias; attention scale 1/sqrt(d_h) with heads
as contiguous column blocks; no position embedding on [CLS]; no masking.

`evaluate(..., mode="no_reuse")` recomputes the context K/V for every sequence
and every element occurrence independently (the candidate-factorized cost
structure of Appendix A.3); `mode="reuse"` computes them once per request and
once per distinct element.  Both must give the same numbers.

Requests whose candidate indices fall outside [0, M) get NaN scores and best
index -1 (the boundary's per-request error behaviour).
"""
from __future__ import annotations

import numpy as np

__all__ = ["layer_norm", "softmax", "mha", "elu_feature", "linear_attention", "context_kv", "elem_self_attention", "encode_elements",
           "seq_encode", "cross_sequence", "score_head", "task_heads", "select_best",
           "distinct_layout", "element_set", "evaluate_request", "evaluate"]


# -- building blocks --------------------------------------------------------

def layer_norm(x, eps=1e-5):
    """Per-row LayerNorm without affine parameters: (x - mean) / sqrt(var + eps),
    var the biased variance over the last axis."""
    x = np.asarray(x, dtype=np.float64)
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps)


def softmax(z):
    """Softmax over the last axis, with the row maximum subtracted first."""
    z = np.asarray(z, dtype=np.float64)
    e = np.exp(z - z.max(axis=-1, keepdims=True))
    return e / e.sum(axis=-1, keepdims=True)


def mha(q, k, v, n_heads):
    """Multi-head scaled dot-product attention of query rows q [n, d] over key
    rows k [m, d] with values v [m, d].  Head h uses columns
    [h*d_h, (h+1)*d_h), d_h = d / n_heads; weights softmax(q_h k_h^T / sqrt(d_h))."""
    n, d = q.shape
    dh = d // n_heads
    out = np.empty((n, d), dtype=np.float64)
    for h in range(n_heads):
        cols = slice(h * dh, (h + 1) * dh)
        w = softmax(q[:, cols] @ k[:, cols].T / np.sqrt(dh))
        out[:, cols] = w @ v[:, cols]
    return out


def elu_feature(x):
    """phi(x) = elu(x) + 1: x + 1 for x > 0, exp(x) otherwise (positive everywhere)."""
    x = np.asarray(x, dtype=np.float64)
    return np.where(x > 0, x + 1.0, np.exp(np.minimum(x, 0.0)))


def linear_attention(q, k, v, n_heads):
    """Kernelized (linear) attention of query rows q [n, d] over key rows k
    [m, d] with values v [m, d], heads as contiguous column blocks: per head,
    out = phi(q) S / (phi(q) . z) with the context state S = phi(k)^T v
    [d_h, d_h] and z = sum over the keys of phi(k) [d_h]."""
    n, d = q.shape
    dh = d // n_heads
    out = np.empty((n, d), dtype=np.float64)
    for h in range(n_heads):
        cols = slice(h * dh, (h + 1) * dh)
        fk = elu_feature(k[:, cols])
        S = fk.T @ np.asarray(v[:, cols], dtype=np.float64)
        z = fk.sum(axis=0)
        fq = elu_feature(q[:, cols])
        out[:, cols] = (fq @ S) / (fq @ z)[:, None]
    return out


def _relu(x):
    return np.maximum(x, 0.0)


def _w(W, name):
    return np.asarray(W[name], dtype=np.float64)


# -- Section 4.2: request context and distinct elements ----------------------

def context_kv(context_b, W, n_layers, eps):
    """Query Context Module: per-layer context keys and values of one request,
    [(K_1, V_1), ..., (K_Ly, V_Ly)], each [C, d]."""
    X = layer_norm(context_b, eps)
    return [(X @ _w(W, f"WK.{l}"), X @ _w(W, f"WV.{l}")) for l in range(n_layers)]


def elem_self_attention(h, W, n_heads, eps):
    """H^(1) of Section 4.2 over the rows of h, one request's element set:
    h + MHA(Z W_Qe, Z W_Ke, Z W_Ve) W_Oe with Z = LN(h), every element
    attending to every element of the set."""
    h = np.asarray(h, dtype=np.float64)
    Z = layer_norm(h, eps)
    return h + mha(Z @ _w(W, "WQe"), Z @ _w(W, "WKe"), Z @ _w(W, "WVe"), n_heads) @ _w(W, "WOe")


def encode_elements(h0, kv, W, n_heads, eps, linear=False):
    """Request-conditioned representation of each element row of h0 [n, d]:
    the cross-attention stack over the context K/V (softmax attention, or
    linear attention when `linear`), then a final LN."""
    h = np.array(h0, dtype=np.float64)
    attend = linear_attention if linear else mha
    for l, (Kl, Vl) in enumerate(kv):
        q = layer_norm(h, eps) @ _w(W, f"WQ.{l}")
        h = h + attend(q, Kl, Vl, n_heads) @ _w(W, f"WO.{l}")
        f = _relu(layer_norm(h, eps) @ _w(W, f"W1.{l}") + _w(W, f"b1.{l}"))
        h = h + f @ _w(W, f"W2.{l}") + _w(W, f"b2.{l}")
    return layer_norm(h, eps)


# -- Section 4.3: index-based assembly and intra-sequence aggregation --------

def seq_encode(elem_rows, W, n_heads, eps):
    """c_k for one sequence whose element representations are elem_rows [L, d]:
    tokens [CLS; rows + P[0..L-1]], one attention block whose output is the
    [CLS] row, residual on [CLS], then a pre-LN FFN with residual."""
    L = elem_rows.shape[0]
    cls = _w(W, "cls")
    x = np.vstack([cls[None, :], elem_rows + _w(W, "P")[:L]])
    o = mha(x @ _w(W, "WQs"), x @ _w(W, "WKs"), x @ _w(W, "WVs"), n_heads)[0]
    c = cls + o @ _w(W, "WOs")
    f = _relu(layer_norm(c, eps) @ _w(W, "W1s") + _w(W, "b1s"))
    return c + f @ _w(W, "W2s") + _w(W, "b2s")


# -- Section 4.4: cross-sequence interaction and score head ------------------

def cross_sequence(Cm, W, n_heads, eps):
    """C' = C + MHA(Z W_Qx, Z W_Kx, Z W_Vx) W_Ox with Z = LN(C), over the K rows."""
    Z = layer_norm(Cm, eps)
    a = mha(Z @ _w(W, "WQx"), Z @ _w(W, "WKx"), Z @ _w(W, "WVx"), n_heads)
    return Cm + a @ _w(W, "WOx")


def score_head(Cp, W, eps, suffix=""):
    """Shared prediction head s_k = ReLU(LN(C'_k) W1h + b1h) . w2h + b2h
    (the head's tensors named W1h, b1h, w2h, b2h followed by `suffix`)."""
    f = _relu(layer_norm(Cp, eps) @ _w(W, "W1h" + suffix) + _w(W, "b1h" + suffix))
    return f @ _w(W, "w2h" + suffix) + _w(W, "b2h" + suffix)[0]


def task_heads(Cp, W, n_tasks, eps):
    """Multi-objective heads (end of Section 4.4): task t's head, of the same
    shape as the single head, with tensors W1h.t, b1h.t, w2h.t, b2h.t, then the
    fusion s_k = sum_t fuse_w[t] s_{k,t} + fuse_b.  Returns (s [K], per-task
    scores [K, T])."""
    st = np.stack([score_head(Cp, W, eps, f".{t}") for t in range(n_tasks)], axis=1)
    return st @ _w(W, "fuse_w") + _w(W, "fuse_b")[0], st


def select_best(s):
    """Eq. 1 argmax over k, ties resolved to the smallest index; -1 when any
    score is NaN."""
    s = np.asarray(s, dtype=np.float64)
    if s.size == 0 or np.isnan(s).any():
        return -1
    return int(np.flatnonzero(s == s.max())[0])


def distinct_layout(cand_b):
    """U(z) of one request (Section 4.1) as the ascending list of distinct pool
    rows, and slot[k, j] = position of cand_b[k, j] in that list."""
    cand_b = np.asarray(cand_b)
    uniq = np.unique(cand_b)
    slots = np.searchsorted(uniq, cand_b).astype(np.int32)
    return uniq.astype(np.int32), slots


def element_set(cand_b, M, cfg):
    """The element set a request encodes and every occurrence's slot in it:
    U(z) (distinct_layout), or with cfg.encode_pool the whole pool
    (U(z) = C(x), Section 4.1): rows 0..M-1, slot = the pool index."""
    if getattr(cfg, "encode_pool", False):
        return np.arange(M, dtype=np.int32), np.asarray(cand_b, dtype=np.int32).copy()
    return distinct_layout(cand_b)


# -- whole evaluator ---------------------------------------------------------

def evaluate_request(context_b, pool_b, cand_b, W, cfg, mode="reuse", tasks_out=None):
    """Scores [K] of one request's K candidate sequences.  With several task
    heads the scores are the fused ones and, when tasks_out is a list, the
    per-task scores [K, T] are appended to it."""
    H, Ly, eps = cfg.n_heads, cfg.n_layers, cfg.ln_eps
    K, L = cand_b.shape
    pool_b = np.asarray(pool_b, np.float64)
    uniq, slots = element_set(cand_b, pool_b.shape[0], cfg)
    self_attn = getattr(cfg, "elem_self_attn", False)
    lin = getattr(cfg, "linear_context_attn", False)
    if mode == "reuse":
        kv = context_kv(context_b, W, Ly, eps)
        h0 = pool_b[uniq]
        if self_attn:
            h0 = elem_self_attention(h0, W, H, eps)
        Henc = encode_elements(h0, kv, W, H, eps, linear=lin)
        rows = [Henc[slots[k]] for k in range(K)]
    elif mode == "no_reuse":
        rows = []
        for k in range(K):
            kv = context_kv(context_b, W, Ly, eps)          # per sequence
            r = []
            for j, m in enumerate(cand_b[k]):               # per occurrence
                if self_attn:                               # H^(1) over the set, recomputed
                    h0 = elem_self_attention(pool_b[uniq], W, H, eps)[[slots[k, j]]]
                else:
                    h0 = pool_b[[m]]
                r.append(encode_elements(h0, kv, W, H, eps, linear=lin))
            rows.append(np.vstack(r))
    else:
        raise ValueError(mode)
    Cm = np.vstack([seq_encode(rows[k], W, H, eps) for k in range(K)])
    Cp = cross_sequence(Cm, W, H, eps) if getattr(cfg, "cross_seq", True) else Cm
    T = int(getattr(cfg, "n_tasks", 1))
    if T == 1:
        s = score_head(Cp, W, eps)
        if tasks_out is not None:
            tasks_out.append(s[:, None])
        return s
    s, st = task_heads(Cp, W, T, eps)
    if tasks_out is not None:
        tasks_out.append(st)
    return s


def evaluate(context, pool, cand_idx, W, cfg, mode="reuse", requests=None, with_tasks=False):
    """E_theta over a batch.  Returns (scores [B, K] float64, best [B] int32,
    U [B] int32, slots [B, K, L] int32), plus the per-task scores [B, K, T]
    when with_tasks.  `requests` restricts the work to a subset of request
    indices (the other rows stay NaN / -1)."""
    context = np.asarray(context)
    pool = np.asarray(pool)
    cand_idx = np.asarray(cand_idx)
    B, K, L = cand_idx.shape
    M = pool.shape[1]
    scores = np.full((B, K), np.nan)
    best = np.full(B, -1, dtype=np.int32)
    U = np.zeros(B, dtype=np.int32)
    slots = np.full((B, K, L), -1, dtype=np.int32)
    T = int(getattr(cfg, "n_tasks", 1))
    tasks = np.full((B, K, T), np.nan)
    for b in (range(B) if requests is None else requests):
        cb = cand_idx[b]
        if cb.size and (cb.min() < 0 or cb.max() >= M):
            continue
        uniq, sl = element_set(cb, M, cfg)
        U[b] = len(uniq)
        slots[b] = sl
        if K == 0:
            continue
        out = []
        scores[b] = evaluate_request(context[b], pool[b], cb, W, cfg, mode, tasks_out=out)
        tasks[b] = out[0]
        best[b] = select_best(scores[b])
    if with_tasks:
        return scores, best, U, slots, tasks
    return scores, best, U, slots
