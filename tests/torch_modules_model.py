"""The evaluator assembled from stock torch.nn layers, used only to pin the oracle.

Each stage is a library module (nn.LayerNorm without affine parameters,
nn.MultiheadAttention without biases, nn.Linear), so head splitting, the
1/sqrt(d_h) scale, the softmax axis and the projection conventions come from
PyTorch rather than from the oracle's own code.  It scores the sequences
candidate by candidate for the element side (context K/V and element
encodings rebuilt for every sequence, the E^ind structure of Section 4), then
applies the cross-sequence block and head of Section 4.4.
"""
import numpy as np
import torch
import torch.nn as nn

DT = torch.float64


def _t(a):
    return torch.as_tensor(np.asarray(a, dtype=np.float64))


def _mha(d, H, WQ, WK, WV, WO):
    m = nn.MultiheadAttention(d, H, bias=False, batch_first=True, dtype=DT)
    with torch.no_grad():
        m.in_proj_weight.copy_(torch.cat([_t(WQ).T, _t(WK).T, _t(WV).T], 0))
        m.out_proj.weight.copy_(_t(WO).T)
    return m.eval()


def _linear(W, b):
    W = _t(W)
    lin = nn.Linear(W.shape[0], W.shape[1], bias=True, dtype=DT)
    with torch.no_grad():
        lin.weight.copy_(W.T)
        lin.bias.copy_(_t(b).reshape(-1))
    return lin.eval()


class TorchEvaluator:
    def __init__(self, W, cfg):
        d, H = cfg.d, cfg.n_heads
        self.cfg = cfg
        self.ln = nn.LayerNorm(d, eps=cfg.ln_eps, elementwise_affine=False, dtype=DT)
        self.layers = []
        for l in range(cfg.n_layers):
            attn = _mha(d, H, W[f"WQ.{l}"], W[f"WK.{l}"], W[f"WV.{l}"], W[f"WO.{l}"])
            ffn = nn.Sequential(_linear(W[f"W1.{l}"], W[f"b1.{l}"]), nn.ReLU(),
                                _linear(W[f"W2.{l}"], W[f"b2.{l}"]))
            self.layers.append((attn, ffn))
        self.cls = _t(W["cls"])
        self.P = _t(W["P"])
        self.seq_attn = _mha(d, H, W["WQs"], W["WKs"], W["WVs"], W["WOs"])
        self.seq_ffn = nn.Sequential(_linear(W["W1s"], W["b1s"]), nn.ReLU(),
                                     _linear(W["W2s"], W["b2s"]))
        self.x_attn = _mha(d, H, W["WQx"], W["WKx"], W["WVx"], W["WOx"])
        self.head = nn.Sequential(_linear(W["W1h"], W["b1h"]), nn.ReLU(),
                                  _linear(np.asarray(W["w2h"]).reshape(-1, 1), W["b2h"]))

    @torch.no_grad()
    def score_sequence_rep(self, context_b, pool_b, seq):
        """c_k of one sequence, rebuilding everything for it alone."""
        X = self.ln(_t(context_b))[None]                    # [1, C, d]
        h = _t(pool_b)[list(seq)][None]                     # [1, L, d]
        for attn, ffn in self.layers:
            h = h + attn(self.ln(h), X, X, need_weights=False)[0]
            h = h + ffn(self.ln(h))
        r = self.ln(h)[0]
        L = r.shape[0]
        x = torch.cat([self.cls[None], r + self.P[:L]], 0)[None]
        c = self.cls + self.seq_attn(x, x, x, need_weights=False)[0][0, 0]
        return c + self.seq_ffn(self.ln(c))

    @torch.no_grad()
    def scores(self, context_b, pool_b, cand_b):
        Cm = torch.stack([self.score_sequence_rep(context_b, pool_b, s) for s in cand_b])[None]
        Z = self.ln(Cm)
        Cp = Cm + self.x_attn(Z, Z, Z, need_weights=False)[0]
        return self.head(self.ln(Cp))[0, :, 0].numpy()

    def best(self, s):
        return int(torch.argmax(torch.as_tensor(s)))
