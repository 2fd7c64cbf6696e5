"""One mixture-of-experts MLP block, composed from the oracle's primitives.
TEST INFRASTRUCTURE, like the rest of this package.

Sec. 5 analyses an MoE model whose routing activates only a subset of the
experts per token, so only the active experts' weights are read.  Here each
expert is the paper's gated MLP: 2-bit gate/up with optional adapters, SiLU(g) u,
4-bit down.  Per token t:
  1. the router logits of t (an input) select the top-k experts, the larger
     logit first and the lower expert index first among equal logits;
  2. the routing weights are the softmax of the selected logits;
  3. each selected expert e computes h_e = SiLU(g_e) u_e on RMSNorm(x)
     (stored as bf16, as the dense block stores h) and y_e = h_e deq(Wd_e)^T
     in fp64;
  4. y = x + sum_j w_j y_{e_j}, rounded to bf16 once.
"""
from __future__ import annotations

import numpy as np

from . import bf16_bits_to_f64, down, f64_to_bf16_bits, gateup


def route(logits, k: int):
    """(expert indices [T, k], weights [T, k]) from router logits [T, E]."""
    lg = np.asarray(logits, np.float64)
    t, e = lg.shape
    assert 1 <= k <= e
    idx = np.empty((t, k), np.int64)
    for i in range(t):
        order = sorted(range(e), key=lambda j: (-lg[i, j], j))
        idx[i] = order[:k]
    sel = np.take_along_axis(lg, idx, axis=1)
    w = np.exp(sel - sel.max(axis=1, keepdims=True))
    return idx, w / w.sum(axis=1, keepdims=True)


def moe_block(x_bits, logits, k: int, experts, group_gu: int, group_down: int, lora_scale: float = 0.0):
    """Steps 1-4 for x_bits [T, d] (bf16 bits).  experts: list of dicts with
    keys gate, up, down ((q, s, z) tuples) and optionally lora (A_cat, B_gate,
    B_up as bf16 bits).  Returns (y fp64 [T, d], y bf16 bits, expert indices, weights)."""
    x_bits = np.ascontiguousarray(x_bits, np.uint16)
    idx, w = route(logits, k)
    y = bf16_bits_to_f64(x_bits).copy()
    for t in range(x_bits.shape[0]):
        xt = x_bits[t:t + 1]
        for j in range(k):
            ex = experts[int(idx[t, j])]
            la, lbg, lbu = ex.get("lora") or (None, None, None)
            _, h_bits = gateup(xt, ex["gate"], ex["up"], group_gu, la, lbg, lbu, lora_scale=lora_scale,
                               prenorm=True)
            ye, _ = down(h_bits, ex["down"], group_down, None)
            y[t] += w[t, j] * ye[0]
    return y, f64_to_bf16_bits(y), idx, w
