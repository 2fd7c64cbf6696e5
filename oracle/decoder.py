"""One decode step of a whole decoder layer, composed from the oracle's
primitives.  TEST INFRASTRUCTURE, like the rest of this package.

The paper's MLP block (Eq. 1 on gate/up, Sec. 3.3) sits inside a decoder
layer whose other operators Sec. 5 counts among those whose cost does not
depend on the weight precision.  In the W4/W2-GateUp configuration every
linear layer outside gate/up is INT4 (Sec. 7 step 4), so the attention
projections are 4-bit here.  The attention itself follows the dense models'
standard decode form.  Per sequence b, with one new token:
  1. xin = RMSNorm(x) (unit weight, eps 1e-6), unrounded;
  2. q, k, v = xin deq(Wq)^T, xin deq(Wk)^T, xin deq(Wv)^T (4-bit);
  3. q and k normalized per head (unit-weight RMSNorm over each head);
  4. RoPE at position len[b] on q and k;
  5. k, v rounded to bf16 and appended to the cache at position len[b];
  6. o = attention over positions 0..len[b] (grouped-query heads);
  7. o rounded to bf16 (stored between the attention and the projection);
  8. x1 = x + bf16(o) deq(Wo)^T, rounded to bf16;
  9. the MLP block on x1 (RMSNorm, 2-bit gate/up with the adapters, SiLU(g) u,
     4-bit down + residual), as in the oracle's gateup / down.
Every step is one oracle primitive or a plain numpy line.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

from . import (RMS_EPS, attn_decode, bf16_bits_to_f64, down, f64_to_bf16_bits, gateup, qproj, rms_scale,
               rope)


@dataclass
class AttnShape:
    n_heads: int
    n_kv: int
    head_dim: int
    theta: float = 1e6


def head_rms_norm(x, n_heads: int, hd: int, eps: float = RMS_EPS) -> np.ndarray:
    """Unit-weight RMSNorm over each head's hd values of x [m, n_heads * hd] (fp64)."""
    v = np.asarray(x, np.float64).reshape(-1, n_heads, hd)
    return (v / np.sqrt(np.mean(v * v, axis=2, keepdims=True) + eps)).reshape(-1, n_heads * hd)


def decoder_layer_decode(x_bits, lens, k_cache, v_cache, shape: AttnShape, wq, wk, wv, wo, group_attn: int,
                         gate, up, wd, group_gu: int, group_down: int, lora=None, lora_scale: float = 0.0):
    """Steps 1-9 above for x_bits [B, d] (bf16 bits).

    k_cache, v_cache: bf16 bits [B, n_kv, max_len, hd], not modified; lens[b]
    positions of sequence b are filled.  wq, wk, wv, wo, gate, up, wd: (q, s, z)
    tuples.  lora: (A_cat, B_gate, B_up) bf16 bits or None.
    Returns a dict with y (fp64 and bf16 bits), x1 bits, o bits and the new caches.
    """
    x_bits = np.ascontiguousarray(x_bits, np.uint16)
    b, d = x_bits.shape
    H, Hkv, hd = shape.n_heads, shape.n_kv, shape.head_dim
    lens = np.asarray(lens, np.int64)
    assert np.all(lens + 1 <= k_cache.shape[2])
    xin = bf16_bits_to_f64(x_bits) * rms_scale(x_bits)[:, None]                       # 1
    q = qproj(xin, wq, group_attn)                                                    # 2
    k = qproj(xin, wk, group_attn)
    v = qproj(xin, wv, group_attn)
    q = head_rms_norm(q, H, hd)                                                       # 3
    k = head_rms_norm(k, Hkv, hd)
    q = np.stack([rope(q[i].reshape(H, hd), int(lens[i]), shape.theta) for i in range(b)])       # 4
    k = np.stack([rope(k[i].reshape(Hkv, hd), int(lens[i]), shape.theta) for i in range(b)])
    kc, vc = np.array(k_cache, np.uint16, copy=True), np.array(v_cache, np.uint16, copy=True)   # 5
    for i in range(b):
        kc[i, :, lens[i]] = f64_to_bf16_bits(k[i])
        vc[i, :, lens[i]] = f64_to_bf16_bits(v[i].reshape(Hkv, hd))
    o = attn_decode(q, kc, vc, lens + 1)                                              # 6
    o_bits = f64_to_bf16_bits(o.reshape(b, H * hd))                                   # 7
    _, x1_bits = down(o_bits, wo, group_attn, x_bits)                                 # 8
    la, lbg, lbu = lora if lora is not None else (None, None, None)                   # 9
    _, h_bits = gateup(x1_bits, gate, up, group_gu, la, lbg, lbu, lora_scale=lora_scale, prenorm=True)
    y, y_bits = down(h_bits, wd, group_down, x1_bits)
    return {"y": y, "y_bits": y_bits, "x1_bits": x1_bits, "o_bits": o_bits, "k_cache": kc, "v_cache": vc}
