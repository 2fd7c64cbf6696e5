"""Seeded synthetic inputs shared by the CUDA path, the tests and the bench.

This module only draws random numbers and names workload shapes; it holds none
of the method's arithmetic (no quantization, no matmul, no activation).  The
recipe follows the workloads the paper analyses (Sec. 5.1: Qwen3-4B /
Qwen3-14B-class dense gated MLPs), with the real weights replaced by draws:

  * weights   W ~ N(0, 0.02) in fp32, before quantization;
  * activations x ~ N(0, 1), rounded to bf16;
  * LoRA      A, B ~ N(0, 0.01), rounded to bf16 (the paper's standard
              initialisation sets B = 0, which would make the adapter term
              vanish, so both factors are drawn);
  * layer l of a stack uses seed ``base + l``.
"""
from __future__ import annotations

from dataclasses import dataclass

import torch


@dataclass(frozen=True)
class MLPConfig:
    name: str
    d: int            # hidden size (input of gate/up, output of down)
    inter: int        # intermediate size (output of gate/up, input of down)
    group_gu: int     # group size of the gate/up codes
    group_down: int   # group size of the down codes
    r: int            # LoRA rank on gate and up
    layers: int       # depth of the stack
    lora_alpha: float  # LoRA alpha; the adapter term is scaled by alpha / r

    @property
    def lora_scale(self) -> float:
        return self.lora_alpha / self.r if self.r else 0.0


# Shapes of the paper's dense models (Qwen3-4B, an 8B-class and the 14B-class
# model), plus a small single-layer case.  alpha = 2r as in the paper's
# hyper-parameter table (r = 32, alpha = 64).
CONFIGS = {
    "small_d256_i768": MLPConfig("small_d256_i768", 256, 768, 64, 64, 8, 1, 16.0),
    "qwen3_4b": MLPConfig("qwen3_4b", 2560, 9728, 128, 128, 16, 36, 32.0),
    "dense_8b": MLPConfig("dense_8b", 4096, 14336, 128, 128, 32, 32, 64.0),
    "dense_14b": MLPConfig("dense_14b", 5120, 17408, 128, 128, 32, 40, 64.0),
}


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def weights(shape, seed: int, std: float = 0.02, device="cpu") -> torch.Tensor:
    """fp32 weights ~ N(0, std)."""
    g = _gen(seed, device)
    return torch.randn(tuple(shape), generator=g, device=device, dtype=torch.float32) * std


def activations(shape, seed: int, device="cpu") -> torch.Tensor:
    """bf16 activations ~ N(0, 1)."""
    g = _gen(seed, device)
    return torch.randn(tuple(shape), generator=g, device=device, dtype=torch.float32).to(torch.bfloat16)


def lora(d: int, inter: int, r: int, seed: int, std: float = 0.01, device="cpu"):
    """(A_cat [2r, d], B_gate [inter, r], B_up [inter, r]) in bf16, all ~ N(0, std).

    Rows 0..r-1 of A_cat are A_gate, rows r..2r-1 are A_up.
    """
    g = _gen(seed, device)
    a = torch.randn((2 * r, d), generator=g, device=device) * std
    bg = torch.randn((inter, r), generator=g, device=device) * std
    bu = torch.randn((inter, r), generator=g, device=device) * std
    return a.to(torch.bfloat16), bg.to(torch.bfloat16), bu.to(torch.bfloat16)


def layer_weights(cfg: MLPConfig, seed: int, device="cpu"):
    """fp32 (W_gate [inter, d], W_up [inter, d], W_down [d, inter]) of one layer."""
    wg = weights((cfg.inter, cfg.d), seed * 3 + 0, device=device)
    wu = weights((cfg.inter, cfg.d), seed * 3 + 1, device=device)
    wd = weights((cfg.d, cfg.inter), seed * 3 + 2, device=device)
    return wg, wu, wd


def bf16_bits(t: torch.Tensor):
    """bf16 tensor -> numpy uint16 bit patterns (CPU copy)."""
    return t.detach().to("cpu").contiguous().view(torch.int16).numpy().view("uint16")


def from_bf16_bits(a, device="cpu") -> torch.Tensor:
    """numpy uint16 bit patterns -> bf16 tensor."""
    import numpy as np
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.uint16).view(np.int16)).view(torch.bfloat16).to(device)
