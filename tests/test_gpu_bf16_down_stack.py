"""The BF16/W2-GateUp configuration (Sec. 6.1: gate/up at INT2, the down
projection in BF16) as a stack through wq_mlp_forward: 2-bit gate/up with the
adapters, the dense bf16 down, the residual stream in bf16.  Each layer is
checked teacher-forced against the oracle (gate/up on the GPU's input, the
bf16 down on the GPU's h), on the launch chain and on the GEMM chain, and a
stack that mixes 4-bit and bf16 down layers."""
import numpy as np
import pytest
import torch

import oracle as orc
from paper_2606_04238_gb300 import synth
from tests.gpu_util import check_bf16, upload_packed

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def wq():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2606_04238_gb300 import wq as mod
    return mod


def _stack(wq, d, inter, group, r, n, dense_mask, seed):
    layers, ents = [], []
    for l in range(n):
        wg = synth.weights((inter, d), seed + 3 * l)
        wu = synth.weights((inter, d), seed + 3 * l + 1)
        wd = synth.weights((d, inter), seed + 3 * l + 2)
        qg, qu = orc.quantize(wg.numpy(), group, 2)[:3], orc.quantize(wu.numpy(), group, 2)[:3]
        a, bg, bu = synth.lora(d, inter, r, seed + 100 + l)
        ent = dict(g=qg, u=qu, a=synth.bf16_bits(a), bg=synth.bf16_bits(bg), bu=synth.bf16_bits(bu))
        if dense_mask[l]:
            wdb = wd.to(torch.bfloat16)
            ent["wd_bf16"] = synth.bf16_bits(wdb)
            down = wq.dense_weight(wdb.cuda())
        else:
            qd = orc.quantize(wd.numpy(), group, 4)[:3]
            ent["wd_q"] = qd
            down = upload_packed(*qd, group, 4)
        layers.append(wq.MLPLayer(upload_packed(*qg, group, 2), upload_packed(*qu, group, 2), down, lora_a=a.cuda(),
                                  lora_b_gate=bg.cuda(), lora_b_up=bu.cuda(), lora_scale=2.0))
        ents.append(ent)
    return layers, ents


def _check(wq, layers, ents, group, m, d, what):
    x = synth.activations((m, d), 7 + m).cuda()
    _, states, h_states = wq.mlp_forward_states(x, layers, prenorm=True, with_h=True)
    torch.cuda.synchronize()
    assert wq.device_status() == 0
    exact = 0.97 if wq.mlp_forward_info(m, layers)["route"] != wq.ROUTE_GEMM_CHAIN else 0.6
    prev = synth.bf16_bits(x.cpu())
    for l, ent in enumerate(ents):
        h_ref, _ = orc.gateup(prev, ent["g"], ent["u"], group, ent["a"], ent["bg"], ent["bu"], lora_scale=2.0, prenorm=True)
        check_bf16(h_states[l], h_ref, f"{what} layer {l} h", min_exact=exact)
        hb = synth.bf16_bits(h_states[l].cpu())
        if "wd_bf16" in ent:
            y_ref, _ = orc.down_bf16(hb, ent["wd_bf16"], prev)
        else:
            y_ref, _ = orc.down(hb, ent["wd_q"], group, prev)
        check_bf16(states[l], y_ref, f"{what} layer {l} y", min_exact=exact)
        prev = synth.bf16_bits(states[l].cpu())


@pytest.mark.parametrize("m", [1, 4, 16, 65])
def test_bf16_down_stack(wq, m):
    layers, ents = _stack(wq, 256, 768, 64, 8, 3, [True, True, True], 11)
    _check(wq, layers, ents, 64, m, 256, f"bf16 down m={m}")


def test_mixed_down_stack(wq):
    layers, ents = _stack(wq, 256, 768, 64, 8, 4, [False, True, False, True], 21)
    for m in (1, 5):
        _check(wq, layers, ents, 64, m, 256, f"mixed m={m}")


def test_qwen3_4b_bf16_down_stack(wq):
    cfg = synth.CONFIGS["qwen3_4b"]
    layers, ents = _stack(wq, cfg.d, cfg.inter, 128, 16, 2, [True, True], 31)
    info = wq.mlp_forward_info(1, layers)
    assert info["route"] == wq.ROUTE_GEMV_CHAIN and info["down"]["rb"] == -1
    _check(wq, layers, ents, 128, 1, cfg.d, "qwen3_4b bf16 down")
