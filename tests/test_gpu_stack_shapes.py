"""The MLP stack at the benchmarked layer shapes vs the oracle.

Every layer's output and its MLP activation h come from
wq_mlp_forward_states, which runs the same launches as wq_mlp_forward (the
call the benchmark times) with each layer writing into slots of its own.
Each kernel is checked teacher-forced: the oracle's gate/up of layer l takes
the GPU's output of layer l-1, and the oracle's down takes the GPU's h of
layer l (a bf16 h element that rounds the other way from the oracle's moves
y by far more than the down kernel's own rounding at 9728 features).  The launch chain of
the Qwen3-4B-shaped stack is pinned to the plans the benchmark's headline
runs (gate/up 4 row tiles a CTA, 20 blocks a panel, 4 warps along k; down
one row tile a CTA over all 76 blocks; the binary16 panel of h handed from
gate/up to down), so that a planner change cannot move the headline onto an
untested configuration.
"""
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


_CACHE = {}


def _stack(wq, name, n_layers):
    """n_layers distinct layers of a named shape: oracle quantization, oracle
    packing, uploaded; the oracle's copies alongside."""
    key = (name, n_layers)
    if key in _CACHE:
        return _CACHE[key]
    cfg = synth.CONFIGS[name]
    layers, ents = [], []
    for l in range(n_layers):
        wg, wu, wd = synth.layer_weights(cfg, l)
        qg = orc.quantize(wg.numpy(), cfg.group_gu, 2)[:3]
        qu = orc.quantize(wu.numpy(), cfg.group_gu, 2)[:3]
        qd = orc.quantize(wd.numpy(), cfg.group_down, 4)[:3]
        a, bg, bu = synth.lora(cfg.d, cfg.inter, cfg.r, 10_000 + l)
        ents.append(dict(g=qg, u=qu, d=qd, a=synth.bf16_bits(a), bg=synth.bf16_bits(bg), bu=synth.bf16_bits(bu)))
        layers.append(wq.MLPLayer(upload_packed(*qg, cfg.group_gu, 2), upload_packed(*qu, cfg.group_gu, 2),
                                  upload_packed(*qd, cfg.group_down, 4), lora_a=a.cuda(), lora_b_gate=bg.cuda(),
                                  lora_b_up=bu.cuda(), lora_scale=cfg.lora_scale))
    _CACHE[key] = (cfg, layers, ents)
    return _CACHE[key]


def _teacher_forced(cfg, ents, x, states, h_states, what):
    """Each kernel of each layer against the oracle on the GPU's own inputs:
    gate/up on the layer's input x, down on the GPU's h and x."""
    prev = synth.bf16_bits(x.cpu())
    for l, ent in enumerate(ents):
        h_ref, _ = orc.gateup(prev, ent["g"], ent["u"], cfg.group_gu, ent["a"], ent["bg"], ent["bu"],
                              lora_scale=cfg.lora_scale, prenorm=True)
        check_bf16(h_states[l], h_ref, f"{what} layer {l} h (teacher-forced)")
        y_ref, _ = orc.down(synth.bf16_bits(h_states[l].cpu()), ent["d"], cfg.group_down, prev)
        check_bf16(states[l], y_ref, f"{what} layer {l} y (teacher-forced)")
        prev = synth.bf16_bits(states[l].cpu())


def test_qwen3_4b_chain_runs_the_headline_plans(wq):
    cfg, layers, _ = _stack(wq, "qwen3_4b", 3)
    info = wq.mlp_forward_info(1, layers, prenorm=True, chain=True)
    assert info["route"] == wq.ROUTE_GEMV_CHAIN
    assert info["gateup"] == dict(rb=4, kp=20, wk=4, tpw=1, panels=1, ctas=152), info
    assert info["down"] == dict(rb=1, kp=76, wk=8, tpw=1, panels=1, ctas=160), info
    assert info["panel"], "the gate/up launch no longer hands the down launch its binary16 panel"


@pytest.mark.parametrize("m", [1, 2, 4, 8, 16])
def test_qwen3_4b_chain_teacher_forced(wq, m):
    cfg, layers, ents = _stack(wq, "qwen3_4b", 3)
    info = wq.mlp_forward_info(m, layers, prenorm=True, chain=True)
    assert info["route"] == wq.ROUTE_GEMV_CHAIN, info
    x = synth.activations((m, cfg.d), 2024 + m).cuda()
    ws = wq.workspace(m, cfg.d, cfg.inter, cfg.r)
    y, states, h_states = wq.mlp_forward_states(x, layers, prenorm=True, ws=ws, chain=True, with_h=True)
    y_plain = wq.mlp_forward(x, layers, prenorm=True, ws=ws, chain=True)
    torch.cuda.synchronize()
    assert wq.device_status() == 0
    # the states run and the plain run are the same launches
    assert torch.equal(y.view(torch.int16), y_plain.view(torch.int16))
    assert torch.equal(states[-1].view(torch.int16), y.view(torch.int16))
    _teacher_forced(cfg, ents, x, states, h_states, f"qwen3_4b chain m={m} (panel={info['panel']})")


def test_dense_14b_prefill_layer(wq):
    """One 14B-shaped layer at 512 tokens (the prefill leg's shape) through the
    tcgen05 dequant-GEMM chain: h and y on a sample of tokens spread over the
    four 128-token tiles against the oracle, each kernel teacher-forced (the
    bf16 bound; the GEMM path's share of bit-exact elements)."""
    cfg, layers, ents = _stack(wq, "dense_14b", 1)
    m = 512
    info = wq.mlp_forward_info(m, layers, prenorm=True)
    assert info["route"] == wq.ROUTE_GEMM_CHAIN
    x = synth.activations((m, cfg.d), 77).cuda()
    ws = wq.workspace(m, cfg.d, cfg.inter, cfg.r)
    y, _, h_states = wq.mlp_forward_states(x, layers, prenorm=True, ws=ws, with_h=True)
    torch.cuda.synchronize()
    assert wq.device_status() == 0
    rows = np.array([0, 1, 127, 128, 200, 255, 256, 383, 384, 511])
    idx = torch.from_numpy(rows).cuda()
    ent = ents[0]
    xb = synth.bf16_bits(x.cpu())[rows]
    h_ref, _ = orc.gateup(xb, ent["g"], ent["u"], cfg.group_gu, ent["a"], ent["bg"], ent["bu"],
                          lora_scale=cfg.lora_scale, prenorm=True)
    check_bf16(h_states[0][idx], h_ref, "dense_14b m=512 h, sampled tokens", min_exact=0.6)
    y_ref, _ = orc.down(synth.bf16_bits(h_states[0][idx].cpu()), ent["d"], cfg.group_down, xb)
    check_bf16(y[idx], y_ref, "dense_14b m=512 y, sampled tokens", min_exact=0.6)
