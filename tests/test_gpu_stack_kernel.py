"""The single-launch stack kernel (wq_mlp_forward's route for 1..8 tokens)
against the oracle.

Each layer's h and y come from wq_mlp_forward_states and are checked
teacher-forced, kernel phase by kernel phase: the oracle's gate/up takes the
GPU's input of the layer, the oracle's down the GPU's h.  Shapes cover the
Qwen3-4B layer (every CTA's down slice is its own h), the 14B layer and a
small layer (the down slices need other CTAs' h: the extra barrier), 4-bit
gate/up (the uniform-W4 comparator), groups 32/64/128, no adapter, no
RMSNorm, and a stack longer than one launch carries.
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


def _layers(wq, d, inter, group, r, n, bits_gu=2, seed=0):
    layers, ents = [], []
    for l in range(n):
        wg = synth.weights((inter, d), 1000 * seed + 3 * l)
        wu = synth.weights((inter, d), 1000 * seed + 3 * l + 1)
        wd = synth.weights((d, inter), 1000 * seed + 3 * l + 2)
        qg = orc.quantize(wg.numpy(), group, bits_gu)[:3]
        qu = orc.quantize(wu.numpy(), group, bits_gu)[:3]
        qd = orc.quantize(wd.numpy(), group, 4)[:3]
        ent = dict(g=qg, u=qu, d=qd, r=r)
        kw = {}
        if r:
            a, bg, bu = synth.lora(d, inter, r, 7000 + l + 100 * seed)
            ent.update(a=synth.bf16_bits(a), bg=synth.bf16_bits(bg), bu=synth.bf16_bits(bu))
            kw = dict(lora_a=a.cuda(), lora_b_gate=bg.cuda(), lora_b_up=bu.cuda(), lora_scale=2.0)
        layers.append(wq.MLPLayer(upload_packed(*qg, group, bits_gu), upload_packed(*qu, group, bits_gu),
                                  upload_packed(*qd, group, 4), **kw))
        ents.append(ent)
    return layers, ents


def _check(wq, layers, ents, group, m, prenorm, what, x_seed=5):
    d = layers[0].gate.k
    inter = layers[0].gate.n
    info = wq.mlp_forward_info(m, layers, prenorm=prenorm, stack=True)
    assert info["route"] == wq.ROUTE_STACK, info
    x = synth.activations((m, d), x_seed).cuda()
    ws = wq.workspace(m, d, inter, layers[0].r)
    y, states, h_states = wq.mlp_forward_states(x, layers, prenorm=prenorm, ws=ws, with_h=True, stack=True)
    y2 = wq.mlp_forward(x, layers, prenorm=prenorm, ws=ws, stack=True)
    torch.cuda.synchronize()
    assert wq.device_status() == 0
    assert torch.equal(y.view(torch.int16), y2.view(torch.int16)), "two runs differ"
    assert torch.equal(states[-1].view(torch.int16), y.view(torch.int16))
    prev = synth.bf16_bits(x.cpu())
    for l, ent in enumerate(ents):
        kw = {}
        if ent["r"]:
            kw = dict(lora_a=ent["a"], lora_b_gate=ent["bg"], lora_b_up=ent["bu"], lora_scale=2.0)
        h_ref, _ = orc.gateup(prev, ent["g"], ent["u"], group, kw.get("lora_a"), kw.get("lora_b_gate"),
                              kw.get("lora_b_up"), lora_scale=kw.get("lora_scale", 0.0), prenorm=prenorm)
        check_bf16(h_states[l], h_ref, f"{what} layer {l} h")
        y_ref, _ = orc.down(synth.bf16_bits(h_states[l].cpu()), ent["d"], group, prev)
        check_bf16(states[l], y_ref, f"{what} layer {l} y")
        prev = synth.bf16_bits(states[l].cpu())
    return info


@pytest.mark.parametrize("m", [1, 2, 3, 8])
def test_qwen3_4b_stack_kernel(wq, m):
    cfg = synth.CONFIGS["qwen3_4b"]
    layers, ents = _layers(wq, cfg.d, cfg.inter, 128, 16, 3)
    info = _check(wq, layers, ents, 128, m, True, f"qwen3_4b m={m}")
    assert info["stack"]["h_barrier"] == 0, info  # each CTA's down slice is its own h


def test_dense_14b_stack_kernel(wq):
    cfg = synth.CONFIGS["dense_14b"]
    layers, ents = _layers(wq, cfg.d, cfg.inter, 128, 32, 2, seed=1)
    info = _check(wq, layers, ents, 128, 1, True, "dense_14b m=1")
    assert info["stack"]["h_barrier"] == 1, info


@pytest.mark.parametrize("group,r,prenorm,bits", [(64, 8, True, 2), (32, 16, True, 2), (64, 0, False, 2),
                                                  (128, 0, True, 4), (32, 0, True, 4)])
def test_small_stack_kernel(wq, group, r, prenorm, bits):
    layers, ents = _layers(wq, 256, 768, group, r, 4, bits_gu=bits, seed=2)
    _check(wq, layers, ents, group, 4, prenorm, f"small g{group} r{r} bits{bits}")


def test_mid_stack_kernel_every_group(wq):
    # 2432 = 152 row tiles of 16: one gate/up tile a CTA, down slices shared by 4 CTAs
    for group in (32, 64, 128):
        layers, ents = _layers(wq, 1024, 2432, group, 8, 2, seed=3 + group)
        _check(wq, layers, ents, group, 5, True, f"mid g{group}")


def test_stack_longer_than_one_launch(wq):
    # 70 layers: two launches (64 + 6), the second starting from the first's output
    layers, ents = _layers(wq, 256, 768, 64, 8, 70, seed=9)
    _check(wq, layers, ents, 64, 2, True, "70 layers")


def test_stack_kernel_in_cuda_graph(wq):
    cfg = synth.CONFIGS["qwen3_4b"]
    layers, _ = _layers(wq, cfg.d, cfg.inter, 128, 16, 4, seed=4)
    m = 1
    x = synth.activations((m, cfg.d), 11).cuda()
    ws = wq.workspace(m, cfg.d, cfg.inter, 16)
    table = wq.LayerTable(layers)
    y_eager = wq.mlp_forward(x, layers, prenorm=True, ws=ws, table=table, stack=True).clone()
    y = torch.empty_like(x)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        wq.mlp_forward(x, layers, prenorm=True, y=y, ws=ws, table=table, stack=True)
    torch.cuda.current_stream().wait_stream(s)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        wq.mlp_forward(x, layers, prenorm=True, y=y, ws=ws, table=table, stack=True)
    for _ in range(5):
        y.zero_()
        g.replay()
    torch.cuda.synchronize()
    assert wq.device_status() == 0
    assert torch.equal(y.view(torch.int16), y_eager.view(torch.int16))


def test_stack_kernel_and_chain_share_a_workspace(wq):
    # the stack kernel, the launch chain and the GEMM path in turn on one workspace
    cfg = synth.CONFIGS["qwen3_4b"]
    layers, _ = _layers(wq, cfg.d, cfg.inter, 128, 16, 2, seed=6)
    ws = wq.workspace(130, cfg.d, cfg.inter, 16)
    outs = []
    for rep in range(2):
        for m, chain in ((1, False), (1, True), (130, False), (4, False)):
            x = synth.activations((m, cfg.d), 40 + m).cuda()
            outs.append(wq.mlp_forward(x, layers, prenorm=True, ws=ws, chain=chain, stack=not chain))
    torch.cuda.synchronize()
    assert wq.device_status() == 0
    for a_, b_ in zip(outs[:4], outs[4:]):
        assert torch.equal(a_.view(torch.int16), b_.view(torch.int16))


def test_default_route_follows_the_measured_crossover(wq):
    cfg = synth.CONFIGS["qwen3_4b"]
    layers, _ = _layers(wq, cfg.d, cfg.inter, 128, 16, 2, seed=12)
    assert wq.mlp_forward_info(1, layers)["route"] == wq.ROUTE_GEMV_CHAIN
    for m in (2, 4, 8):
        assert wq.mlp_forward_info(m, layers)["route"] == wq.ROUTE_STACK
    assert wq.mlp_forward_info(16, layers)["route"] == wq.ROUTE_GEMV_CHAIN
