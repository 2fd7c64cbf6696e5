"""The MLP stack (wq_mlp_forward) vs the oracle, layer by layer.

Each layer is checked teacher-forced: the oracle's layer l takes the GPU's
output of layer l-1 as its input, so a kernel error cannot hide behind the
drift of 36 bf16 roundings.  The end-to-end error is checked with the same
bound on short stacks."""
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


def _build_stack(wq, cfg, n_layers, bits_gu=2, lora=True):
    layers, orc_layers = [], []
    for l in range(n_layers):
        wg, wu, wd = synth.layer_weights(cfg, l)
        qg = orc.quantize(wg.numpy(), cfg.group_gu, bits_gu)[:3]
        qu = orc.quantize(wu.numpy(), cfg.group_gu, bits_gu)[:3]
        qd = orc.quantize(wd.numpy(), cfg.group_down, 4)[:3]
        ent = dict(g=qg, u=qu, d=qd)
        kw = {}
        if lora and bits_gu == 2:
            a, bg, bu = synth.lora(cfg.d, cfg.inter, cfg.r, 500 + l)
            ent.update(a=synth.bf16_bits(a), bg=synth.bf16_bits(bg), bu=synth.bf16_bits(bu))
            kw = dict(lora_a=a.cuda(), lora_b_gate=bg.cuda(), lora_b_up=bu.cuda(), lora_scale=cfg.lora_scale)
        layers.append(wq.MLPLayer(upload_packed(*qg, cfg.group_gu, bits_gu), upload_packed(*qu, cfg.group_gu, bits_gu),
                                  upload_packed(*qd, cfg.group_down, 4), **kw))
        orc_layers.append(ent)
    return layers, orc_layers


def _orc_layer(cfg, ent, x_bits, prenorm):
    h, hb = orc.gateup(x_bits, ent["g"], ent["u"], cfg.group_gu, ent.get("a"), ent.get("bg"), ent.get("bu"),
                       lora_scale=cfg.lora_scale if "a" in ent else 0.0, prenorm=prenorm)
    y, yb = orc.down(hb, ent["d"], cfg.group_down, x_bits)
    return y, yb


@pytest.mark.parametrize("m", [1, 4, 16])
@pytest.mark.parametrize("bits_gu", [2, 4])
def test_stack_teacher_forced(wq, m, bits_gu):
    cfg = synth.CONFIGS["small_d256_i768"]
    n_layers = 6
    layers, ent = _build_stack(wq, cfg, n_layers, bits_gu)
    x = synth.activations((m, cfg.d), 42).cuda()
    ws = wq.workspace(m, cfg.d, cfg.inter, cfg.r)
    prefix = [x]
    for l in range(1, n_layers + 1):
        prefix.append(wq.mlp_forward(x, layers[:l], prenorm=True, ws=ws))
    torch.cuda.synchronize()
    assert wq.device_status() == 0
    for l in range(n_layers):
        ref, _ = _orc_layer(cfg, ent[l], synth.bf16_bits(prefix[l]), prenorm=True)
        check_bf16(prefix[l + 1], ref, f"layer {l} (teacher-forced) m={m} bits={bits_gu}")
    # end to end on the oracle's own chain
    xb = synth.bf16_bits(x)
    for l in range(n_layers):
        y, xb = _orc_layer(cfg, ent[l], xb, prenorm=True)
    check_bf16(prefix[-1], y, f"stack end-to-end m={m}", min_exact=0.5, depth=n_layers)


def test_stack_equals_layer_calls(wq):
    cfg = synth.CONFIGS["small_d256_i768"]
    layers, _ = _build_stack(wq, cfg, 3)
    m = 2
    x = synth.activations((m, cfg.d), 3).cuda()
    ws = wq.workspace(m, cfg.d, cfg.inter, cfg.r)
    y_stack = wq.mlp_forward(x, layers, prenorm=True, ws=ws)
    cur = x
    for L in layers:
        h = wq.gateup_w2_lora(cur, L.gate, L.up, L.lora_a, L.lora_b_gate, L.lora_b_up, L.lora_scale, prenorm=True,
                              ws=ws)
        cur = wq.down_w4(h, L.down, residual=cur, ws=ws)
    torch.cuda.synchronize()
    assert torch.equal(y_stack.view(torch.int16), cur.view(torch.int16))


def test_stack_in_cuda_graph(wq):
    cfg = synth.CONFIGS["small_d256_i768"]
    layers, _ = _build_stack(wq, cfg, 4)
    m = 1
    x = synth.activations((m, cfg.d), 5).cuda()
    ws = wq.workspace(m, cfg.d, cfg.inter, cfg.r)
    table = wq.LayerTable(layers)
    y_eager = wq.mlp_forward(x, layers, prenorm=True, ws=ws, table=table).clone()
    y = torch.empty_like(x)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        wq.mlp_forward(x, layers, prenorm=True, y=y, ws=ws, table=table)  # warm-up outside capture
    torch.cuda.current_stream().wait_stream(s)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        wq.mlp_forward(x, layers, prenorm=True, y=y, ws=ws, table=table)
    for _ in range(3):
        y.zero_()
        g.replay()
    torch.cuda.synchronize()
    assert torch.equal(y.view(torch.int16), y_eager.view(torch.int16))
