"""App. B's W3-GateUp variant on the GPU: 3-bit gate/up codes (two bit
planes) through wq_gateup_w3_lora and the decode stack, vs the oracle.

The kernels read a 3-bit code as the 2-bit low plane plus one bit of the
second plane shifted next to it, so a mistake in the plane layout, the shift
or the mask shows as a wrong product.  Shapes: ragged rows and feature
blocks, every group size (g32 is the paper's INT3 setting), 1..64 tokens
(3-bit codes stay on the dequant-GEMV kernels at every token count), with
and without the RMSNorm and the adapter; a two-layer stack teacher-forced
per layer; the Qwen3-4B shape at g32.
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


def _q(shape, group, bits, seed, std=0.02):
    w = (np.random.default_rng(seed).standard_normal(shape) * std).astype(np.float32)
    return orc.quantize(w, group, bits)[:3]


W3_CASES = [
    # d, inter, group, r
    (256, 768, 32, 8),
    (192, 200, 64, 16),     # ragged rows and features
    (384, 80, 32, 0),
    (512, 1000, 128, 32),
    (4096, 48, 32, 8),      # few rows, many feature blocks
]


@pytest.mark.parametrize("d,inter,group,r", W3_CASES)
@pytest.mark.parametrize("m", [1, 3, 9, 16, 40, 64])
@pytest.mark.parametrize("prenorm", [False, True])
def test_gateup_w3_lora(wq, d, inter, group, r, m, prenorm):
    qg, qu = _q((inter, d), group, 3, d + inter), _q((inter, d), group, 3, d + inter + 1)
    assert qg[0].max() == 7  # every code value occurs
    x = synth.activations((m, d), 100 + m)
    kw, okw = {}, {}
    if r:
        a, bg, bu = synth.lora(d, inter, r, d + r)
        kw = dict(lora_a=a.cuda(), lora_b_gate=bg.cuda(), lora_b_up=bu.cuda())
        okw = dict(lora_a=synth.bf16_bits(a), lora_b_gate=synth.bf16_bits(bg), lora_b_up=synth.bf16_bits(bu))
    h = wq.gateup_w3_lora(x.cuda(), upload_packed(*qg, group, 3), upload_packed(*qu, group, 3), lora_scale=2.0,
                          prenorm=prenorm, **kw)
    torch.cuda.synchronize()
    assert wq.device_status() == 0
    ref, _ = orc.gateup(synth.bf16_bits(x), qg, qu, group, okw.get("lora_a"), okw.get("lora_b_gate"),
                        okw.get("lora_b_up"), lora_scale=2.0, prenorm=prenorm)
    check_bf16(h, ref, f"W3 h d={d} I={inter} g={group} r={r} m={m} prenorm={prenorm}")


def test_w3_above_64_tokens_is_refused(wq):
    d, inter, group = 256, 256, 32
    qg = _q((inter, d), group, 3, 1)
    g = upload_packed(*qg, group, 3)
    x = synth.activations((65, d), 2).cuda()
    with pytest.raises(wq.WQError):
        wq.gateup_w3_lora(x, g, g)


def _layers(wq, d, inter, group, r, n, seed):
    layers, ents = [], []
    for l in range(n):
        qg, qu, qd = _q((inter, d), group, 3, seed + 3 * l), _q((inter, d), group, 3, seed + 3 * l + 1), \
            _q((d, inter), group, 4, seed + 3 * l + 2)
        a, bg, bu = synth.lora(d, inter, r, seed + 100 + l)
        layers.append(wq.MLPLayer(upload_packed(*qg, group, 3), upload_packed(*qu, group, 3),
                                  upload_packed(*qd, group, 4), lora_a=a.cuda(), lora_b_gate=bg.cuda(),
                                  lora_b_up=bu.cuda(), lora_scale=2.0))
        ents.append(dict(g=qg, u=qu, d=qd, a=synth.bf16_bits(a), bg=synth.bf16_bits(bg), bu=synth.bf16_bits(bu)))
    return layers, ents


def _stack_check(wq, d, inter, group, r, n, m, seed, what):
    layers, ents = _layers(wq, d, inter, group, r, n, seed)
    info = wq.mlp_forward_info(m, layers, prenorm=True)
    assert info["route"] == wq.ROUTE_GEMV_CHAIN, info
    x = synth.activations((m, d), seed + 7).cuda()
    y, states, h_states = wq.mlp_forward_states(x, layers, prenorm=True, with_h=True)
    torch.cuda.synchronize()
    assert wq.device_status() == 0
    prev = synth.bf16_bits(x.cpu())
    for l, e in enumerate(ents):
        h_ref, _ = orc.gateup(prev, e["g"], e["u"], group, e["a"], e["bg"], e["bu"], lora_scale=2.0, prenorm=True)
        check_bf16(h_states[l], h_ref, f"{what} layer {l} h")
        y_ref, _ = orc.down(synth.bf16_bits(h_states[l].cpu()), e["d"], group, prev)
        check_bf16(states[l], y_ref, f"{what} layer {l} y")
        prev = synth.bf16_bits(states[l].cpu())


@pytest.mark.parametrize("m", [1, 4, 24])
def test_w3_stack_teacher_forced(wq, m):
    _stack_check(wq, 512, 1024, 32, 16, 2, m, 900 + m, f"W3 stack m={m}")


def test_w3_qwen3_4b_g32(wq):
    cfg = synth.CONFIGS["qwen3_4b"]
    _stack_check(wq, cfg.d, cfg.inter, 32, cfg.r, 2, 1, 1234, "W3 Qwen3-4B g32")
