"""The dequant-GEMM path at few tokens (at most 64): the launch with swapped
operands (weights as the M = 128 operand, tokens as N = 16..64) vs the fp64
oracle.

Covers token counts that round up to every N (9, 16, 17, 33, 48, 64), ragged
row tiles and feature blocks, every group size, the adapter's stages, the
RMSNorm, split feature axes (2 to 32 splits whose fp32 partial sums the last
split adds in order) and a single split, 4-bit gate/up (two projections of
4-bit codes), down with a residual in bf16 and fp32 (the exact two-part
weights), and a stack of two 8B-shaped layers at 16 tokens.  Calls with
d >= 4096 take the GEMM path above 8 tokens, the others above 16.
"""
import numpy as np
import pytest
import torch

import oracle as orc
from paper_2606_04238_gb300 import synth
from tests.gpu_util import check_bf16, check_f32, upload_packed

pytestmark = pytest.mark.gpu

MIN_EXACT = 0.6  # share of bf16 outputs equal to the oracle's own rounding (binary16 weights)


@pytest.fixture(scope="module")
def wq():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2606_04238_gb300 import wq as mod
    return mod


def _q(shape, group, bits, seed):
    w = (np.random.default_rng(seed).standard_normal(shape) * 0.02).astype(np.float32)
    return orc.quantize(w, group, bits)[:3]


GATEUP_CASES = [
    # d, inter, group, r, token counts
    (4096, 256, 128, 16, (9, 16, 33, 64)),   # 2 row tiles, 32 blocks: 16 splits of 2 blocks
    (4096, 200, 64, 8, (12, 48)),            # ragged rows, 2 row tiles
    (512, 1024, 32, 0, (17, 64)),            # 8 row tiles, 4 blocks: 2 splits, no adapter
    (384, 640, 128, 32, (17, 40)),           # 3 blocks, 5 row tiles: one split
]


@pytest.mark.parametrize("d,inter,group,r,ms", GATEUP_CASES)
@pytest.mark.parametrize("prenorm", [False, True])
def test_swap_gateup(wq, d, inter, group, r, ms, prenorm):
    qg, qu = _q((inter, d), group, 2, d + inter), _q((inter, d), group, 2, d + inter + 1)
    g, u = upload_packed(*qg, group, 2), upload_packed(*qu, group, 2)
    kw, okw = {}, {}
    if r:
        a, bg, bu = synth.lora(d, inter, r, d + r)
        kw = dict(lora_a=a.cuda(), lora_b_gate=bg.cuda(), lora_b_up=bu.cuda())
        okw = dict(lora_a=synth.bf16_bits(a), lora_b_gate=synth.bf16_bits(bg), lora_b_up=synth.bf16_bits(bu))
    for m in ms:
        x = synth.activations((m, d), 10 + m)
        h = wq.gateup_w2_lora(x.cuda(), g, u, lora_scale=2.0, prenorm=prenorm, **kw)
        torch.cuda.synchronize()
        assert wq.device_status() == 0
        ref, _ = orc.gateup(synth.bf16_bits(x), qg, qu, group, okw.get("lora_a"), okw.get("lora_b_gate"),
                            okw.get("lora_b_up"), lora_scale=2.0, prenorm=prenorm)
        check_bf16(h, ref, f"swap h d={d} I={inter} g={group} r={r} m={m} prenorm={prenorm}", min_exact=MIN_EXACT)


@pytest.mark.parametrize("m", [17, 64])
def test_swap_gateup_w4(wq, m):
    d, inter, group = 512, 384, 64
    qg, qu = _q((inter, d), group, 4, 15), _q((inter, d), group, 4, 16)
    x = synth.activations((m, d), 17 + m)
    h = wq.gateup_w4(x.cuda(), upload_packed(*qg, group, 4), upload_packed(*qu, group, 4), prenorm=True)
    torch.cuda.synchronize()
    assert wq.device_status() == 0
    ref, _ = orc.gateup(synth.bf16_bits(x), qg, qu, group, None, None, None, lora_scale=0.0, prenorm=True)
    check_bf16(h, ref, f"swap W4 h m={m}", min_exact=MIN_EXACT)


DOWN_CASES = [
    # d (output rows), inter (features), group, token counts
    (384, 8192, 128, (17, 33, 64)),   # 3 row tiles, 64 blocks: 32 splits
    (4096, 512, 64, (9, 16)),         # 32 row tiles, 4 blocks: 2 splits
    (200, 1024, 32, (24,)),           # ragged rows
]


@pytest.mark.parametrize("d,inter,group,ms", DOWN_CASES)
def test_swap_down(wq, d, inter, group, ms):
    qd = _q((d, inter), group, 4, d * 3 + inter)
    dn = upload_packed(*qd, group, 4)
    for m in ms:
        h = (synth.activations((m, inter), 20 + m) * 0.5).to(torch.bfloat16)
        res = synth.activations((m, d), 30 + m)
        y = wq.down_w4(h.cuda(), dn, residual=res.cuda())
        y0 = wq.down_w4(h.cuda(), dn)
        y32 = wq.down_w4(h.cuda(), dn, residual=res.cuda(), out_f32=True)
        torch.cuda.synchronize()
        assert wq.device_status() == 0
        ref, _ = orc.down(synth.bf16_bits(h), qd, group, synth.bf16_bits(res))
        ref0, _ = orc.down(synth.bf16_bits(h), qd, group, None)
        check_bf16(y, ref, f"swap y d={d} I={inter} g={group} m={m}", min_exact=MIN_EXACT)
        check_bf16(y0, ref0, f"swap y (no residual) d={d} m={m}", min_exact=MIN_EXACT)
        check_f32(y32, ref, f"swap y fp32 d={d} m={m}")


def test_swap_is_deterministic(wq):
    d, inter, group = 384, 8192, 128
    qd = _q((d, inter), group, 4, 7)
    dn = upload_packed(*qd, group, 4)
    h = synth.activations((33, inter), 8).cuda()
    ys = [wq.down_w4(h, dn) for _ in range(3)]
    torch.cuda.synchronize()
    assert all(torch.equal(ys[0].view(torch.int16), y.view(torch.int16)) for y in ys[1:])


def test_swap_stack_8b_16_tokens(wq):
    """Two 8B-shaped layers at 16 tokens through wq_mlp_forward (the dequant-
    GEMM chain), each kernel teacher-forced on sampled tokens."""
    cfg = synth.CONFIGS["dense_8b"]
    m = 16
    layers, ents = [], []
    for l in range(2):
        wg, wu, wd = synth.layer_weights(cfg, l)
        qg = orc.quantize(wg.numpy(), cfg.group_gu, 2)[:3]
        qu = orc.quantize(wu.numpy(), cfg.group_gu, 2)[:3]
        qd = orc.quantize(wd.numpy(), cfg.group_down, 4)[:3]
        a, bg, bu = synth.lora(cfg.d, cfg.inter, cfg.r, 300 + l)
        layers.append(wq.MLPLayer(upload_packed(*qg, cfg.group_gu, 2), upload_packed(*qu, cfg.group_gu, 2),
                                  upload_packed(*qd, cfg.group_down, 4), lora_a=a.cuda(), lora_b_gate=bg.cuda(),
                                  lora_b_up=bu.cuda(), lora_scale=cfg.lora_scale))
        ents.append(dict(g=qg, u=qu, d=qd, a=synth.bf16_bits(a), bg=synth.bf16_bits(bg), bu=synth.bf16_bits(bu)))
    assert wq.mlp_forward_info(m, layers, prenorm=True)["route"] == wq.ROUTE_GEMM_CHAIN
    x = synth.activations((m, cfg.d), 310).cuda()
    _, states, h_states = wq.mlp_forward_states(x, layers, prenorm=True, with_h=True)
    torch.cuda.synchronize()
    assert wq.device_status() == 0
    rows = np.array([0, 5, 15])
    prev = synth.bf16_bits(x.cpu())
    for l, e in enumerate(ents):
        h_ref, _ = orc.gateup(prev[rows], e["g"], e["u"], cfg.group_gu, e["a"], e["bg"], e["bu"],
                              lora_scale=cfg.lora_scale, prenorm=True)
        check_bf16(h_states[l][rows], h_ref, f"8B m=16 layer {l} h", min_exact=MIN_EXACT)
        y_ref, _ = orc.down(synth.bf16_bits(h_states[l][rows].cpu()), e["d"], cfg.group_down, prev[rows])
        check_bf16(states[l][rows], y_ref, f"8B m=16 layer {l} y", min_exact=MIN_EXACT)
        prev = synth.bf16_bits(states[l].cpu())
