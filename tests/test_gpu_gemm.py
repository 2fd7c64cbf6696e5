"""The batched dequant-GEMM path (token counts above the decode GEMV's 64,
tcgen05 tensor cores) vs the fp64 oracle, through the same C ABI calls.

The GEMM multiplies binary16 copies of the activations by the dequantized
weights s (q - z) rounded once to binary16 (relative error <= 2^-11 per
weight) with fp32 accumulation, so the bf16 outputs keep the oracle bound
2e-3 (max|oracle| + 1) but match the oracle's own bf16 rounding less often
than the exact decode path; the fp32-output down call splits every weight
into two exact binary16 parts and keeps the 1e-4 relative bound.  Shapes span
ragged token tiles (65, 130, 257 tokens), ragged row tiles and feature blocks,
every group size, with and without the adapter and the RMSNorm.
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
    # d, inter, group, r
    (256, 768, 64, 8),
    (192, 200, 64, 16),    # ragged rows (200) and features (192 = 1.5 blocks)
    (384, 640, 32, 0),
    (512, 1024, 128, 32),
]


@pytest.mark.parametrize("d,inter,group,r", GATEUP_CASES)
@pytest.mark.parametrize("m", [65, 130, 257])
@pytest.mark.parametrize("prenorm", [False, True])
def test_gemm_gateup_w2_lora(wq, d, inter, group, r, m, prenorm):
    qg, qu = _q((inter, d), group, 2, d + inter), _q((inter, d), group, 2, d + inter + 1)
    x = synth.activations((m, d), 300 + m)
    kw, oa, obg, obu = {}, None, None, None
    if r:
        a, bg, bu = synth.lora(d, inter, r, 41 + r)
        kw = dict(lora_a=a.cuda(), lora_b_gate=bg.cuda(), lora_b_up=bu.cuda(), lora_scale=2.0)
        oa, obg, obu = synth.bf16_bits(a), synth.bf16_bits(bg), synth.bf16_bits(bu)
    h = wq.gateup_w2_lora(x.cuda(), upload_packed(*qg, group, 2), upload_packed(*qu, group, 2), prenorm=prenorm, **kw)
    torch.cuda.synchronize()
    assert wq.device_status() == 0
    ref, _ = orc.gateup(synth.bf16_bits(x), qg, qu, group, oa, obg, obu, lora_scale=2.0 if r else 0.0, prenorm=prenorm)
    check_bf16(h, ref, f"GEMM h d={d} I={inter} g={group} r={r} m={m} prenorm={prenorm}", min_exact=MIN_EXACT)


@pytest.mark.parametrize("m", [65, 200])
def test_gemm_gateup_w4(wq, m):
    d, inter, group = 256, 512, 128
    qg, qu = _q((inter, d), group, 4, 5), _q((inter, d), group, 4, 6)
    x = synth.activations((m, d), 7)
    h = wq.gateup_w4(x.cuda(), upload_packed(*qg, group, 4), upload_packed(*qu, group, 4), prenorm=True)
    torch.cuda.synchronize()
    assert wq.device_status() == 0
    ref, _ = orc.gateup(synth.bf16_bits(x), qg, qu, group, None, None, None, lora_scale=0.0, prenorm=True)
    check_bf16(h, ref, f"GEMM W4 h m={m}", min_exact=MIN_EXACT)


DOWN_CASES = [
    # d, inter, group
    (256, 768, 64),
    (200, 384, 32),       # ragged output rows
    (512, 1024, 128),
    (384, 960, 64),       # ragged feature blocks (7.5)
]


@pytest.mark.parametrize("d,inter,group", DOWN_CASES)
@pytest.mark.parametrize("m", [65, 130])
@pytest.mark.parametrize("residual", [False, True])
def test_gemm_down_w4(wq, d, inter, group, m, residual):
    qd = _q((d, inter), group, 4, d * 3 + inter)
    h = synth.activations((m, inter), 11 + m) * 0.5
    h = h.to(torch.bfloat16)
    res = synth.activations((m, d), 13 + m) if residual else None
    dn = upload_packed(*qd, group, 4)
    y = wq.down_w4(h.cuda(), dn, residual=None if res is None else res.cuda())
    y32 = wq.down_w4(h.cuda(), dn, residual=None if res is None else res.cuda(), out_f32=True)
    torch.cuda.synchronize()
    assert wq.device_status() == 0
    ref, _ = orc.down(synth.bf16_bits(h), qd, group, None if res is None else synth.bf16_bits(res))
    check_bf16(y, ref, f"GEMM y d={d} I={inter} g={group} m={m}", min_exact=MIN_EXACT)
    check_f32(y32, ref, f"GEMM y(f32) d={d} I={inter} g={group} m={m}")


@pytest.mark.parametrize("m", [100, 300])
def test_gemm_stack_matches_oracle(wq, m):
    """wq_mlp_forward above the decode limit: the GEMM chain (inputs kernel,
    gate/up handing h in binary16 to down) vs the oracle, teacher-forced per
    layer through the single-layer calls, and end to end."""
    cfg = synth.CONFIGS["small_d256_i768"]
    n_layers = 3
    layers, ents = [], []
    for l in range(n_layers):
        wg, wu, wd = synth.layer_weights(cfg, l)
        qg = orc.quantize(wg.numpy(), cfg.group_gu, 2)[:3]
        qu = orc.quantize(wu.numpy(), cfg.group_gu, 2)[:3]
        qd = orc.quantize(wd.numpy(), cfg.group_down, 4)[:3]
        a, bg, bu = synth.lora(cfg.d, cfg.inter, cfg.r, 900 + l)
        ents.append(dict(g=qg, u=qu, d=qd, a=synth.bf16_bits(a), bg=synth.bf16_bits(bg), bu=synth.bf16_bits(bu)))
        layers.append(wq.MLPLayer(upload_packed(*qg, cfg.group_gu, 2), upload_packed(*qu, cfg.group_gu, 2),
                                  upload_packed(*qd, cfg.group_down, 4), lora_a=a.cuda(), lora_b_gate=bg.cuda(),
                                  lora_b_up=bu.cuda(), lora_scale=cfg.lora_scale))
    x = synth.activations((m, cfg.d), 77)
    ws = wq.workspace(m, cfg.d, cfg.inter, cfg.r)
    y = wq.mlp_forward(x.cuda(), layers, prenorm=True, ws=ws)
    # teacher-forced: layer l of the oracle on the GPU's own layer l-1 output
    cur = x.cuda()
    for l, ent in enumerate(ents):
        out = wq.mlp_forward(cur, layers[l:l + 1], prenorm=True, ws=ws)
        torch.cuda.synchronize()
        _, hb = orc.gateup(synth.bf16_bits(cur.cpu()), ent["g"], ent["u"], cfg.group_gu, ent["a"], ent["bg"], ent["bu"],
                           lora_scale=cfg.lora_scale, prenorm=True)
        ref, _ = orc.down(hb, ent["d"], cfg.group_down, synth.bf16_bits(cur.cpu()))
        check_bf16(out, ref, f"GEMM stack layer {l} m={m}", min_exact=MIN_EXACT)
        cur = out
    torch.cuda.synchronize()
    assert wq.device_status() == 0
    assert torch.equal(y, cur), "the stack call differs from its layers called one by one"


@pytest.mark.parametrize("m", [257, 300, 512])
def test_gemm_two_token_halves(wq, m):
    """Enough 256-token x 128-row tiles for every SM: each CTA takes two token
    halves of 128 that share the dequantized B tile (the last CTA of m = 300
    holds one half).  Gate/up with the adapter and the RMSNorm, then down with
    a residual, in bf16 and fp32."""
    d, inter, group, r = 256, 9728, 64, 16
    qg, qu = _q((inter, d), group, 2, 71), _q((inter, d), group, 2, 72)
    a, bg, bu = synth.lora(d, inter, r, 73)
    x = synth.activations((m, d), 74 + m)
    h = wq.gateup_w2_lora(x.cuda(), upload_packed(*qg, group, 2), upload_packed(*qu, group, 2), prenorm=True,
                          lora_a=a.cuda(), lora_b_gate=bg.cuda(), lora_b_up=bu.cuda(), lora_scale=2.0)
    torch.cuda.synchronize()
    assert wq.device_status() == 0
    ref, _ = orc.gateup(synth.bf16_bits(x), qg, qu, group, synth.bf16_bits(a), synth.bf16_bits(bg),
                        synth.bf16_bits(bu), lora_scale=2.0, prenorm=True)
    check_bf16(h, ref, f"GEMM h (two halves) m={m}", min_exact=MIN_EXACT)
    # down: 9728 output rows from 256 features
    qd = _q((inter, d), group, 4, 75)
    hd = (synth.activations((m, d), 76 + m) * 0.5).to(torch.bfloat16)
    res = synth.activations((m, inter), 77 + m)
    dn = upload_packed(*qd, group, 4)
    y = wq.down_w4(hd.cuda(), dn, residual=res.cuda())
    y32 = wq.down_w4(hd.cuda(), dn, residual=res.cuda(), out_f32=True)
    torch.cuda.synchronize()
    assert wq.device_status() == 0
    ref, _ = orc.down(synth.bf16_bits(hd), qd, group, synth.bf16_bits(res))
    check_bf16(y, ref, f"GEMM y (two halves) m={m}", min_exact=MIN_EXACT)
    check_f32(y32, ref, f"GEMM y(f32) (two halves) m={m}")


def test_planless_decode_shape_takes_gemm(wq):
    """64 tokens of the 14B-shaped layer (d=5120, inter=17408): the decode
    GEMV kernels have no launch configuration at this size, so the calls (and
    the stack) take the dequant-GEMM path under the same results contract."""
    cfg = synth.CONFIGS["dense_14b"]
    m = 64
    wg, wu, wd = synth.layer_weights(cfg, 0)
    qg = orc.quantize(wg.numpy(), cfg.group_gu, 2)[:3]
    qu = orc.quantize(wu.numpy(), cfg.group_gu, 2)[:3]
    qd = orc.quantize(wd.numpy(), cfg.group_down, 4)[:3]
    del wg, wu, wd
    a, bg, bu = synth.lora(cfg.d, cfg.inter, cfg.r, 17)
    x = synth.activations((m, cfg.d), 19)
    layer = wq.MLPLayer(upload_packed(*qg, cfg.group_gu, 2), upload_packed(*qu, cfg.group_gu, 2),
                        upload_packed(*qd, cfg.group_down, 4), lora_a=a.cuda(), lora_b_gate=bg.cuda(),
                        lora_b_up=bu.cuda(), lora_scale=cfg.lora_scale)
    ws = wq.workspace(m, cfg.d, cfg.inter, cfg.r)
    h = wq.gateup_w2_lora(x.cuda(), layer.gate, layer.up, layer.lora_a, layer.lora_b_gate, layer.lora_b_up,
                          cfg.lora_scale, prenorm=True, ws=ws)
    y = wq.mlp_forward(x.cuda(), [layer], prenorm=True, ws=ws)
    torch.cuda.synchronize()
    assert wq.device_status() == 0
    xb = synth.bf16_bits(x)
    ref_h, hb = orc.gateup(xb, qg, qu, cfg.group_gu, synth.bf16_bits(a), synth.bf16_bits(bg), synth.bf16_bits(bu),
                           lora_scale=cfg.lora_scale, prenorm=True)
    check_bf16(h, ref_h, "14B gate/up m=64", min_exact=MIN_EXACT)
    ref_y, _ = orc.down(synth.bf16_bits(h.cpu()), qd, cfg.group_down, xb)  # teacher-forced on the GPU's h
    check_bf16(y, ref_y, "14B stack m=64", min_exact=MIN_EXACT)


@pytest.mark.parametrize("m", [65, 200])
def test_gemm_stream_k_split_tiles(wq, m):
    """Few output tiles over a long feature axis (8192 features, 64 blocks):
    the launch runs stream-K, every tile split over several CTAs, the LoRA
    stages in the last part; gate/up with adapter and RMSNorm, then down
    (8192 -> 384 rows) with a residual in bf16 and fp32."""
    d, inter, group, r = 8192, 384, 128, 16
    qg, qu = _q((inter, d), group, 2, 91), _q((inter, d), group, 2, 92)
    a, bg, bu = synth.lora(d, inter, r, 93)
    x = synth.activations((m, d), 94 + m)
    h = wq.gateup_w2_lora(x.cuda(), upload_packed(*qg, group, 2), upload_packed(*qu, group, 2), prenorm=True,
                          lora_a=a.cuda(), lora_b_gate=bg.cuda(), lora_b_up=bu.cuda(), lora_scale=2.0)
    torch.cuda.synchronize()
    assert wq.device_status() == 0
    ref, _ = orc.gateup(synth.bf16_bits(x), qg, qu, group, synth.bf16_bits(a), synth.bf16_bits(bg),
                        synth.bf16_bits(bu), lora_scale=2.0, prenorm=True)
    check_bf16(h, ref, f"GEMM h (stream-K) m={m}", min_exact=MIN_EXACT)
    qd = _q((inter, d), group, 4, 95)  # down: inter (384) output rows from d (8192) features
    hd = (synth.activations((m, d), 96 + m) * 0.5).to(torch.bfloat16)
    res = synth.activations((m, inter), 97 + m)
    dn = upload_packed(*qd, group, 4)
    y = wq.down_w4(hd.cuda(), dn, residual=res.cuda())
    y32 = wq.down_w4(hd.cuda(), dn, residual=res.cuda(), out_f32=True)
    torch.cuda.synchronize()
    assert wq.device_status() == 0
    ref, _ = orc.down(synth.bf16_bits(hd), qd, group, synth.bf16_bits(res))
    check_bf16(y, ref, f"GEMM y (stream-K) m={m}", min_exact=MIN_EXACT)
    check_f32(y32, ref, f"GEMM y(f32) (stream-K) m={m}")
