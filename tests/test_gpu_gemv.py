"""Fused dequant-GEMV kernels vs the fp64 oracle (Eq. 1 LoRA, Sec. 3.3 gated
MLP with 2-bit gate/up and 4-bit down), through the C ABI.

Shapes span several row tiles and feature blocks, ragged row and feature
tails, every supported group size and both panel modes (one CTA per row
block, and split panels finished by the last-arriving CTA).  The GEMV kernels
take 1..16 tokens; the 17/33/64-token cases here take the dequant-GEMM path.
"""
import numpy as np
import pytest
import torch

import oracle as orc
from paper_2606_04238_gb300 import synth
from tests.gpu_util import check_bf16, check_f32, upload_packed

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def wq():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2606_04238_gb300 import wq as mod
    return mod


def _layer(d, inter, g_gu, g_d, r, seed, bits_gu=2):
    rng = np.random.default_rng(seed)
    wg = (rng.standard_normal((inter, d)) * 0.02).astype(np.float32)
    wu = (rng.standard_normal((inter, d)) * 0.02).astype(np.float32)
    wd = (rng.standard_normal((d, inter)) * 0.02).astype(np.float32)
    L = {"g": orc.quantize(wg, g_gu, bits_gu)[:3], "u": orc.quantize(wu, g_gu, bits_gu)[:3],
         "d": orc.quantize(wd, g_d, 4)[:3] if inter % g_d == 0 else None}
    if r:
        a, bg, bu = synth.lora(d, inter, r, seed + 7)
        L.update(a=a, bg=bg, bu=bu)
    return L


def _dev_lora(L):
    if "a" not in L:
        return None, None, None
    return L["a"].cuda(), L["bg"].cuda(), L["bu"].cuda()


def _orc_lora(L):
    if "a" not in L:
        return None, None, None
    return synth.bf16_bits(L["a"]), synth.bf16_bits(L["bg"]), synth.bf16_bits(L["bu"])


GATEUP_CASES = [
    # d, inter, group, r
    (256, 768, 64, 8),      # the small single-layer workload
    (192, 200, 64, 16),     # ragged rows (200 = 12.5 tiles) and features (192 = 1.5 blocks)
    (384, 80, 32, 0),       # group 32, no adapter
    (512, 1000, 128, 32),   # group 128, ragged rows
    (4096, 48, 128, 8),     # few rows, many feature blocks
    (8192, 16, 128, 8),     # one row tile, 64 feature blocks
    (16384, 32, 64, 8),     # two row tiles, 128 feature blocks
]


@pytest.mark.parametrize("d,inter,group,r", GATEUP_CASES)
@pytest.mark.parametrize("m", [1, 3, 8, 9, 16])
@pytest.mark.parametrize("prenorm", [False, True])
def test_gateup_w2_lora(wq, d, inter, group, r, m, prenorm):
    L = _layer(d, inter, group, 64, r, seed=d + inter + r)
    x = synth.activations((m, d), 100 + m)
    g = upload_packed(*L["g"], group, 2)
    u = upload_packed(*L["u"], group, 2)
    a, bg, bu = _dev_lora(L)
    h = wq.gateup_w2_lora(x.cuda(), g, u, a, bg, bu, lora_scale=2.0, prenorm=prenorm)
    torch.cuda.synchronize()
    oa, obg, obu = _orc_lora(L)
    ref, _ = orc.gateup(synth.bf16_bits(x), L["g"], L["u"], group, oa, obg, obu, lora_scale=2.0, prenorm=prenorm)
    check_bf16(h, ref, f"h d={d} I={inter} g={group} r={r} m={m} prenorm={prenorm}")


@pytest.mark.parametrize("m", [17, 33, 64])
def test_gateup_w2_many_tokens(wq, m):
    """Above 16 tokens the call takes the dequant-GEMM path (weights rounded
    once to binary16): the bound is unchanged, the share of outputs equal to
    the oracle's own bf16 rounding is that path's (0.6)."""
    d, inter, group, r = 512, 384, 64, 16
    L = _layer(d, inter, group, 64, r, seed=5)
    x = synth.activations((m, d), 7)
    g, u = upload_packed(*L["g"], group, 2), upload_packed(*L["u"], group, 2)
    a, bg, bu = _dev_lora(L)
    h = wq.gateup_w2_lora(x.cuda(), g, u, a, bg, bu, lora_scale=2.0, prenorm=True)
    torch.cuda.synchronize()
    ref, _ = orc.gateup(synth.bf16_bits(x), L["g"], L["u"], group, *_orc_lora(L), lora_scale=2.0, prenorm=True)
    check_bf16(h, ref, f"h m={m}", min_exact=0.6)


@pytest.mark.parametrize("d,inter,group", [(256, 768, 64), (384, 200, 32), (512, 1000, 128)])
@pytest.mark.parametrize("m", [1, 5, 16])
def test_gateup_w4(wq, d, inter, group, m):
    L = _layer(d, inter, group, 64, 0, seed=3 * d + m, bits_gu=4)
    x = synth.activations((m, d), 11 + m)
    g, u = upload_packed(*L["g"], group, 4), upload_packed(*L["u"], group, 4)
    h = wq.gateup_w4(x.cuda(), g, u, prenorm=True)
    torch.cuda.synchronize()
    ref, _ = orc.gateup(synth.bf16_bits(x), L["g"], L["u"], group, prenorm=True)
    check_bf16(h, ref, f"h(w4) d={d} I={inter} m={m}")


DOWN_CASES = [(256, 768, 64), (200, 384, 32), (1000, 512, 128), (48, 4096, 128), (256, 192, 64), (64, 8192, 128)]


@pytest.mark.parametrize("d,inter,group", DOWN_CASES)
@pytest.mark.parametrize("m", [1, 4, 8, 12, 16])
@pytest.mark.parametrize("residual", [False, True])
def test_down_w4(wq, d, inter, group, m, residual):
    rng = np.random.default_rng(d * 7 + inter + m)
    wd = (rng.standard_normal((d, inter)) * 0.02).astype(np.float32)
    qd = orc.quantize(wd, group, 4)[:3]
    dn = upload_packed(*qd, group, 4)
    h = synth.activations((m, inter), 3 + m)
    res = synth.activations((m, d), 4 + m) if residual else None
    y = wq.down_w4(h.cuda(), dn, residual=None if res is None else res.cuda())
    y32 = wq.down_w4(h.cuda(), dn, residual=None if res is None else res.cuda(), out_f32=True)
    torch.cuda.synchronize()
    ref, _ = orc.down(synth.bf16_bits(h), qd, group, None if res is None else synth.bf16_bits(res))
    check_bf16(y, ref, f"y d={d} I={inter} m={m}")
    check_f32(y32, ref, f"y(f32) d={d} I={inter} m={m}")


def test_split_panels_are_exercised(wq):
    # some of the parity cases above must take the multi-panel path (last-
    # arriving CTA adds the panel partials), and some the single-panel path
    gu = [wq.plan_info(wq.KIND_GATEUP_W2, i, d, m, g, r)["panels"]
          for d, i, g, r in GATEUP_CASES for m in (1, 3, 8, 9, 16)]
    dn = [wq.plan_info(wq.KIND_DOWN_W4, d, i, m, g)["panels"]
          for d, i, g in DOWN_CASES for m in (1, 4, 8, 12, 16)]
    assert max(gu) > 1 and min(gu) == 1
    assert max(dn) > 1 and min(dn) == 1


def test_deterministic_across_calls(wq):
    d, inter, group, r = 4096, 48, 128, 8
    L = _layer(d, inter, group, 64, r, seed=1)
    x = synth.activations((4, d), 2).cuda()
    g, u = upload_packed(*L["g"], group, 2), upload_packed(*L["u"], group, 2)
    a, bg, bu = _dev_lora(L)
    ws = wq.workspace(4, d, inter, r)
    outs = [wq.gateup_w2_lora(x, g, u, a, bg, bu, lora_scale=2.0, ws=ws).clone() for _ in range(3)]
    torch.cuda.synchronize()
    for o in outs[1:]:
        assert torch.equal(o.view(torch.int16), outs[0].view(torch.int16))
    assert wq.device_status() == 0


def test_zero_tokens_is_noop(wq):
    L = _layer(256, 64, 64, 64, 0, seed=9)
    g, u = upload_packed(*L["g"], 64, 2), upload_packed(*L["u"], 64, 2)
    x = torch.empty((0, 256), dtype=torch.bfloat16, device="cuda")
    h = wq.gateup_w2_lora(x, g, u, ws=wq.workspace(1, 256, 64))
    assert h.shape == (0, 64)


def test_workspace_too_small_is_rejected(wq):
    L = _layer(256, 64, 64, 64, 0, seed=9)
    g, u = upload_packed(*L["g"], 64, 2), upload_packed(*L["u"], 64, 2)
    x = synth.activations((2, 256), 1).cuda()
    small = torch.zeros(64, dtype=torch.uint8, device="cuda")
    with pytest.raises(wq.WQError) as e:
        wq.gateup_w2_lora(x, g, u, ws=small)
    assert e.value.status == -7
