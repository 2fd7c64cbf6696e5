"""The mixture-of-experts block on the GPU (wq_moe_forward) vs the oracle.

Checked per step, teacher-forced on the GPU's own intermediates:
- the routing: expert indices equal the oracle's top-k (ties to the lower
  index) exactly, the softmax weights within fp32 rounding;
- h of every slot (token t, choice j) against the oracle's gate/up of the
  selected expert on x[t];
- every slot's fp32 expert output against the oracle's down on the GPU's h;
- y against x + sum_j w_j y_j from the GPU's weights and slot outputs;
and the block end to end against oracle.moe.moe_block.  Shapes: a small
block with every expert quantized, ties in the router logits, and a
GPT-OSS-20B-shaped block (d = 2880, 32 experts of width 2880, top-4, g64)
whose unselected experts hold NaN scales, so that reading one would show.
"""
import numpy as np
import pytest
import torch

import oracle as orc
from oracle import moe as omoe
from paper_2606_04238_gb300 import synth
from tests.gpu_util import check_bf16, check_f32

pytestmark = pytest.mark.gpu

NAN_F16 = np.uint16(0x7E00)


@pytest.fixture(scope="module")
def wq():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2606_04238_gb300 import wq as mod
    return mod


def _q(shape, group, bits, seed):
    w = (np.random.default_rng(seed).standard_normal(shape) * 0.02).astype(np.float32)
    return orc.quantize(w, group, bits)[:3]


def _stack_packed(qs, n, k, group, bits, dev="cuda"):
    """Experts' (q, s, z) (None: an expert whose scales and zeros are NaN)
    packed by the oracle and stacked row-wise into one device QWeight."""
    from paper_2606_04238_gb300 import wq
    codes, metas = [], []
    for q in qs:
        if q is None:
            zq = np.zeros((n, k), np.uint8)
            zs = np.zeros((n, k // group), np.uint16)
            c, m = orc.tile_pack(zq, zs, zs, group, bits)
            m = np.full_like(m, NAN_F16)
        else:
            c, m = orc.tile_pack(*q, group, bits)
        codes.append(c)
        metas.append(m)
    c = np.concatenate(codes)
    m = np.concatenate(metas)
    return wq.QWeight(torch.from_numpy(c.view(np.int32)).to(dev), torch.from_numpy(m.view(np.int16)).to(dev),
                      n * len(qs), k, group, bits)


def _build(wq, d, inter, E, top_k, group, r, seed, real=None):
    """E experts (only those in `real` quantized when given); returns the
    device MoELayer and the oracle's expert list."""
    ents, g, u, dn = [], [], [], []
    for e in range(E):
        if real is not None and e not in real:
            ents.append(None)
            g.append(None), u.append(None), dn.append(None)
            continue
        qg, qu, qd = _q((inter, d), group, 2, seed + 10 * e), _q((inter, d), group, 2, seed + 10 * e + 1), \
            _q((d, inter), group, 4, seed + 10 * e + 2)
        ents.append(dict(gate=qg, up=qu, down=qd))
        g.append(qg), u.append(qu), dn.append(qd)
    kw = {}
    if r:
        _, bg, bu = synth.lora(d, E * inter, r, seed + 7)  # lora_b rows stacked [E*inter, r]
        a_all = synth.weights((E * 2 * r, d), seed + 8, std=0.01).to(torch.bfloat16)  # [E][2r][d]
        kw = dict(lora_a=a_all.cuda(), lora_b_gate=bg.cuda(), lora_b_up=bu.cuda(), lora_scale=2.0)
        ab, bgb, bub = synth.bf16_bits(a_all), synth.bf16_bits(bg), synth.bf16_bits(bu)
        for e, ent in enumerate(ents):
            if ent is not None:
                ent["lora"] = (ab[e * 2 * r:(e + 1) * 2 * r], bgb[e * inter:(e + 1) * inter],
                               bub[e * inter:(e + 1) * inter])
    experts = wq.MLPLayer(_stack_packed(g, inter, d, group, 2), _stack_packed(u, inter, d, group, 2),
                          _stack_packed(dn, d, inter, group, 4), **kw)
    return wq.MoELayer(experts, E, top_k), ents


def _check_block(wq, layer, ents, x, logits, group, what, lora_scale):
    m, d = x.shape
    k = layer.top_k
    y, idx, wt, hs, ys = wq.moe_forward(x.cuda(), logits.cuda(), layer, prenorm=True, with_slots=True)
    torch.cuda.synchronize()
    assert wq.device_status() == 0
    xb = synth.bf16_bits(x)
    lg = logits.numpy().astype(np.float64)
    ridx, rw = omoe.route(lg, k)
    assert np.array_equal(idx.cpu().numpy(), ridx), f"{what}: expert indices {idx.cpu().numpy()} vs {ridx}"
    np.testing.assert_allclose(wt.cpu().numpy(), rw, rtol=2e-6, atol=1e-7, err_msg=f"{what}: routing weights")
    hb = synth.bf16_bits(hs.cpu())
    for t in range(m):
        for j in range(k):
            s = t * k + j
            ent = ents[int(ridx[t, j])]
            la, lbg, lbu = ent.get("lora") or (None, None, None)
            h_ref, _ = orc.gateup(xb[t:t + 1], ent["gate"], ent["up"], group, la, lbg, lbu, lora_scale=lora_scale,
                                  prenorm=True)
            check_bf16(hs[s:s + 1], h_ref, f"{what} h of slot {s} (expert {ridx[t, j]})")
            y_ref, _ = orc.down(hb[s:s + 1], ent["down"], group, None)
            check_f32(ys[s:s + 1], y_ref, f"{what} expert output of slot {s}")
    # the combine step from the GPU's own weights and slot outputs
    comb = orc.bf16_bits_to_f64(xb) + np.einsum(
        "tj,tjn->tn", wt.cpu().numpy().astype(np.float64), ys.cpu().numpy().astype(np.float64).reshape(m, k, d))
    check_bf16(y, comb, f"{what} combined y")
    # end to end: bf16 roundings of h between the oracle and the GPU
    ref, _, _, _ = omoe.moe_block(xb, lg, k, ents, group, group, lora_scale=lora_scale)
    check_bf16(y, ref, f"{what} y end to end", min_exact=0.5, depth=2)


@pytest.mark.parametrize("m", [1, 3])
@pytest.mark.parametrize("r", [0, 8])
def test_small_moe_block(wq, m, r):
    d, inter, E, k, group = 256, 256, 8, 2, 64
    layer, ents = _build(wq, d, inter, E, k, group, r, 100 + r)
    x = synth.activations((m, d), 7 + m)
    logits = torch.from_numpy(np.random.default_rng(9 + m).standard_normal((m, E)).astype(np.float32))
    _check_block(wq, layer, ents, x, logits, group, f"small m={m} r={r}", 2.0 if r else 0.0)


def test_router_ties_go_to_the_lower_index(wq):
    d, inter, E, k, group = 256, 128, 6, 3, 32
    layer, ents = _build(wq, d, inter, E, k, group, 0, 300)
    x = synth.activations((2, d), 11)
    logits = torch.tensor([[0.5, 1.0, 1.0, 0.5, 1.0, -2.0], [0.25, 0.25, 0.25, 0.25, 0.25, 0.25]],
                          dtype=torch.float32)
    _check_block(wq, layer, ents, x, logits, group, "ties", 0.0)


@pytest.mark.parametrize("m", [1, 2])
def test_gpt_oss_shaped_block(wq, m):
    d, inter, E, k, group, r = 2880, 2880, 32, 4, 64, 16
    logits = torch.from_numpy(np.random.default_rng(500 + m).standard_normal((m, E)).astype(np.float32))
    sel = set(int(e) for e in omoe.route(logits.numpy().astype(np.float64), k)[0].ravel())
    layer, ents = _build(wq, d, inter, E, k, group, r, 400, real=sel)
    x = synth.activations((m, d), 600 + m)
    _check_block(wq, layer, ents, x, logits, group, f"gpt-oss m={m}", 2.0)


def test_bad_arguments_are_refused(wq):
    d, inter, E, k, group = 256, 128, 4, 2, 64
    layer, _ = _build(wq, d, inter, E, k, group, 0, 700)
    x = synth.activations((1, d), 1).cuda()
    logits = torch.zeros((1, E), dtype=torch.float32, device="cuda")
    for bad in (wq.MoELayer(layer.experts, E, 0), wq.MoELayer(layer.experts, E, E + 1),
                wq.MoELayer(layer.experts, 3, 2)):
        with pytest.raises(wq.WQError):
            wq.moe_forward(x, logits, bad, ws=torch.zeros(1 << 20, dtype=torch.uint8, device="cuda"))
    ws = wq.moe_workspace(1, layer)
    with pytest.raises(wq.WQError):
        wq.moe_forward(x, logits, layer, ws=ws[:64])
