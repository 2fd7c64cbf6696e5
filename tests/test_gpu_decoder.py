"""One decode step of a decoder layer on the GPU vs the oracle.

The stages run through the C ABI one by one and are checked teacher-forced:
the 4-bit qkv projection (fp32 output), the attention step (RMSNorm scale,
per-head q/k norm, RoPE, bf16 cache append, grouped-query softmax attention)
fed with the GPU's own projections, the output projection with the residual,
then the MLP block.  The composite call wq_decoder_layer_forward is checked
end to end against the oracle's decoder layer.  Cache entries past the new
position hold NaN: reading one would show.  Shapes: a small layer, the
Qwen3-4B attention (32 query heads, 8 kv heads, head_dim 128) at contexts
of 1000 and 4096, a context long enough for ~150 splits, 1 and 8 query heads
per kv head, and the first token of an empty cache.
"""
import numpy as np
import pytest
import torch

import oracle as orc
from oracle import decoder as odec
from paper_2606_04238_gb300 import synth
from tests.gpu_util import check_bf16, check_f32, upload_packed

pytestmark = pytest.mark.gpu

NAN_BF16 = 0x7FC0


@pytest.fixture(scope="module")
def wq():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2606_04238_gb300 import wq as mod
    return mod


def _q(shape, group, bits, seed):
    w = (np.random.default_rng(seed).standard_normal(shape) * 0.02).astype(np.float32)
    return orc.quantize(w, group, bits)[:3]


def _cat(*ws):
    return tuple(np.concatenate([w[i] for w in ws], axis=0) for i in range(3))


def _build(wq, d, inter, H, Hkv, hd, g_attn, g_mlp, r, seed, bits_gu=2):
    wqm, wkm, wvm = _q((H * hd, d), g_attn, 4, seed), _q((Hkv * hd, d), g_attn, 4, seed + 1), _q((Hkv * hd, d), g_attn, 4, seed + 2)
    wom = _q((d, H * hd), g_attn, 4, seed + 3)
    gate, up, wd = _q((inter, d), g_mlp, bits_gu, seed + 4), _q((inter, d), g_mlp, bits_gu, seed + 5), _q((d, inter), g_mlp, 4, seed + 6)
    kw, lora = {}, None
    if r:
        a, bg, bu = synth.lora(d, inter, r, seed + 7)
        kw = dict(lora_a=a.cuda(), lora_b_gate=bg.cuda(), lora_b_up=bu.cuda(), lora_scale=2.0)
        lora = (synth.bf16_bits(a), synth.bf16_bits(bg), synth.bf16_bits(bu))
    mlp = wq.MLPLayer(upload_packed(*gate, g_mlp, bits_gu), upload_packed(*up, g_mlp, bits_gu), upload_packed(*wd, g_mlp, 4), **kw)
    layer = wq.DecoderLayer(upload_packed(*_cat(wqm, wkm, wvm), g_attn, 4), upload_packed(*wom, g_attn, 4), mlp, H, Hkv, hd)
    ora = dict(wq=wqm, wk=wkm, wv=wvm, wo=wom, gate=gate, up=up, wd=wd, lora=lora)
    return layer, ora


def _caches(B, Hkv, max_len, hd, lens, seed):
    rng = np.random.default_rng(seed)
    kc = np.full((B, Hkv, max_len, hd), NAN_BF16, np.uint16)
    vc = np.full((B, Hkv, max_len, hd), NAN_BF16, np.uint16)
    for b, n in enumerate(lens):
        kc[b, :, :n] = orc.f64_to_bf16_bits(rng.standard_normal((Hkv, n, hd)))
        vc[b, :, :n] = orc.f64_to_bf16_bits(rng.standard_normal((Hkv, n, hd)))
    return kc, vc


def _dev(bits):
    return synth.from_bf16_bits(bits, device="cuda")


def _attn_from_qkv(qkv, x_bits, lens, kc, vc, H, Hkv, hd, theta):
    """Steps 3-7 of the oracle's decoder layer, fed with the GPU's fp32 projections (before the RMSNorm scale)."""
    B = x_bits.shape[0]
    rs = orc.rms_scale(x_bits)[:, None]
    qkv = np.asarray(qkv, np.float64) * rs
    q, k, v = qkv[:, :H * hd], qkv[:, H * hd:(H + Hkv) * hd], qkv[:, (H + Hkv) * hd:]
    q = odec.head_rms_norm(q, H, hd)
    k = odec.head_rms_norm(k, Hkv, hd)
    q = np.stack([orc.rope(q[i].reshape(H, hd), int(lens[i]), theta) for i in range(B)])
    k = np.stack([orc.rope(k[i].reshape(Hkv, hd), int(lens[i]), theta) for i in range(B)])
    kc, vc = kc.copy(), vc.copy()
    k_new, v_new = np.empty((B, Hkv, hd)), np.empty((B, Hkv, hd))
    for i in range(B):
        k_new[i] = k[i]
        v_new[i] = v[i].reshape(Hkv, hd)
        kc[i, :, lens[i]] = orc.f64_to_bf16_bits(k[i])
        vc[i, :, lens[i]] = orc.f64_to_bf16_bits(v[i].reshape(Hkv, hd))
    o = orc.attn_decode(q, kc, vc, np.asarray(lens) + 1)
    return o.reshape(B, H * hd), k_new, v_new


def _stages(wq, layer, ora, d, inter, H, Hkv, hd, g_attn, g_mlp, B, lens, max_len, seed, what):
    x = synth.activations((B, d), seed)
    x_bits = synth.bf16_bits(x)
    kc, vc = _caches(B, Hkv, max_len, hd, lens, seed + 1)
    kd, vd = _dev(kc), _dev(vc)
    lens_d = torch.tensor(lens, dtype=torch.int32, device="cuda")
    xd = x.cuda()
    qkv = wq.down_w4(xd, layer.qkv, out_f32=True)
    o = wq.attn_decode(qkv, xd, lens_d, kd, vd, H, Hkv, layer.rope_theta)
    x1 = wq.down_w4(o, layer.o, residual=xd)
    torch.cuda.synchronize()
    assert wq.device_status() == 0
    # projection (fp32 output against the fp64 product of the unscaled input)
    ref_qkv = orc.qproj(orc.bf16_bits_to_f64(x_bits), _cat(ora["wq"], ora["wk"], ora["wv"]), g_attn)
    check_f32(qkv, ref_qkv, f"{what} qkv projection")
    # attention from the GPU's projections
    o_ref, k_new, v_new = _attn_from_qkv(qkv.cpu().numpy(), x_bits, lens, kc, vc, H, Hkv, hd, layer.rope_theta)
    check_bf16(o, o_ref, f"{what} attention output")
    kd_h, vd_h = synth.bf16_bits(kd), synth.bf16_bits(vd)
    for i, n in enumerate(lens):
        check_bf16(kd[i, :, n], k_new[i], f"{what} appended k, sequence {i}")
        check_bf16(vd[i, :, n], v_new[i], f"{what} appended v, sequence {i}")
        assert np.array_equal(kd_h[i, :, :n], kc[i, :, :n]) and np.array_equal(vd_h[i, :, :n], vc[i, :, :n])
        assert np.all(kd_h[i, :, n + 1:] == NAN_BF16) and np.all(vd_h[i, :, n + 1:] == NAN_BF16)
    # output projection with the residual, from the GPU's o
    x1_ref, _ = orc.down(synth.bf16_bits(o), ora["wo"], g_attn, x_bits)
    check_bf16(x1, x1_ref, f"{what} x1")
    return x, kc, vc


@pytest.mark.parametrize("lens", [[0, 5, 40], [63, 1, 17]])
def test_small_decoder_stages(wq, lens):
    d, inter, H, Hkv, hd = 256, 768, 4, 2, 64
    layer, ora = _build(wq, d, inter, H, Hkv, hd, 64, 64, 8, 11)
    _stages(wq, layer, ora, d, inter, H, Hkv, hd, 64, 64, len(lens), lens, 64, 21, f"small lens={lens}")


@pytest.mark.parametrize("H,Hkv", [(4, 4), (16, 2)])
def test_heads_per_kv_head(wq, H, Hkv):
    d, inter, hd = 512, 1024, 128
    layer, ora = _build(wq, d, inter, H, Hkv, hd, 128, 128, 0, 31)
    _stages(wq, layer, ora, d, inter, H, Hkv, hd, 128, 128, 2, [7, 300], 512, 41, f"H={H} Hkv={Hkv}")


def test_qwen3_4b_attention(wq):
    cfg = synth.CONFIGS["qwen3_4b"]
    H, Hkv, hd = 32, 8, 128
    layer, ora = _build(wq, cfg.d, cfg.inter, H, Hkv, hd, 128, 128, 16, 51)
    _stages(wq, layer, ora, cfg.d, cfg.inter, H, Hkv, hd, 128, 128, 2, [1000, 4095], 4096, 61, "qwen3_4b")


def test_long_context_splits(wq):
    d, inter, H, Hkv, hd = 512, 1024, 8, 2, 128
    layer, ora = _build(wq, d, inter, H, Hkv, hd, 128, 128, 0, 71)
    _stages(wq, layer, ora, d, inter, H, Hkv, hd, 128, 128, 1, [20000], 20480, 81, "long context")


def test_decoder_layer_end_to_end(wq):
    d, inter, H, Hkv, hd = 512, 1024, 8, 2, 64
    layer, ora = _build(wq, d, inter, H, Hkv, hd, 64, 64, 8, 91)
    lens, max_len = [3, 100], 128
    x = synth.activations((2, d), 101)
    kc, vc = _caches(2, Hkv, max_len, hd, lens, 102)
    kd, vd = _dev(kc), _dev(vc)
    y = wq.decoder_layer_forward(x.cuda(), torch.tensor(lens, dtype=torch.int32, device="cuda"), layer, kd, vd)
    torch.cuda.synchronize()
    assert wq.device_status() == 0
    ref = odec.decoder_layer_decode(synth.bf16_bits(x), lens, kc, vc, odec.AttnShape(H, Hkv, hd, layer.rope_theta),
                                    ora["wq"], ora["wk"], ora["wv"], ora["wo"], 64, ora["gate"], ora["up"], ora["wd"],
                                    64, 64, lora=ora["lora"], lora_scale=2.0)
    # several bf16 roundings (o, x1, h) between the input and y: the bound of a depth-3 chain
    check_bf16(y, ref["y"], "decoder layer y", min_exact=0.5, depth=3)
    for i, n in enumerate(lens):
        check_bf16(kd[i, :, n], orc.bf16_bits_to_f64(ref["k_cache"][i, :, n]), f"cache k, sequence {i}", min_exact=0.9)


@pytest.mark.parametrize("lora", [True, False])
def test_qwen3_4b_decoder_layer_end_to_end(wq, lora):
    """The composite call at the Qwen3-4B shape, where the output projection
    hands the MLP its input's tile partials and gate/up hands down the ready
    binary16 panel of h (the decode route of the benchmark's decoder leg)."""
    cfg = synth.CONFIGS["qwen3_4b"]
    H, Hkv, hd = 32, 8, 128
    layer, ora = _build(wq, cfg.d, cfg.inter, H, Hkv, hd, 128, 128, 16 if lora else 0, 111)
    lens, max_len = [1000], 1024
    x = synth.activations((1, cfg.d), 112)
    kc, vc = _caches(1, Hkv, max_len, hd, lens, 113)
    kd, vd = _dev(kc), _dev(vc)
    y = wq.decoder_layer_forward(x.cuda(), torch.tensor(lens, dtype=torch.int32, device="cuda"), layer, kd, vd)
    torch.cuda.synchronize()
    assert wq.device_status() == 0
    ref = odec.decoder_layer_decode(synth.bf16_bits(x), lens, kc, vc, odec.AttnShape(H, Hkv, hd, layer.rope_theta),
                                    ora["wq"], ora["wk"], ora["wv"], ora["wo"], 128, ora["gate"], ora["up"], ora["wd"],
                                    128, 128, lora=ora["lora"], lora_scale=2.0)
    check_bf16(y, ref["y"], "qwen3_4b decoder layer y", min_exact=0.5, depth=3)


def test_length_outside_the_cache_is_refused_on_the_device(wq):
    d, H, Hkv, hd, max_len = 256, 4, 2, 64, 16
    x = synth.activations((1, d), 5).cuda()
    qkv = torch.zeros((1, (H + 2 * Hkv) * hd), dtype=torch.float32, device="cuda")
    kc = torch.zeros((1, Hkv, max_len, hd), dtype=torch.bfloat16, device="cuda")
    vc = torch.zeros_like(kc)
    wq.attn_decode(qkv, x, torch.tensor([max_len], dtype=torch.int32, device="cuda"), kc, vc, H, Hkv, 1e6)
    torch.cuda.synchronize()
    assert wq.device_status() == -1
    assert wq.device_status() == 0  # read and cleared
    assert torch.count_nonzero(kc).item() == 0
