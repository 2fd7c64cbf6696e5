"""Pins for the oracle's decode step of a whole decoder layer (oracle/decoder.py).

The primitives are checked against library routines: the fp64 quantized
projection against numpy's matmul of the dequantized matrix, and the
per-head RMSNorm against torch's rms_norm.  The composition is checked by
reductions to oracles pinned elsewhere:
- the first token of an empty cache attends only to itself, so the stored
  attention output is its own bf16 value vector;
- a zero output projection leaves x unchanged, so the layer is the MLP block
  alone;
- the cache gains exactly one position per sequence.
"""
import numpy as np
import pytest
import torch

from oracle import decoder as dec


def _w(orc, rng, n, k, group, bits, std=0.02):
    return orc.quantize((rng.standard_normal((n, k)) * std).astype(np.float32), group, bits)[:3]


def _bits(a):
    t = torch.from_numpy(np.asarray(a, np.float64)).float().to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def _layer(orc, rng, d=256, H=4, Hkv=2, hd=64, inter=512):
    return dict(
        shape=dec.AttnShape(H, Hkv, hd),
        wq=_w(orc, rng, H * hd, d, 128, 4), wk=_w(orc, rng, Hkv * hd, d, 128, 4),
        wv=_w(orc, rng, Hkv * hd, d, 128, 4), wo=_w(orc, rng, d, H * hd, 128, 4), group_attn=128,
        gate=_w(orc, rng, inter, d, 64, 2), up=_w(orc, rng, inter, d, 64, 2), wd=_w(orc, rng, d, inter, 128, 4),
        group_gu=64, group_down=128)


def test_qproj_matches_numpy(orc):
    rng = np.random.default_rng(0)
    w = _w(orc, rng, 96, 256, 64, 4)
    x = rng.standard_normal((3, 256))
    np.testing.assert_allclose(orc.qproj(x, w, 64), x @ orc.dequant(*w, 64).T, rtol=1e-12, atol=1e-14)


def test_head_rms_norm_matches_torch(orc):
    rng = np.random.default_rng(1)
    x = rng.standard_normal((2, 4 * 64)) * 3.0
    want = torch.nn.functional.rms_norm(torch.from_numpy(x.reshape(2, 4, 64)), (64,), eps=1e-6).numpy()
    np.testing.assert_allclose(dec.head_rms_norm(x, 4, 64), want.reshape(2, 256), rtol=1e-12, atol=1e-14)


def test_first_token_attends_to_itself(orc):
    rng = np.random.default_rng(2)
    L = _layer(orc, rng)
    b, lmax, sh = 2, 8, L["shape"]
    x = _bits(rng.standard_normal((b, 256)))
    kc = np.zeros((b, sh.n_kv, lmax, sh.head_dim), np.uint16)
    out = dec.decoder_layer_decode(x, [0, 0], kc, kc.copy(), **L)
    rep = sh.n_heads // sh.n_kv
    for i in range(b):
        for h in range(sh.n_heads):
            got = out["o_bits"][i, h * sh.head_dim:(h + 1) * sh.head_dim]
            np.testing.assert_array_equal(got, out["v_cache"][i, h // rep, 0])


def test_zero_output_projection_leaves_the_mlp_block(orc):
    rng = np.random.default_rng(3)
    L = _layer(orc, rng)
    q, s, z = L["wo"]
    L["wo"] = (np.full_like(q, 5), s, np.full_like(z, np.float16(5.0).view(np.uint16)))  # s (5 - 5) = 0
    b, lmax, sh = 2, 8, L["shape"]
    x = _bits(rng.standard_normal((b, 256)))
    kc = _bits(rng.standard_normal((b, sh.n_kv, lmax, sh.head_dim)))
    out = dec.decoder_layer_decode(x, [3, 7], kc, kc.copy(), **L)
    np.testing.assert_array_equal(out["x1_bits"], x)
    _, h_bits = orc.gateup(x, L["gate"], L["up"], 64, prenorm=True)
    y, y_bits = orc.down(h_bits, L["wd"], 128, x)
    np.testing.assert_array_equal(out["y_bits"], y_bits)
    np.testing.assert_array_equal(out["y"], y)


@pytest.mark.parametrize("lens", [[0, 4], [7, 1]])
def test_cache_gains_one_position(orc, lens):
    rng = np.random.default_rng(4)
    L = _layer(orc, rng)
    b, lmax, sh = 2, 8, L["shape"]
    x = _bits(rng.standard_normal((b, 256)))
    kc = _bits(rng.standard_normal((b, sh.n_kv, lmax, sh.head_dim)))
    vc = _bits(rng.standard_normal((b, sh.n_kv, lmax, sh.head_dim)))
    out = dec.decoder_layer_decode(x, lens, kc, vc, **L)
    for i, n in enumerate(lens):
        for c0, c1 in ((kc, out["k_cache"]), (vc, out["v_cache"])):
            changed = np.any(c0[i] != c1[i], axis=(0, 2))
            assert not np.any(np.delete(changed, n))
    assert np.all(np.isfinite(out["y"]))


def _np_deq(w, group):
    q, s, z = w
    sf = np.repeat(s.view(np.float16).astype(np.float64), group, axis=1)
    zf = np.repeat(z.view(np.float16).astype(np.float64), group, axis=1)
    return sf * (q.astype(np.float64) - zf)


def _bf16_round(a):
    return torch.from_numpy(np.asarray(a, np.float64)).to(torch.bfloat16).double().numpy()


def _rope_complex(x, pos, theta):
    hd = x.shape[-1]
    half = hd // 2
    z = x[..., :half] + 1j * x[..., half:]
    z = z * np.exp(1j * pos * theta ** (-2.0 * np.arange(half) / hd))
    return np.concatenate([z.real, z.imag], axis=-1)


def test_attention_path_matches_library_steps(orc):
    """Steps 1-8 rebuilt from library routines only (numpy matmul of numpy-
    dequantized matrices, torch rms_norm, complex RoPE, torch fp64 attention):
    the appended key and value, the attention output and x1 must agree with
    the composition over several cached positions."""
    rng = np.random.default_rng(5)
    L = _layer(orc, rng)
    sh = L["shape"]
    H, Hkv, hd = sh.n_heads, sh.n_kv, sh.head_dim
    b, lmax, lens = 2, 9, [4, 8]
    x = _bits(rng.standard_normal((b, 256)))
    kc = _bits(rng.standard_normal((b, Hkv, lmax, hd)))
    vc = _bits(rng.standard_normal((b, Hkv, lmax, hd)))
    out = dec.decoder_layer_decode(x, lens, kc, vc, **L)

    xf = torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).view(torch.bfloat16).double()
    xin = torch.nn.functional.rms_norm(xf, (256,), eps=1e-6).numpy()
    q = xin @ _np_deq(L["wq"], 128).T
    k = xin @ _np_deq(L["wk"], 128).T
    v = xin @ _np_deq(L["wv"], 128).T
    norm = lambda a, n: torch.nn.functional.rms_norm(torch.from_numpy(a.reshape(b, n, hd)), (hd,), eps=1e-6).numpy()
    q, k = norm(q, H), norm(k, Hkv)
    for i in range(b):
        q[i] = _rope_complex(q[i], lens[i], sh.theta)
        k[i] = _rope_complex(k[i], lens[i], sh.theta)
    kf = torch.from_numpy(np.ascontiguousarray(kc).view(np.int16)).view(torch.bfloat16).double().numpy().copy()
    vf = torch.from_numpy(np.ascontiguousarray(vc).view(np.int16)).view(torch.bfloat16).double().numpy().copy()
    x1 = np.empty((b, 256))
    for i in range(b):
        kf[i, :, lens[i]] = _bf16_round(k[i])
        vf[i, :, lens[i]] = _bf16_round(v[i].reshape(Hkv, hd))
        n = lens[i] + 1
        kt = torch.from_numpy(kf[i, :, :n]).repeat_interleave(H // Hkv, dim=0)
        vt = torch.from_numpy(vf[i, :, :n]).repeat_interleave(H // Hkv, dim=0)
        o = torch.nn.functional.scaled_dot_product_attention(torch.from_numpy(q[i][:, None, :]), kt, vt)[:, 0]
        o = _bf16_round(o.numpy().reshape(H * hd))
        got_o = torch.from_numpy(out["o_bits"][i].view(np.int16)).view(torch.bfloat16).double().numpy()
        np.testing.assert_allclose(got_o, o, rtol=2.0 ** -7, atol=1e-12)       # at most one bf16 rounding flip
        assert np.mean(got_o == o) > 0.95
        x1[i] = xf[i].numpy() + got_o @ _np_deq(L["wo"], 128).T
    got_k = torch.from_numpy(out["k_cache"].view(np.int16)).view(torch.bfloat16).double().numpy()
    got_v = torch.from_numpy(out["v_cache"].view(np.int16)).view(torch.bfloat16).double().numpy()
    for i in range(b):
        np.testing.assert_allclose(got_k[i, :, lens[i]], kf[i, :, lens[i]], rtol=2.0 ** -7, atol=1e-12)
        np.testing.assert_allclose(got_v[i, :, lens[i]], vf[i, :, lens[i]], rtol=2.0 ** -7, atol=1e-12)
        assert np.mean(got_k[i, :, lens[i]] == kf[i, :, lens[i]]) > 0.95
    got_x1 = torch.from_numpy(out["x1_bits"].view(np.int16)).view(torch.bfloat16).double().numpy()
    np.testing.assert_allclose(got_x1, _bf16_round(x1), rtol=2.0 ** -7, atol=1e-12)
