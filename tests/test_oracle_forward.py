"""Pins for the oracle's forward pass (Eq. 1 LoRA, Sec. 3.3 gated MLP).

Checked against library routines and closed forms: numpy fp64 matmul of a
dequantized matrix written out independently, torch's fp64 SiLU and RMSNorm,
the LoRA-zero and B = 0 special cases, and a rank-1 closed form.
"""
import numpy as np
import pytest
import torch


def _np_deq(q, s_bits, z_bits, group):
    s = np.repeat(s_bits.view(np.float16).astype(np.float64), group, axis=1)
    z = np.repeat(z_bits.view(np.float16).astype(np.float64), group, axis=1)
    return s * (q.astype(np.float64) - z)


def _bf16_to_f64(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).double().numpy()


def _rand_bf16(rng, shape, std=1.0):
    t = torch.from_numpy(rng.standard_normal(shape) * std).float().to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def _layer(orc, rng, d, inter, group_gu, group_d, bits_gu=2):
    wg = (rng.standard_normal((inter, d)) * 0.02).astype(np.float32)
    wu = (rng.standard_normal((inter, d)) * 0.02).astype(np.float32)
    wd = (rng.standard_normal((d, inter)) * 0.02).astype(np.float32)
    g = orc.quantize(wg, group_gu, bits_gu)[:3]
    u = orc.quantize(wu, group_gu, bits_gu)[:3]
    dn = orc.quantize(wd, group_d, 4)[:3] if inter % group_d == 0 else None
    return g, u, dn


def test_dequant_matches_numpy(orc):
    rng = np.random.default_rng(0)
    w = (rng.standard_normal((40, 256)) * 0.02).astype(np.float32)
    q, s, z, _ = orc.quantize(w, 64, 2)
    np.testing.assert_array_equal(orc.dequant(q, s, z, 64), _np_deq(q, s, z, 64))


@pytest.mark.parametrize("m", [1, 3])
def test_gateup_no_lora_matches_numpy_matmul(orc, m):
    rng = np.random.default_rng(m)
    d, inter = 256, 96
    g, u, _ = _layer(orc, rng, d, inter, 64, 64)
    x = _rand_bf16(rng, (m, d))
    h, hb = orc.gateup(x, g, u, 64)
    xf = _bf16_to_f64(x)
    gg = xf @ _np_deq(*g, 64).T
    uu = xf @ _np_deq(*u, 64).T
    want = torch.nn.functional.silu(torch.from_numpy(gg)).numpy() * uu
    np.testing.assert_allclose(h, want, rtol=1e-12, atol=1e-14)
    # the bf16 output is the round-to-nearest of the fp64 value
    np.testing.assert_array_equal(hb, orc.f64_to_bf16_bits(h))


def test_lora_special_cases(orc):
    rng = np.random.default_rng(3)
    d, inter, r = 256, 80, 8
    g, u, _ = _layer(orc, rng, d, inter, 128, 128)
    x = _rand_bf16(rng, (2, d))
    a = _rand_bf16(rng, (2 * r, d), 0.01)
    bg = _rand_bf16(rng, (inter, r), 0.01)
    bu = _rand_bf16(rng, (inter, r), 0.01)
    base, _ = orc.gateup(x, g, u, 128)
    h0, _ = orc.gateup(x, g, u, 128, a, bg, bu, lora_scale=0.0)
    np.testing.assert_array_equal(h0, base)
    zeros = np.zeros_like(bg)
    hz, _ = orc.gateup(x, g, u, 128, a, zeros, zeros, lora_scale=2.0)
    np.testing.assert_array_equal(hz, base)
    h1, _ = orc.gateup(x, g, u, 128, a, bg, bu, lora_scale=2.0)
    assert np.max(np.abs(h1 - base)) > 1e-6


def test_lora_rank1_closed_form(orc):
    # r = 1: g = x Wg^T + alpha (x . a_g) b_g, u likewise.
    rng = np.random.default_rng(4)
    d, inter = 128, 48
    g, u, _ = _layer(orc, rng, d, inter, 64, 64)
    x = _rand_bf16(rng, (1, d))
    a = _rand_bf16(rng, (2, d), 0.1)
    bg = _rand_bf16(rng, (inter, 1), 0.1)
    bu = _rand_bf16(rng, (inter, 1), 0.1)
    alpha = 1.75
    h, _ = orc.gateup(x, g, u, 64, a, bg, bu, lora_scale=alpha)
    xf, af = _bf16_to_f64(x)[0], _bf16_to_f64(a)
    gg = _np_deq(*g, 64) @ xf + alpha * (xf @ af[0]) * _bf16_to_f64(bg)[:, 0]
    uu = _np_deq(*u, 64) @ xf + alpha * (xf @ af[1]) * _bf16_to_f64(bu)[:, 0]
    want = gg / (1 + np.exp(-gg)) * uu
    np.testing.assert_allclose(h[0], want, rtol=1e-12, atol=1e-14)


@pytest.mark.parametrize("prenorm", [False, True])
def test_lora_rank8_matches_numpy_matmul(orc, prenorm):
    # Eq. 1 on both projections with numpy matmuls as the steps:
    #   g = xin Wg^T + alpha (xin A_g^T) B_g^T,  u likewise,  h = SiLU(g) u.
    # A rank above 1 with inter != r != d separates every index of A and B.
    rng = np.random.default_rng(9)
    d, inter, r, m = 192, 72, 8, 3
    g, u, _ = _layer(orc, rng, d, inter, 64, 64)
    x = _rand_bf16(rng, (m, d))
    a = _rand_bf16(rng, (2 * r, d), 0.05)
    bg = _rand_bf16(rng, (inter, r), 0.05)
    bu = _rand_bf16(rng, (inter, r), 0.05)
    alpha = 2.0
    h, _ = orc.gateup(x, g, u, 64, a, bg, bu, lora_scale=alpha, prenorm=prenorm)
    xf = _bf16_to_f64(x)
    if prenorm:
        xf = xf / np.sqrt(np.mean(xf * xf, axis=1, keepdims=True) + 1e-6)
    af = _bf16_to_f64(a)
    gg = xf @ _np_deq(*g, 64).T + alpha * (xf @ af[:r].T) @ _bf16_to_f64(bg).T
    uu = xf @ _np_deq(*u, 64).T + alpha * (xf @ af[r:].T) @ _bf16_to_f64(bu).T
    want = torch.nn.functional.silu(torch.from_numpy(gg)).numpy() * uu
    np.testing.assert_allclose(h, want, rtol=1e-11, atol=1e-13)


def test_rms_scale_matches_torch_rms_norm(orc):
    rng = np.random.default_rng(5)
    x = _rand_bf16(rng, (4, 512), 3.0)
    rs = orc.rms_scale(x)
    xf = _bf16_to_f64(x)
    want = torch.nn.functional.rms_norm(torch.from_numpy(xf), (512,), eps=1e-6).numpy()
    # the normalized input is used unrounded: x * rs equals torch's fp64 RMSNorm
    np.testing.assert_allclose(xf * rs[:, None], want, rtol=1e-13, atol=0)


def test_gateup_prenorm_is_scale_invariant(orc):
    # with eps = 0, RMSNorm(2^k x) = RMSNorm(x) exactly (powers of two scale
    # bf16 values, sums of squares and square roots without rounding), so the
    # whole gate/up output must be bit-identical; a dropped or misplaced
    # normalization breaks this
    rng = np.random.default_rng(6)
    d, inter = 256, 64
    g, u, _ = _layer(orc, rng, d, inter, 64, 64)
    a = _rand_bf16(rng, (2, d), 0.1)
    bg = _rand_bf16(rng, (inter, 1), 0.1)
    bu = _rand_bf16(rng, (inter, 1), 0.1)
    x = _rand_bf16(rng, (2, d), 5.0)
    x4 = torch.from_numpy(_bf16_to_f64(x) * 4.0).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    h1, _ = orc.gateup(x, g, u, 64, a, bg, bu, lora_scale=1.5, prenorm=True, eps=0.0)
    h2, _ = orc.gateup(x4, g, u, 64, a, bg, bu, lora_scale=1.5, prenorm=True, eps=0.0)
    np.testing.assert_array_equal(h1, h2)
    h0, _ = orc.gateup(x, g, u, 64, a, bg, bu, lora_scale=1.5, prenorm=False)
    assert not np.allclose(h0, h1)


def test_gateup_prenorm_matches_numpy(orc):
    rng = np.random.default_rng(16)
    d, inter = 256, 48
    g, u, _ = _layer(orc, rng, d, inter, 64, 64)
    a = _rand_bf16(rng, (2, d), 0.1)
    bg = _rand_bf16(rng, (inter, 1), 0.1)
    bu = _rand_bf16(rng, (inter, 1), 0.1)
    x = _rand_bf16(rng, (3, d), 2.0)
    h, _ = orc.gateup(x, g, u, 64, a, bg, bu, lora_scale=0.75, prenorm=True)
    xf, af = _bf16_to_f64(x), _bf16_to_f64(a)
    xn = xf / np.sqrt((xf * xf).mean(axis=1, keepdims=True) + 1e-6)
    gg = xn @ _np_deq(*g, 64).T + 0.75 * (xn @ af[0])[:, None] * _bf16_to_f64(bg)[:, 0][None, :]
    uu = xn @ _np_deq(*u, 64).T + 0.75 * (xn @ af[1])[:, None] * _bf16_to_f64(bu)[:, 0][None, :]
    want = gg / (1 + np.exp(-gg)) * uu
    np.testing.assert_allclose(h, want, rtol=1e-11, atol=1e-13)


def test_down_with_residual_matches_numpy(orc):
    rng = np.random.default_rng(7)
    d, inter = 96, 256
    wd = (rng.standard_normal((d, inter)) * 0.02).astype(np.float32)
    dn = orc.quantize(wd, 64, 4)[:3]
    h = _rand_bf16(rng, (3, inter))
    res = _rand_bf16(rng, (3, d))
    y, yb = orc.down(h, dn, 64, res)
    want = _bf16_to_f64(res) + _bf16_to_f64(h) @ _np_deq(*dn, 64).T
    np.testing.assert_allclose(y, want, rtol=1e-12, atol=1e-13)
    y0, _ = orc.down(h, dn, 64, None)
    np.testing.assert_allclose(y0, _bf16_to_f64(h) @ _np_deq(*dn, 64).T, rtol=1e-12, atol=1e-13)
    np.testing.assert_array_equal(yb, orc.f64_to_bf16_bits(y))


def test_empty_token_batch(orc):
    rng = np.random.default_rng(8)
    g, u, dn = _layer(orc, rng, 128, 64, 64, 64)
    x = np.zeros((0, 128), np.uint16)
    h, hb = orc.gateup(x, g, u, 64)
    assert h.shape == (0, 64)
    y, _ = orc.down(hb, dn, 64, x)
    assert y.shape == (0, 128)


def _grid_bf16(rng, shape, lim=255, exp=-8):
    """bf16 bit patterns of m * 2^exp, |m| <= lim < 256 (exact in bf16; fp64 sums of their products are exact)."""
    v = rng.integers(-lim, lim + 1, size=shape).astype(np.float32) * np.float32(2.0 ** exp)
    return (v.view(np.uint32) >> 16).astype(np.uint16)


def test_down_bf16_matches_numpy(orc):
    """BF16/W2-GateUp down layer (Sec. 6.1): y = residual + h Wd^T with a bf16 Wd."""
    rng = np.random.default_rng(17)
    d, inter, m = 80, 384, 5
    h, wd, res = _grid_bf16(rng, (m, inter)), _grid_bf16(rng, (d, inter), exp=-12), _grid_bf16(rng, (m, d))
    y, yb = orc.down_bf16(h, wd, res)
    want = _bf16_to_f64(res) + _bf16_to_f64(h) @ _bf16_to_f64(wd).T  # every sum exact: equal bit for bit
    np.testing.assert_array_equal(y, want)
    np.testing.assert_array_equal(yb, orc.f64_to_bf16_bits(y))
    y0, _ = orc.down_bf16(h, wd, None)
    np.testing.assert_array_equal(y0, _bf16_to_f64(h) @ _bf16_to_f64(wd).T)
    hg, wg = _rand_bf16(rng, (3, inter)), _rand_bf16(rng, (d, inter), 0.02)
    yg, _ = orc.down_bf16(hg, wg, None)
    np.testing.assert_allclose(yg, _bf16_to_f64(hg) @ _bf16_to_f64(wg).T, rtol=1e-12, atol=1e-13)


def test_down_bf16_agrees_with_the_4bit_down_on_bf16_exact_weights(orc):
    """A 4-bit matrix whose dequantized values bf16 holds exactly (scale 2^-6,
    q - z in [-15, 15]) gives the same y through both down definitions."""
    rng = np.random.default_rng(18)
    d, inter, group, m = 48, 256, 64, 4
    q = rng.integers(0, 16, size=(d, inter)).astype(np.uint8)
    s = np.full((d, inter // group), np.float16(2.0 ** -6)).view(np.uint16)
    z = rng.integers(0, 16, size=(d, inter // group)).astype(np.float16).view(np.uint16)
    deq = _np_deq(q, s, z, group)
    wd = (deq.astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)
    assert np.array_equal(_bf16_to_f64(wd), deq)
    h, res = _rand_bf16(rng, (m, inter)), _rand_bf16(rng, (m, d))
    y4, _ = orc.down(h, (q, s, z), group, res)
    y16, _ = orc.down_bf16(h, wd, res)
    np.testing.assert_allclose(y16, y4, rtol=1e-13, atol=1e-14)


def test_down_bf16_empty_and_bad_args(orc):
    y, yb = orc.down_bf16(np.zeros((0, 64), np.uint16), np.zeros((32, 64), np.uint16))
    assert y.shape == (0, 32) and yb.shape == (0, 32)
    with pytest.raises(AssertionError):
        orc.down_bf16(np.zeros((1, 64), np.uint16), np.zeros((32, 48), np.uint16))
