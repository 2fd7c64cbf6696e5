"""Pins for the oracle's decode-step attention and rotary embedding (the rest
of a decoder layer around the MLP block; Sec. 5 counts the KV-cache reads
among the operators whose cost does not depend on the weight precision).

Checked against independent formulations:
- torch's scaled_dot_product_attention in fp64, with the key/value heads
  expanded by repeat_interleave;
- closed forms: one cached position returns V exactly, identical keys give
  the mean of V;
- cache entries past a sequence's length are never read;
- RoPE against complex multiplication by e^{i a}, plus norm preservation,
  the relative-position property and the identity at position 0.
"""
import numpy as np
import pytest
import torch


def _bf16_bits(a):
    t = torch.from_numpy(np.asarray(a, np.float64)).float().to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def _bf16_f64(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).double().numpy()


def _case(rng, b, h, hkv, hd, lmax):
    q = rng.standard_normal((b, h, hd))
    k = _bf16_bits(rng.standard_normal((b, hkv, lmax, hd)))
    v = _bf16_bits(rng.standard_normal((b, hkv, lmax, hd)))
    return q, k, v


@pytest.mark.parametrize("b,h,hkv,hd,lmax", [(2, 8, 2, 64, 40), (3, 4, 4, 32, 17), (1, 32, 8, 128, 300)])
def test_attn_matches_torch_sdpa(orc, b, h, hkv, hd, lmax):
    rng = np.random.default_rng(b * 100 + h + lmax)
    q, k, v = _case(rng, b, h, hkv, hd, lmax)
    lens = rng.integers(1, lmax + 1, size=b)
    lens[0] = lmax
    o = orc.attn_decode(q, k, v, lens)
    kf, vf = _bf16_f64(k), _bf16_f64(v)
    for i in range(b):
        L = int(lens[i])
        qt = torch.from_numpy(q[i][:, None, :])                                        # [H, 1, hd]
        kt = torch.from_numpy(kf[i, :, :L]).repeat_interleave(h // hkv, dim=0)        # [H, L, hd]
        vt = torch.from_numpy(vf[i, :, :L]).repeat_interleave(h // hkv, dim=0)
        want = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt)[:, 0].numpy()
        np.testing.assert_allclose(o[i], want, rtol=1e-12, atol=1e-13)


def test_one_position_returns_v(orc):
    rng = np.random.default_rng(1)
    q, k, v = _case(rng, 2, 4, 2, 16, 8)
    o = orc.attn_decode(q, k, v, [1, 1])
    vf = _bf16_f64(v)
    for i in range(2):
        for hh in range(4):
            np.testing.assert_array_equal(o[i, hh], vf[i, hh // 2, 0])


def test_identical_keys_average_v(orc):
    rng = np.random.default_rng(2)
    b, h, hkv, hd, lmax = 1, 2, 1, 32, 11
    q, k, v = _case(rng, b, h, hkv, hd, lmax)
    k[:] = k[:, :, :1]  # every position holds the same key
    o = orc.attn_decode(q, k, v, [lmax])
    want = _bf16_f64(v)[0, 0].mean(axis=0)
    for hh in range(h):
        np.testing.assert_allclose(o[0, hh], want, rtol=1e-13, atol=1e-14)


def test_positions_past_the_length_are_not_read(orc):
    rng = np.random.default_rng(3)
    q, k, v = _case(rng, 2, 4, 2, 16, 12)
    lens = [5, 9]
    o = orc.attn_decode(q, k, v, lens)
    k2, v2 = k.copy(), v.copy()
    for i, L in enumerate(lens):
        k2[i, :, L:] = 0x7FC0  # NaN patterns past the length
        v2[i, :, L:] = 0x7FC0
    np.testing.assert_array_equal(orc.attn_decode(q, k2, v2, lens), o)


@pytest.mark.parametrize("hd,theta", [(64, 1e4), (128, 1e6)])
def test_rope_matches_complex_rotation(orc, hd, theta):
    rng = np.random.default_rng(hd)
    x = rng.standard_normal((3, hd))
    pos = 1234
    got = orc.rope(x, pos, theta)
    half = hd // 2
    z = x[:, :half] + 1j * x[:, half:]
    ang = pos * theta ** (-2.0 * np.arange(half) / hd)
    zr = z * np.exp(1j * ang)
    np.testing.assert_allclose(got, np.concatenate([zr.real, zr.imag], axis=1), rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(np.linalg.norm(got, axis=1), np.linalg.norm(x, axis=1), rtol=1e-13)
    np.testing.assert_array_equal(orc.rope(x, 0, theta), x)


def test_rope_scores_depend_on_relative_position(orc):
    rng = np.random.default_rng(9)
    q, k = rng.standard_normal((1, 64)), rng.standard_normal((1, 64))
    base = (orc.rope(q, 30, 1e6) * orc.rope(k, 7, 1e6)).sum()
    for shift in (1, 100, 5000):
        moved = (orc.rope(q, 30 + shift, 1e6) * orc.rope(k, 7 + shift, 1e6)).sum()
        assert abs(moved - base) < 1e-9 * (1 + abs(base))


def test_attention_rejects_bad_arguments(orc):
    rng = np.random.default_rng(4)
    q, k, v = _case(rng, 1, 6, 4, 16, 8)   # 6 query heads over 4 key/value heads
    with pytest.raises(ValueError):
        orc.attn_decode(q, k, v, [3])
    q, k, v = _case(rng, 1, 4, 2, 16, 8)
    for lens in ([0], [9]):
        with pytest.raises(ValueError):
            orc.attn_decode(q, k, v, lens)
    with pytest.raises(ValueError):
        orc.rope(np.zeros((1, 15)), 3, 1e4)
