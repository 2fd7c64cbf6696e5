"""Pins for the oracle's IEEE conversions (binary16 and bfloat16 rounding).

Each conversion is checked against an implementation outside the oracle:
numpy's float16 cast, torch's bfloat16 cast (for values exactly representable
in fp32, where torch's cast is a single correct rounding), and an exact
rational-arithmetic rounding written here for fp64 inputs.
"""
from fractions import Fraction

import numpy as np
import pytest
import torch


def _edge_f32():
    vals = [0.0, -0.0, 1.0, -1.0, 65504.0, 65519.99, 65520.0, 70000.0, 6.1035156e-05,
            5.9604645e-08, 2.9802322e-08, 2.9802326e-08, 1e-10, 0.1, 1.0 / 3.0, 2049.0, 2051.0,
            -2049.0, 1025.5, 0.5 + 2 ** -12, np.inf, -np.inf]
    # exact ties between adjacent binary16 values in every binade
    for e in range(-24, 16):
        vals.append(2.0 ** e * (1 + 2 ** -11))
        vals.append(2.0 ** e * (1 + 3 * 2 ** -11))
    return np.array(vals, dtype=np.float32)


def test_f32_to_f16_matches_numpy(orc):
    rng = np.random.default_rng(1)
    a = np.concatenate([
        _edge_f32(),
        rng.standard_normal(200000).astype(np.float32) * np.float32(0.03),
        (rng.standard_normal(200000) * 1e4).astype(np.float32),
        (rng.standard_normal(50000) * 1e-6).astype(np.float32),
        rng.integers(0, 2 ** 32, 100000, dtype=np.uint64).astype(np.uint32).view(np.float32),
    ])
    a = a[~np.isnan(a)]
    got = orc.f32_to_f16_bits(a)
    with np.errstate(over="ignore"):
        want = a.astype(np.float16).view(np.uint16)
    np.testing.assert_array_equal(got, want)


def test_f16_to_f64_matches_numpy(orc):
    bits = np.arange(0, 1 << 16, dtype=np.uint32).astype(np.uint16)
    got = orc.f16_bits_to_f64(bits)
    want = bits.view(np.float16).astype(np.float64)
    both_nan = np.isnan(got) & np.isnan(want)
    np.testing.assert_array_equal(got[~both_nan], want[~both_nan])
    assert np.array_equal(np.isnan(got), np.isnan(want))


def test_bf16_roundtrip_all_patterns(orc):
    bits = np.arange(0, 1 << 16, dtype=np.uint32).astype(np.uint16)
    vals = orc.bf16_bits_to_f64(bits)
    want = torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).to(torch.float64).numpy()
    fin = ~np.isnan(want)
    np.testing.assert_array_equal(vals[fin], want[fin])
    back = orc.f64_to_bf16_bits(vals[fin])
    np.testing.assert_array_equal(back, bits[fin])


def test_f64_to_bf16_matches_torch_on_fp32_values(orc):
    rng = np.random.default_rng(2)
    a = np.concatenate([
        rng.standard_normal(300000).astype(np.float32),
        (rng.standard_normal(100000) * 1e30).astype(np.float32),
        rng.integers(0, 2 ** 32, 100000, dtype=np.uint64).astype(np.uint32).view(np.float32),
    ])
    a = a[np.isfinite(a)]
    got = orc.f64_to_bf16_bits(a.astype(np.float64))
    want = torch.from_numpy(a).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(got, want)


def _bf16_exact(v: float) -> int:
    """Round an fp64 value to bfloat16 with exact rational arithmetic (ties to even)."""
    if v == 0:
        return 0x8000 if np.signbit(v) else 0
    sign = 0x8000 if v < 0 else 0
    a = Fraction(abs(v))
    e = 0
    while a >= 2:
        a /= 2
        e += 1
    while a < 1:
        a *= 2
        e -= 1
    E = max(e, -126)
    scaled = Fraction(abs(v)) / Fraction(2) ** (E - 7)
    fl = scaled.numerator // scaled.denominator
    rem = scaled - fl
    if rem > Fraction(1, 2) or (rem == Fraction(1, 2) and fl % 2 == 1):
        fl += 1
    r = Fraction(fl) * Fraction(2) ** (E - 7)
    if r >= Fraction(2) ** 128:
        return sign | 0x7F80
    f = np.float32(float(r))
    return sign | int(f.view(np.uint32) >> 16)


def test_f64_to_bf16_exact_rounding_of_fp64_values(orc):
    # fp64 values near bf16 ties: a cast through fp32 would round twice.
    rng = np.random.default_rng(3)
    base = rng.standard_normal(2000)
    vals = list(base)
    for b in base[:500]:
        t = float(np.float32(b))
        vals += [t * (1 + 2.0 ** -9), t * (1 + 2.0 ** -9 + 2.0 ** -30), t * (1 + 2.0 ** -9 - 2.0 ** -30)]
    vals += [1 + 2.0 ** -8, 1 + 2.0 ** -8 + 2.0 ** -40, 1 + 3 * 2.0 ** -8, 1e-40, -3e-39, 3.4e38, 3.3961e38]
    vals = np.array(vals, dtype=np.float64)
    got = orc.f64_to_bf16_bits(vals)
    want = np.array([_bf16_exact(float(v)) for v in vals], dtype=np.uint16)
    np.testing.assert_array_equal(got, want)
