"""Pins for the oracle's Stage-1 quantizer (Sec. 4.1 / Sec. 3.3 bit-widths).

The quantizer reading (asymmetric min-max RTN per group, fp16 scale and zero)
is checked against: hand-worked examples (tests/golden), an independent numpy
float32 brute force, the exact-grid closed form, and the rounding bound
|w - deq(w)| <= s/2 inside the clamp range.
"""
import json
import os

import numpy as np
import pytest

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "quant_worked_examples.json")


def np_quantize(w, group, bits):
    """Independent float32 brute force of the same reading (numpy casts and rint)."""
    w = np.asarray(w, np.float32)
    qmax = np.float32(2 ** bits - 1)
    n, k = w.shape
    wg = w.reshape(n, k // group, group)
    mn = wg.min(axis=2)
    mx = wg.max(axis=2)
    with np.errstate(over="ignore"):
        s16 = ((mx - mn) / qmax).astype(np.float16)
    s16[s16 == 0] = np.float16(1.0)
    sf = s16.astype(np.float32)
    zf = np.clip(np.rint(-mn / sf), np.float32(0), qmax) + np.float32(0)
    q = np.clip(np.rint(wg / sf[..., None]) + zf[..., None], np.float32(0), qmax)
    return (q.reshape(n, k).astype(np.uint8), s16.view(np.uint16),
            zf.astype(np.float16).view(np.uint16))


def test_golden_worked_examples(orc):
    with open(GOLDEN) as f:
        ex = json.load(f)["examples"]
    for e in ex:
        w = np.array([e["w"]], np.float32)
        q, s, z, nf = orc.quantize(w, group=w.shape[1], bits=e["bits"])
        assert nf == 0
        assert int(s[0, 0]) == int(e["s_f16_bits"], 16), e["name"]
        assert orc.f16_bits_to_f64(z)[0, 0] == e["z"], e["name"]
        assert q[0].tolist() == e["q"], e["name"]


@pytest.mark.parametrize("bits", [2, 3, 4])
@pytest.mark.parametrize("group", [32, 64, 128])
@pytest.mark.parametrize("dist", ["n002", "n1", "uniform", "mixed"])
def test_matches_numpy_brute_force(orc, bits, group, dist):
    rng = np.random.default_rng(bits * 1000 + group + len(dist))
    n, k = 48, 512
    if dist == "n002":
        w = rng.standard_normal((n, k)) * 0.02
    elif dist == "n1":
        w = rng.standard_normal((n, k))
    elif dist == "uniform":
        w = rng.uniform(-3, 1, (n, k))
    else:
        w = rng.standard_normal((n, k)) * 0.02
        w[0] = 0.25                    # constant rows
        w[1] = -0.0
        w[2] = np.abs(w[2]) + 1.0      # all-positive
        w[3] = -np.abs(w[3]) - 1.0     # all-negative
        w[4, :group] = 1e5             # scale overflows binary16
        w[5] = rng.standard_normal(k) * 1e-7   # scales in the binary16 subnormal range
        w[6, ::2] = 0.0
        w[6, 1::2] = -0.0
    w = w.astype(np.float32)
    q, s, z, nf = orc.quantize(w, group, bits)
    q2, s2, z2 = np_quantize(w, group, bits)
    np.testing.assert_array_equal(s, s2)
    np.testing.assert_array_equal(z, z2)
    np.testing.assert_array_equal(q, q2)
    assert nf == 0


def test_exact_grid_reconstructs(orc):
    # Groups that are exactly {(i - z0) * s : i = 0..qmax} with a binary16 scale.
    rng = np.random.default_rng(7)
    for bits in (2, 3, 4):
        qmax = 2 ** bits - 1
        rows = []
        for _ in range(64):
            s = float(np.float16(rng.uniform(0.001, 0.1)))
            z0 = int(rng.integers(0, qmax + 1))
            codes = np.concatenate([np.arange(qmax + 1), rng.integers(0, qmax + 1, 128 - qmax - 1)])
            rng.shuffle(codes)
            rows.append(((codes - z0) * s).astype(np.float32))
        w = np.stack(rows)
        q, sb, zb, _ = orc.quantize(w, 128, bits)
        deq = orc.dequant(q, sb, zb, 128)
        np.testing.assert_array_equal(deq, w.astype(np.float64))


@pytest.mark.parametrize("bits", [2, 3, 4])
def test_rounding_bound_inside_clamp_range(orc, bits):
    rng = np.random.default_rng(11)
    group = 64
    w = (rng.standard_normal((64, 1024)) * 0.02).astype(np.float32)
    q, s, z, _ = orc.quantize(w, group, bits)
    deq = orc.dequant(q, s, z, group)
    sf = np.repeat(orc.f16_bits_to_f64(s), group, axis=1)
    zf = np.repeat(orc.f16_bits_to_f64(z), group, axis=1)
    qmax = 2 ** bits - 1
    lo, hi = -zf * sf, (qmax - zf) * sf
    inside = (w >= lo - sf / 2) & (w <= hi + sf / 2)
    err = np.abs(w.astype(np.float64) - deq)
    # s/2, plus the one fp32 rounding of w/s before rint
    assert np.all(err[inside] <= sf[inside] * (0.5 + 2.0 ** -20))
    # every weight within [min, max] of its group lies inside the clamp range
    # up to the scale's binary16 rounding
    wg = w.reshape(64, -1, group)
    mn = np.repeat(wg.min(axis=2), group, axis=1)
    mx = np.repeat(wg.max(axis=2), group, axis=1)
    assert np.all(err <= np.maximum(sf * (0.5 + 2.0 ** -20), np.abs(mx - mn) / qmax * 0.51 + 1e-12))


def test_rtn_error_level_sanity(orc):
    # Not a parity pin: relative Frobenius error of RTN on N(0, 0.02) weights.
    rng = np.random.default_rng(5)
    w = (rng.standard_normal((256, 2048)) * 0.02).astype(np.float32)
    levels = {}
    for bits, group in ((2, 128), (2, 64), (3, 32), (4, 128)):
        q, s, z, _ = orc.quantize(w, group, bits)
        deq = orc.dequant(q, s, z, group)
        levels[(bits, group)] = np.linalg.norm(deq - w) / np.linalg.norm(w)
    assert 0.40 < levels[(2, 128)] < 0.60
    assert levels[(2, 64)] < levels[(2, 128)]
    assert levels[(4, 128)] < levels[(3, 32)] < levels[(2, 64)]  # App. B's INT3 g32 between INT4 and INT2
    assert 0.06 < levels[(4, 128)] < 0.14


def test_nonfinite_weights_are_counted(orc):
    w = np.zeros((2, 64), np.float32)
    w[1, 3] = np.nan
    w[1, 9] = np.inf
    _, _, _, nf = orc.quantize(w, 64, 2)
    assert nf == 2


def test_rejects_bad_group(orc):
    with pytest.raises(ValueError):
        orc.quantize(np.zeros((2, 96), np.float32), 64, 2)
