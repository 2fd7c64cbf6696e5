"""Pins for the oracle's adapter merge (Eq. 1 with the adapter folded into the
matrix; Sec. 4.2 allows merging the trained adapters into the quantized
weights, Sec. 7 step 5 deploys either form).

The merged matrix deq(W) + alpha B A is checked against numpy's own float16
/ bfloat16 decoding and matmul on inputs for which the fp64 sums are exact
(so the single rounding to fp32 must agree bit for bit), against a 1-ulp
bound on N(0, 0.01) adapters, and through the requantization: with alpha = 0
RTN reproduces every group that holds both end codes (a fixed point of the
quantizer), and a shift of a whole group by a multiple of its step moves
its zero point and leaves its codes and scale alone.
"""
import numpy as np
import pytest


def bf16_bits_np(v):
    """bf16 bit patterns of values that bf16 holds exactly (checked)."""
    f = np.asarray(v, np.float32)
    b = (f.view(np.uint32) >> 16).astype(np.uint16)
    assert np.array_equal((b.astype(np.uint32) << 16).view(np.float32), f)
    return b


def bf16_to_f64_np(b):
    return (np.asarray(b, np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def deq_np(q, s, z, group):
    """deq(W) from numpy's float16 decoding (independent of the oracle's)."""
    sf = np.repeat(s.view(np.float16).astype(np.float64), group, axis=1)
    zf = np.repeat(z.view(np.float16).astype(np.float64), group, axis=1)
    return sf * (q.astype(np.float64) - zf)


def grid_adapter(rng, n, k, r):
    """B [n, r], A [r, k] with entries m * 2^-12, |m| < 256: exact in bf16, and
    every fp64 sum of their products is exact."""
    b = rng.integers(-255, 256, size=(n, r)).astype(np.float64) * 2.0 ** -12
    a = rng.integers(-255, 256, size=(r, k)).astype(np.float64) * 2.0 ** -12
    return bf16_bits_np(b), bf16_bits_np(a)


@pytest.mark.parametrize("bits,group,r,alpha", [(2, 128, 16, 2.0), (4, 64, 8, 0.5), (2, 32, 1, 2.0),
                                                (4, 128, 64, 0.125)])
def test_merge_equals_numpy_on_exact_inputs(orc, bits, group, r, alpha):
    rng = np.random.default_rng(100 + r)
    n, k = 24, 256
    w = rng.normal(0, 0.02, (n, k)).astype(np.float32)
    q, s, z, _ = orc.quantize(w, group, bits)
    lb, la = grid_adapter(rng, n, k, r)
    got = orc.merge_lora(q, s, z, group, lb, la, alpha)
    want = (deq_np(q, s, z, group) + alpha * (bf16_to_f64_np(lb) @ bf16_to_f64_np(la))).astype(np.float32)
    assert got.dtype == np.float32
    assert np.array_equal(got.view(np.uint32), want.view(np.uint32))


def test_merge_within_one_ulp_of_numpy_on_gaussian_adapters(orc):
    rng = np.random.default_rng(7)
    n, k, r, group = 48, 384, 16, 128
    w = rng.normal(0, 0.02, (n, k)).astype(np.float32)
    q, s, z, _ = orc.quantize(w, group, 2)
    lb = orc.f64_to_bf16_bits(rng.normal(0, 0.01, (n, r)))
    la = orc.f64_to_bf16_bits(rng.normal(0, 0.01, (r, k)))
    got = orc.merge_lora(q, s, z, group, lb, la, 2.0)
    want = (deq_np(q, s, z, group) + 2.0 * (bf16_to_f64_np(lb) @ bf16_to_f64_np(la))).astype(np.float32)
    ulp = np.spacing(np.abs(want))
    assert np.all(np.abs(got.astype(np.float64) - want) <= ulp)
    assert np.mean(got == want) > 0.999


@pytest.mark.parametrize("bits,group", [(2, 128), (2, 32), (4, 128), (4, 64)])
def test_alpha_zero_is_the_dequantized_matrix_and_a_fixed_point(orc, bits, group):
    rng = np.random.default_rng(bits * 1000 + group)
    n, k, r = 32, 512, 8
    w = rng.normal(0, 0.02, (n, k)).astype(np.float32)
    q, s, z, _ = orc.quantize(w, group, bits)
    lb = orc.f64_to_bf16_bits(rng.normal(0, 0.01, (n, r)))
    la = orc.f64_to_bf16_bits(rng.normal(0, 0.01, (r, k)))
    for args in ((lb, la, 0.0), (lb[:, :0], la[:0], 2.0)):  # alpha = 0, and rank 0
        wm = orc.merge_lora(q, s, z, group, *args)
        assert np.array_equal(wm.astype(np.float64), deq_np(q, s, z, group))  # s (q - z) is exact in fp32
    q2, s2, z2, nf = orc.quantize(wm, group, bits)
    assert nf == 0
    qmax = 2 ** bits - 1
    qg = q.reshape(n, k // group, group)
    full = (qg.min(axis=2) == 0) & (qg.max(axis=2) == qmax)  # groups that use both end codes
    assert full.mean() > 0.5
    assert np.array_equal(s2[full], s[full]) and np.array_equal(z2[full], z[full])
    assert np.array_equal(q2.reshape(n, k // group, group)[full], qg[full])


def test_group_shift_moves_only_the_zero_point(orc):
    """B A = c on one group, c a multiple of the group's step s: the group's
    range moves by c, so the requantized group keeps its scale and codes and
    its zero point moves by -c / s (inside [0, qmax])."""
    bits, group, n, k = 4, 64, 16, 128
    rng = np.random.default_rng(3)
    q = rng.integers(0, 16, size=(n, k)).astype(np.uint8)
    q[:, 0], q[:, 64], q[:, 1], q[:, 65] = 0, 0, 15, 15  # both end codes in every group
    s = np.full((n, 2), np.float16(2.0 ** -6)).view(np.uint16)
    z = np.full((n, 2), np.float16(8.0)).view(np.uint16)
    # rank 1: B[:, 0] = 1, A[0, :64] = -3 s (every row's first group moves down by 3 steps)
    lb = bf16_bits_np(np.ones((n, 1)))
    la = bf16_bits_np(np.concatenate([np.full(64, -3 * 2.0 ** -6), np.zeros(64)])[None, :])
    wm = orc.merge_lora(q, s, z, group, lb, la, 1.0)
    q2, s2, z2, _ = orc.quantize(wm, group, bits)
    assert np.array_equal(q2, q) and np.array_equal(s2, s)
    z2f = z2.view(np.float16).astype(np.float64)
    assert np.all(z2f[:, 0] == 11.0) and np.all(z2f[:, 1] == 8.0)


def test_merge_rejects_bad_shapes(orc):
    q = np.zeros((2, 96), np.uint8)
    s = np.zeros((2, 1), np.uint16)
    with pytest.raises(ValueError):
        orc.merge_lora(q, s, s, 64, np.zeros((2, 1), np.uint16), np.zeros((1, 96), np.uint16), 1.0)
