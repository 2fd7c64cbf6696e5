"""Pins for the packed storage format the oracle defines.

Beyond the pack/unpack round trip, the layout is checked against the PTX ISA
definition of the m16n8k16 f16 A-operand fragment: extracting codes from a
lane's words with fixed masks and shifts must hand each lane exactly the
(row, k) elements the fragment assigns to it.  That is the property the
packed format exists for, derived here independently of the oracle's formula.
"""
import numpy as np
import pytest


def _rand_codes(rng, n, k, bits, group):
    q = rng.integers(0, 2 ** bits, (n, k)).astype(np.uint8)
    s = rng.integers(0, 0x7BFF, (n, k // group)).astype(np.uint16)
    z = rng.integers(0, 0x7BFF, (n, k // group)).astype(np.uint16)
    return q, s, z


@pytest.mark.parametrize("bits", [2, 3, 4])
@pytest.mark.parametrize("n,k,group", [(16, 128, 128), (48, 256, 64), (37, 192, 64), (5, 96, 32), (130, 384, 128)])
def test_roundtrip(orc, bits, n, k, group):
    rng = np.random.default_rng(n * k + bits)
    q, s, z = _rand_codes(rng, n, k, bits, group)
    codes, meta = orc.tile_pack(q, s, z, group, bits)
    q2, s2, z2 = orc.tile_unpack(codes, meta, n, k, group, bits)
    np.testing.assert_array_equal(q, q2)
    np.testing.assert_array_equal(s, s2)
    np.testing.assert_array_equal(z, z2)


@pytest.mark.parametrize("bits", [2, 3, 4])
def test_padding_is_zero(orc, bits):
    n, k, group = 21, 160, 32
    q = np.full((n, k), 2 ** bits - 1, np.uint8)
    s = np.full((n, k // group), 0x3C00, np.uint16)
    z = np.full((n, k // group), 0x3C00, np.uint16)
    codes, meta = orc.tile_pack(q, s, z, group, bits)
    rt, kb = 2, 2
    ng = kb * 128 // group
    # every (row, col) outside [n, k] must be zero: rebuild a full padded matrix
    qp, sp, zp = orc.tile_unpack(codes, meta, rt * 16, kb * 128, group, bits)
    assert np.all(qp[n:, :] == 0) and np.all(qp[:, k:] == 0)
    assert np.all(qp[:n, :k] == 2 ** bits - 1)
    assert np.all(sp[n:, :] == 0) and np.all(sp[:, k // group:] == 0)
    assert np.all(zp[n:, :] == 0) and np.all(zp[:, k // group:] == 0)
    assert sp.shape == (rt * 16, ng)


def _fragment_owner(lane, reg, elem):
    """PTX m16n8k16 .f16 A fragment: (row, col) of element `elem` (0/1) of register `reg` (0..3)."""
    group_id, tig = lane // 4, lane % 4
    row = group_id + (8 if reg in (1, 3) else 0)
    col = tig * 2 + elem + (8 if reg in (2, 3) else 0)
    return row, col


def test_w2_layout_matches_mma_fragments(orc):
    rng = np.random.default_rng(0)
    q = rng.integers(0, 4, (16, 128)).astype(np.uint8)
    codes, _ = orc.tile_pack(q, np.zeros((16, 1), np.uint16), np.zeros((16, 1), np.uint16), 128, 2)
    words = codes.reshape(32, 4)            # [lane][word]
    for lane in range(32):
        for wi in range(4):
            w = int(words[lane, wi])
            # v_j: mask (3 << 2j) on the word (j < 4) or on the word >> 8 (j >= 4),
            # one code in each 16-bit half, scaled by 4^(j % 4)
            v = []
            for j in range(8):
                src = w if j < 4 else (w >> 8)
                sh = 2 * (j % 4)
                v.append(((src >> sh) & 3, (src >> (16 + sh)) & 3))
            for s in range(2):                      # two k-steps per word
                kstep = 2 * wi + s
                regs = [v[2 * s], v[4 + 2 * s], v[2 * s + 1], v[4 + 2 * s + 1]]
                for reg in range(4):
                    for elem in range(2):
                        row, col = _fragment_owner(lane, reg, elem)
                        assert regs[reg][elem] == q[row, 16 * kstep + col]


def test_w4_layout_matches_mma_fragments(orc):
    rng = np.random.default_rng(1)
    q = rng.integers(0, 16, (16, 128)).astype(np.uint8)
    codes, _ = orc.tile_pack(q, np.zeros((16, 1), np.uint16), np.zeros((16, 1), np.uint16), 128, 4)
    words = codes.reshape(2, 32, 4)         # [64-feature half][lane][word]
    for half in range(2):
        for lane in range(32):
            for wi in range(4):
                w = int(words[half, lane, wi])
                lo = w & 0x000F000F
                hi = w & 0x00F000F0
                lo8 = (w >> 8) & 0x000F000F
                hi8 = (w >> 8) & 0x00F000F0
                regs = [lo, lo8, hi >> 4, hi8 >> 4]
                kstep = half * 4 + wi
                for reg in range(4):
                    for elem in range(2):
                        row, col = _fragment_owner(lane, reg, elem)
                        val = (regs[reg] >> (16 * elem)) & 0xF
                        assert val == q[row, 16 * kstep + col]


def test_w3_layout_matches_mma_fragments(orc):
    """3-bit codes (App. B) as two planes, read the way a kernel would: the
    2-bit plane's class c taken with the mask 3 << 2c (rows g + 8 from the
    word >> 8), and the plane-1 bit of the same code moved to bit 2c + 2 by
    one shift of the lane's plane-1 word (<< 2 / << 1 for the even 2-bit
    word, >> 6 / >> 7 for the odd one, rows g / g + 8) and the mask 4 << 2c.
    Each 16-bit half of a register must then read q * 4^c for the (row, k)
    the PTX fragment assigns to it, below 1024 (a binary16 subnormal)."""
    rng = np.random.default_rng(2)
    q = rng.integers(0, 8, (16, 128)).astype(np.uint8)
    codes, _ = orc.tile_pack(q, np.zeros((16, 1), np.uint16), np.zeros((16, 1), np.uint16), 128, 3)
    assert codes.size == 192
    lo_words = codes[:128].reshape(32, 4)   # [lane][word]
    hi_words = codes[128:].reshape(32, 2)   # [lane][word]
    shifts = {(0, 0): ("<<", 2), (0, 1): ("<<", 1), (1, 0): (">>", 6), (1, 1): (">>", 7)}  # (word parity, row half)
    for lane in range(32):
        for wi in range(4):
            w, hw = int(lo_words[lane, wi]), int(hi_words[lane, wi // 2])
            for s in range(2):                      # two k-steps per 2-bit word
                kstep = 2 * wi + s
                for reg in range(4):
                    rowhalf = 1 if reg in (1, 3) else 0
                    cls = 2 * s + (1 if reg in (2, 3) else 0)
                    src = (w >> 8) if rowhalf else w
                    lo = src & ((3 << 2 * cls) | (3 << (16 + 2 * cls)))
                    op, n = shifts[(wi % 2, rowhalf)]
                    h = ((hw << n) if op == "<<" else (hw >> n)) & 0xFFFFFFFF
                    hi = h & ((4 << 2 * cls) | (4 << (16 + 2 * cls)))
                    r = lo | hi
                    for elem in range(2):
                        row, col = _fragment_owner(lane, reg, elem)
                        val = (r >> (16 * elem)) & 0xFFFF
                        assert val == int(q[row, 16 * kstep + col]) * 4 ** cls
                        assert val < 1024


def test_meta_layout_matches_fragment_rows(orc):
    # lane -> group_id = lane / 4 reads entry group_id: scales/zeros of rows g and g + 8.
    n, k, group = 16, 256, 64
    s = np.arange(n * (k // group), dtype=np.uint16).reshape(n, k // group) + 1
    z = s + 1000
    q = np.zeros((n, k), np.uint8)
    _, meta = orc.tile_pack(q, s, z, group, 2)
    meta = meta.reshape(-1, 8, 4)           # [(rt, group)][entry][s_g, s_g8, z_g, z_g8]
    for j in range(k // group):
        for g in range(8):
            assert tuple(meta[j, g]) == (s[g, j], s[g + 8, j], z[g, j], z[g + 8, j])
