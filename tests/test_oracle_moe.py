"""Pins for the oracle's mixture-of-experts block (oracle/moe.py; Sec. 5's MoE
model activates a subset of experts per token).

Reductions and invariants, not a retyped formula:
- one expert selected out of one equals the dense MLP oracle bit for bit;
- experts that are not selected are never read (NaN weights there change
  nothing);
- relabelling the experts together with their logits changes nothing;
- two selected experts with equal logits give the mean of their outputs;
- the routing picks the largest logits, the lower index among ties, and its
  weights are a softmax.
"""
import numpy as np
import pytest
import torch


def _bits(a):
    t = torch.from_numpy(np.asarray(a, np.float64)).float().to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def _expert(orc, rng, d=128, inter=256):
    def w(n, k, g, b):
        return orc.quantize((rng.standard_normal((n, k)) * 0.02).astype(np.float32), g, b)[:3]
    return {"gate": w(inter, d, 64, 2), "up": w(inter, d, 64, 2), "down": w(d, inter, 64, 4)}


@pytest.fixture
def moe():
    from oracle import moe as m
    return m


def test_single_expert_is_the_dense_block(orc, moe):
    rng = np.random.default_rng(0)
    ex = _expert(orc, rng)
    x = _bits(rng.standard_normal((3, 128)))
    y, yb, idx, w = moe.moe_block(x, np.zeros((3, 1)), 1, [ex], 64, 64)
    assert np.all(idx == 0) and np.all(w == 1.0)
    _, h_bits = orc.gateup(x, ex["gate"], ex["up"], 64, prenorm=True)
    y_ref, yb_ref = orc.down(h_bits, ex["down"], 64, x)
    np.testing.assert_array_equal(y, y_ref)
    np.testing.assert_array_equal(yb, yb_ref)


def test_unselected_experts_are_not_read(orc, moe):
    rng = np.random.default_rng(1)
    experts = [_expert(orc, rng) for _ in range(6)]
    x = _bits(rng.standard_normal((4, 128)))
    logits = rng.standard_normal((4, 6))
    y, _, idx, _ = moe.moe_block(x, logits, 2, experts, 64, 64)
    used = set(idx.ravel().tolist())
    broken = []
    for e, ex in enumerate(experts):
        if e in used:
            broken.append(ex)
        else:
            q, s, z = ex["down"]
            broken.append({**ex, "down": (q, np.full_like(s, 0x7E00), z)})  # NaN scales
    y2, _, _, _ = moe.moe_block(x, logits, 2, broken, 64, 64)
    np.testing.assert_array_equal(y2, y)


def test_relabelling_experts_changes_nothing(orc, moe):
    rng = np.random.default_rng(2)
    experts = [_expert(orc, rng) for _ in range(5)]
    x = _bits(rng.standard_normal((3, 128)))
    logits = rng.standard_normal((3, 5))
    y, _, _, _ = moe.moe_block(x, logits, 3, experts, 64, 64)
    perm = [3, 0, 4, 1, 2]
    y2, _, _, _ = moe.moe_block(x, logits[:, perm], 3, [experts[p] for p in perm], 64, 64)
    np.testing.assert_allclose(y2, y, rtol=1e-13, atol=1e-15)


def test_equal_logits_average_two_experts(orc, moe):
    rng = np.random.default_rng(3)
    experts = [_expert(orc, rng) for _ in range(3)]
    x = _bits(rng.standard_normal((2, 128)))
    logits = np.array([[1.0, 1.0, -5.0], [1.0, 1.0, -5.0]])
    y, _, idx, w = moe.moe_block(x, logits, 2, experts, 64, 64)
    assert np.array_equal(idx, [[0, 1], [0, 1]]) and np.all(w == 0.5)
    xf = orc.bf16_bits_to_f64(x)
    outs = []
    for e in (0, 1):
        _, hb = orc.gateup(x, experts[e]["gate"], experts[e]["up"], 64, prenorm=True)
        outs.append(orc.down(hb, experts[e]["down"], 64, None)[0])
    np.testing.assert_allclose(y, xf + 0.5 * (outs[0] + outs[1]), rtol=1e-14, atol=1e-15)


def test_routing(moe):
    logits = np.array([[0.5, 2.0, 2.0, -1.0], [3.0, 1.0, 0.0, 1.0]])
    idx, w = moe.route(logits, 2)
    assert idx.tolist() == [[1, 2], [0, 1]]          # ties: the lower index first
    np.testing.assert_allclose(w[0], [0.5, 0.5])
    e = np.exp([3.0, 1.0])
    np.testing.assert_allclose(w[1], e / e.sum(), rtol=1e-15)
    np.testing.assert_allclose(w.sum(axis=1), 1.0, rtol=1e-15)
