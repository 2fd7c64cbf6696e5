"""Adapter merge (wq_merge_lora) vs the oracle: the merged fp32 matrix
deq(W) + alpha B A (Eq. 1 folded into the weights, Sec. 4.2 / Sec. 7 step 5)
and its requantized codes, scales and zeros must match bit for bit; the
merged layer then runs on the decode path with no adapter."""
import numpy as np
import pytest
import torch

import oracle as orc
from paper_2606_04238_gb300 import synth
from tests.gpu_util import check_bf16, upload_packed

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def wq():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2606_04238_gb300 import wq as mod
    return mod


def _case(n, k, group, bits, r, seed):
    rng = np.random.default_rng(seed)
    w = (rng.standard_normal((n, k)) * 0.02).astype(np.float32)
    q, s, z, _ = orc.quantize(w, group, bits)
    a, b, _ = synth.lora(k, n, r, seed + 1) if r else (None, None, None)
    return (q, s, z), (None if r == 0 else a[:r].contiguous()), b


def _oracle_merge(qsz, group, bits, a, b, alpha):
    if b is None:
        n = qsz[0].shape[0]
        wm = orc.merge_lora(*qsz, group, np.zeros((n, 0), np.uint16), np.zeros((0, qsz[0].shape[1]), np.uint16), alpha)
    else:
        wm = orc.merge_lora(*qsz, group, synth.bf16_bits(b), synth.bf16_bits(a), alpha)
    codes, meta = orc.tile_pack(*orc.quantize(wm, group, bits)[:3], group, bits)
    return wm, codes, meta


def _assert_packed(qw, codes, meta):
    torch.cuda.synchronize()
    assert np.array_equal(qw.codes.cpu().numpy().view(np.uint32), codes)
    assert np.array_equal(qw.meta.cpu().numpy().view(np.uint16), meta)


@pytest.mark.parametrize("bits", [2, 3, 4])
@pytest.mark.parametrize("n,k,group,r", [(16, 128, 128, 1), (40, 384, 128, 16), (33, 192, 64, 8),
                                         (200, 384, 32, 64), (1000, 640, 128, 32), (5, 96, 32, 8)])
@pytest.mark.parametrize("alpha", [2.0, 0.37])
def test_merge_bit_exact(wq, bits, n, k, group, r, alpha):
    qsz, a, b = _case(n, k, group, bits, r, seed=n * 7 + k + r + bits)
    src = upload_packed(*qsz, group, bits)
    wm = torch.empty((n, k), dtype=torch.float32, device="cuda")
    out = wq.merge_lora(src, b.cuda(), a.cuda(), alpha, w_merged=wm)
    wm_ref, codes, meta = _oracle_merge(qsz, group, bits, a, b, alpha)
    _assert_packed(out, codes, meta)
    assert np.array_equal(wm.cpu().numpy().view(np.uint32), wm_ref.view(np.uint32))
    assert (out.n, out.k, out.group, out.bits) == (n, k, group, bits)
    # the source is untouched
    c0, m0 = orc.tile_pack(*qsz, group, bits)
    _assert_packed(src, c0, m0)


@pytest.mark.parametrize("bits", [2, 3, 4])
def test_merge_rank0_and_alpha0(wq, bits):
    n, k, group = 48, 256, 64
    qsz, a, b = _case(n, k, group, bits, 8, seed=5 + bits)
    src = upload_packed(*qsz, group, bits)
    for out, args in ((wq.merge_lora(src, None, None, 2.0), (None, None, 2.0)),
                      (wq.merge_lora(src, b.cuda(), a.cuda(), 0.0), (a, b, 0.0))):
        _, codes, meta = _oracle_merge(qsz, group, bits, *args)
        _assert_packed(out, codes, meta)


def test_merge_in_place(wq):
    n, k, group, bits, r = 72, 512, 128, 2, 16
    qsz, a, b = _case(n, k, group, bits, r, seed=11)
    src = upload_packed(*qsz, group, bits)
    out = wq.merge_lora(src, b.cuda(), a.cuda(), 2.0, out=src)
    assert out is src
    _, codes, meta = _oracle_merge(qsz, group, bits, a, b, 2.0)
    _assert_packed(src, codes, meta)


def test_merge_full_size_qwen3_4b_gate(wq):
    cfg = synth.CONFIGS["qwen3_4b"]
    w = synth.weights((cfg.inter, cfg.d), 4321)
    qsz = orc.quantize(w.numpy(), cfg.group_gu, 2)[:3]
    a, bg, _ = synth.lora(cfg.d, cfg.inter, cfg.r, 4322)
    a = a[:cfg.r].contiguous()
    src = upload_packed(*qsz, cfg.group_gu, 2)
    out = wq.merge_lora(src, bg.cuda(), a.cuda(), cfg.lora_scale)
    _, codes, meta = _oracle_merge(qsz, cfg.group_gu, 2, a, bg, cfg.lora_scale)
    _assert_packed(out, codes, meta)


@pytest.mark.parametrize("m", [1, 8, 40])
def test_merged_layer_forward(wq, m):
    """A merged layer on the decode (m <= 16) and GEMM (m > 16) paths, r = 0,
    vs the oracle's gate/up on the oracle's merged codes."""
    d, inter, group, r = 512, 1000, 128, 16
    rng = np.random.default_rng(77)
    wg = (rng.standard_normal((inter, d)) * 0.02).astype(np.float32)
    wu = (rng.standard_normal((inter, d)) * 0.02).astype(np.float32)
    g0, u0 = orc.quantize(wg, group, 2)[:3], orc.quantize(wu, group, 2)[:3]
    a, bg, bu = synth.lora(d, inter, r, 78)
    L = wq.MLPLayer(upload_packed(*g0, group, 2), upload_packed(*u0, group, 2), None,  # no down: gate/up only
                    a.cuda(), bg.cuda(), bu.cuda(), 2.0)
    M = wq.merge_layer(L)
    assert M.r == 0
    x = synth.activations((m, d), 79 + m)
    h = wq.gateup_w2_lora(x.cuda(), M.gate, M.up, prenorm=True)
    torch.cuda.synchronize()
    gm = orc.quantize(orc.merge_lora(*g0, group, synth.bf16_bits(bg), synth.bf16_bits(a[:r]), 2.0), group, 2)[:3]
    um = orc.quantize(orc.merge_lora(*u0, group, synth.bf16_bits(bu), synth.bf16_bits(a[r:]), 2.0), group, 2)[:3]
    ref, _ = orc.gateup(synth.bf16_bits(x), gm, um, group, prenorm=True)
    check_bf16(h, ref, f"merged h m={m}", min_exact=0.6 if m > 16 else 0.97)


def test_merge_argument_errors(wq):
    n, k, group = 32, 128, 64
    qsz, a, b = _case(n, k, group, 2, 8, seed=3)
    src = upload_packed(*qsz, group, 2)
    with pytest.raises(wq.WQError) as e:
        wq.merge_lora(src, b.cuda(), a.cuda(), float("nan"))
    assert e.value.status == -1  # WQ_ERR_ARG
    wm = torch.empty(n * k + 1, dtype=torch.float32, device="cuda")[1:].view(n, k)  # 4-byte offset
    with pytest.raises(wq.WQError) as e:
        wq.merge_lora(src, b.cuda(), a.cuda(), 1.0, w_merged=wm)
    assert e.value.status == -3  # WQ_ERR_ALIGN
    bad = wq.QWeight(src.codes, src.meta, n, k, 48, 2)
    with pytest.raises(wq.WQError) as e:
        wq.merge_lora(bad, b.cuda(), a.cuda(), 1.0)
    assert e.value.status == -2  # WQ_ERR_SHAPE
