"""bf16 down projection (wq_down_bf16, the down layer of the BF16/W2-GateUp
configuration of Sec. 6.1) vs the fp64 oracle through the C ABI: ragged row
tiles, long and short feature ranges, one and two token tiles and several
token blocks, residual or none, bf16 and fp32 output."""
import numpy as np
import pytest
import torch

import oracle as orc
from paper_2606_04238_gb300 import synth
from tests.gpu_util import check_bf16, check_f32

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def wq():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2606_04238_gb300 import wq as mod
    return mod


CASES = [
    # d, inter
    (256, 768),     # the small single-layer workload
    (200, 384),     # ragged rows: 12.5 row tiles
    (48, 8192),     # few rows, 256 feature chunks split over the warps
    (2560, 9728),   # the Qwen3-4B down matrix
    (40, 96),       # fewer chunks (3) than warps
]


@pytest.mark.parametrize("d,inter", CASES)
@pytest.mark.parametrize("m", [1, 3, 8, 9, 16, 17, 40])
@pytest.mark.parametrize("residual", [True, False])
def test_down_bf16(wq, d, inter, m, residual):
    wd = synth.weights((d, inter), d + inter).to(torch.bfloat16)
    h = synth.activations((m, inter), 300 + m)
    res = synth.activations((m, d), 400 + m) if residual else None
    y = wq.down_bf16(h.cuda(), wd.cuda(), None if res is None else res.cuda())
    torch.cuda.synchronize()
    ref, _ = orc.down_bf16(synth.bf16_bits(h), synth.bf16_bits(wd), None if res is None else synth.bf16_bits(res))
    check_bf16(y, ref, f"y d={d} I={inter} m={m} res={residual}")


@pytest.mark.parametrize("m", [1, 16, 33])
def test_down_bf16_f32_output(wq, m):
    d, inter = 320, 2048
    wd = synth.weights((d, inter), 9).to(torch.bfloat16)
    h = synth.activations((m, inter), 10 + m)
    res = synth.activations((m, d), 11 + m)
    y = wq.down_bf16(h.cuda(), wd.cuda(), res.cuda(), out_f32=True)
    torch.cuda.synchronize()
    assert y.dtype == torch.float32
    ref, _ = orc.down_bf16(synth.bf16_bits(h), synth.bf16_bits(wd), synth.bf16_bits(res))
    check_f32(y, ref, f"y f32 m={m}")


def test_down_bf16_deterministic_and_empty(wq):
    d, inter, m = 512, 1024, 5
    wd = synth.weights((d, inter), 21).to(torch.bfloat16).cuda()
    h = synth.activations((m, inter), 22).cuda()
    a = wq.down_bf16(h, wd)
    b = wq.down_bf16(h, wd)
    torch.cuda.synchronize()
    assert torch.equal(a.view(torch.int16), b.view(torch.int16))
    y = torch.full((1, d), 7.0, dtype=torch.bfloat16, device="cuda")
    wq.down_bf16(h[:0], wd, y=y[:0])
    torch.cuda.synchronize()
    assert bool((y == 7.0).all())


def test_down_bf16_argument_errors(wq):
    d = 64
    h = torch.zeros((2, 80), dtype=torch.bfloat16, device="cuda")
    wd = torch.zeros((d, 80), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(wq.WQError) as e:
        wq.down_bf16(h, wd)  # 80 features: not a multiple of 32
    assert e.value.status == -2
    h = torch.zeros((2, 128), dtype=torch.bfloat16, device="cuda")
    wbuf = torch.zeros(d * 128 + 8, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(wq.WQError) as e:
        wq.down_bf16(h, wbuf[1:1 + d * 128].view(d, 128))  # 2-byte offset
    assert e.value.status == -3
