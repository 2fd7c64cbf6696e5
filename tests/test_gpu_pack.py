"""GPU quantizer/packer (wq_pack) vs the oracle: codes, scales and zeros must
match bit for bit (Sec. 4.1 quantization, packed format of include/wq.h)."""
import numpy as np
import pytest
import torch

import oracle as orc

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def wq():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2606_04238_gb300 import wq as mod
    return mod


def _weights(kind, n, k, rng):
    if kind == "n002":
        w = rng.standard_normal((n, k)) * 0.02
    elif kind == "n1":
        w = rng.standard_normal((n, k))
    else:
        w = rng.standard_normal((n, k)) * 0.02
        w[0] = 0.125
        if n > 2:
            w[1] = np.abs(w[1]) + 0.5
            w[2] = -np.abs(w[2]) - 0.5
        if n > 4:
            w[3, ::2] = 0.0
            w[3, 1::2] = -0.0
            w[4] *= 1e-6
    return w.astype(np.float32)


@pytest.mark.parametrize("bits", [2, 3, 4])
@pytest.mark.parametrize("n,k,group", [(16, 128, 128), (768, 256, 64), (37, 192, 64), (200, 384, 32),
                                       (1000, 640, 128), (5, 96, 32)])
@pytest.mark.parametrize("dist", ["n002", "n1", "edge"])
def test_pack_bit_exact(wq, bits, n, k, group, dist):
    rng = np.random.default_rng(n + k + group + bits + len(dist))
    w = _weights(dist, n, k, rng)
    q = wq.pack(torch.from_numpy(w).cuda(), group, bits)
    torch.cuda.synchronize()
    codes, meta = orc.tile_pack(*orc.quantize(w, group, bits)[:3], group, bits)
    np.testing.assert_array_equal(q.meta.cpu().numpy().view(np.uint16), meta)
    np.testing.assert_array_equal(q.codes.cpu().numpy().view(np.uint32), codes)


def test_pack_full_size_qwen3_4b_gate(wq):
    from paper_2606_04238_gb300 import synth
    cfg = synth.CONFIGS["qwen3_4b"]
    w = synth.weights((cfg.inter, cfg.d), 12345)
    q = wq.pack(w.cuda(), 128, 2)
    torch.cuda.synchronize()
    codes, meta = orc.tile_pack(*orc.quantize(w.numpy(), 128, 2)[:3], 128, 2)
    assert np.array_equal(q.meta.cpu().numpy().view(np.uint16), meta)
    assert np.array_equal(q.codes.cpu().numpy().view(np.uint32), codes)


def test_pack_nonfinite_flag(wq):
    w = torch.zeros((32, 128), dtype=torch.float32)
    flag = torch.zeros(1, dtype=torch.int32, device="cuda")
    wq.pack(w.cuda(), 64, 2, nonfinite=flag)
    torch.cuda.synchronize()
    assert int(flag.item()) == 0
    w[7, 100] = float("nan")
    w[20, 3] = float("inf")
    wq.pack(w.cuda(), 64, 2, nonfinite=flag)
    torch.cuda.synchronize()
    assert int(flag.item()) == 1
