"""wq_gateup_w2_lora_noalloc: the fused 2-bit gate/up call for callers that
cannot allocate device memory (the scratch lives in a fixed array inside the
library instead of a caller-provided workspace).

Its output must match the workspace entry point wq_gateup_w2_lora on the same
inputs, on two calls in a row (the second reuses the array the first left
behind).  Collected last, so that a failure here cannot hide another test.
"""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


def _close(got, ref, what):
    # the bound the GEMV parity tests use: 2e-3 (max|ref| + 1) plus half a bf16 ulp of ref
    g = got.float().cpu().numpy().astype(np.float64)
    r = ref.float().cpu().numpy().astype(np.float64)
    tol = 2e-3 * (np.abs(r).max() + 1.0) + np.abs(r) * 2.0 ** -8
    assert np.all(np.abs(g - r) <= tol), f"{what}: max diff {np.abs(g - r).max():.3e}"


@pytest.mark.parametrize("d,inter,group,r,m,prenorm", [
    (256, 768, 64, 8, 1, False),        # the small single-layer workload
    (2560, 9728, 128, 16, 1, True),     # a Qwen3-4B-shaped layer
    (512, 1000, 128, 32, 16, True),     # ragged rows, a 16-token batch
])
def test_noalloc_matches_workspace_entry_point(d, inter, group, r, m, prenorm):
    import __graft_entry__
    __graft_entry__.build()
    from paper_2606_04238_gb300 import synth, wq

    dev = torch.device("cuda:0")
    gen = torch.Generator(device="cpu").manual_seed(d + inter + m)
    wg = (torch.randn((inter, d), generator=gen) * 0.02).to(dev)
    wu = (torch.randn((inter, d), generator=gen) * 0.02).to(dev)
    g, u = wq.pack(wg, group, 2), wq.pack(wu, group, 2)
    a, bg, bu = (t.to(dev) for t in synth.lora(d, inter, r, 77))
    x = synth.activations((m, d), 78).to(dev)

    ws = wq.workspace(m, d, inter, r)
    ref = wq.gateup_w2_lora(x, g, u, a, bg, bu, lora_scale=2.0, prenorm=prenorm, ws=ws)
    h1 = torch.empty_like(ref)
    h2 = torch.empty_like(ref)
    wq.gateup_w2_lora_noalloc(x, g, u, a, bg, bu, lora_scale=2.0, prenorm=prenorm, h=h1)
    wq.gateup_w2_lora_noalloc(x, g, u, a, bg, bu, lora_scale=2.0, prenorm=prenorm, h=h2)
    torch.cuda.synchronize()
    assert wq.device_status() == 0
    _close(h1, ref, "first no-alloc call")
    _close(h2, ref, "second no-alloc call")
    if d == 2560:
        # the Qwen3-4B-shaped case also against the fp64 oracle, with the GEMV tests' bound
        import oracle as orc
        from tests.gpu_util import check_bf16
        qg = orc.quantize(wg.cpu().numpy(), group, 2)[:3]
        qu = orc.quantize(wu.cpu().numpy(), group, 2)[:3]
        ora, _ = orc.gateup(synth.bf16_bits(x.cpu()), qg, qu, group, synth.bf16_bits(a.cpu()),
                            synth.bf16_bits(bg.cpu()), synth.bf16_bits(bu.cpu()), lora_scale=2.0, prenorm=prenorm)
        check_bf16(h1, ora, "no-alloc call vs oracle")
        check_bf16(h2, ora, "second no-alloc call vs oracle")


def test_noalloc_rejects_a_layer_beyond_its_scratch():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2606_04238_gb300 import wq

    # 64 tokens of a 14B-class layer need more than the built-in scratch
    d, inter = 5120, 17408
    need = wq.workspace_bytes(64, d, inter, 32)
    assert need > 4 << 20
    q = wq.empty_qweight(inter, d, 128, 2)
    x = torch.zeros((64, d), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(wq.WQError) as e:
        wq.gateup_w2_lora_noalloc(x, q, q)
    assert e.value.status == -4 and "scratch" in str(e.value)


def test_noalloc_rejects_more_than_16_tokens():
    """Above 16 tokens the workspace entry point takes the dequant-GEMM path;
    the built-in scratch only serves the decode path, so the call refuses."""
    import __graft_entry__
    __graft_entry__.build()
    from paper_2606_04238_gb300 import wq

    d, inter = 256, 768
    q = wq.empty_qweight(inter, d, 64, 2)
    for m in (17, 33, 64):
        x = torch.zeros((m, d), dtype=torch.bfloat16, device="cuda")
        with pytest.raises(wq.WQError) as e:
            wq.gateup_w2_lora_noalloc(x, q, q)
        assert e.value.status == -4 and "m <= 16" in str(e.value)
