"""The benchmark's byte and flop models, against independent counts (CPU).

The roofline fractions divide algorithmic bytes (or flops) by measured time.
These tests recompute them another way:
- the packed weights' sizes come from the library's own wq_packed_sizes;
- the adapter and activation sizes come from the tensors' shapes;
- the prefill flops are a sum of 2 m k n over the layer's matrix products,
  and also the per-unit figure (one 128-token x 128-row x 128-feature block
  of one projection) times the units of a launch.
The DRAM traffic record is checked to be used only while the kernel sources
it was measured on are unchanged.
"""
import json
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


@pytest.fixture(scope="module")
def env():
    from paper_2606_04238_gb300 import _build
    _build.build()
    import bench
    from paper_2606_04238_gb300 import synth, wq
    wq.lib()
    return bench, synth, wq


def _packed(wq, bits, n, k, group):
    cb, mb = wq.packed_sizes(bits, n, k, group)
    return cb + mb


@pytest.mark.parametrize("name", ["qwen3_4b", "dense_8b", "dense_14b"])
@pytest.mark.parametrize("m", [1, 16])
def test_decode_bytes_match_packed_sizes(env, name, m):
    bench, synth, wq = env
    cfg = synth.CONFIGS[name]
    gu, dn = bench.algorithmic_bytes(cfg, m)
    a, bg, bu = synth.lora(cfg.d, cfg.inter, cfg.r, 0)
    lora_bytes = sum(t.numel() * t.element_size() for t in (a, bg, bu))
    acts_gu = (m * cfg.d + m * cfg.inter) * 2              # x in, h out (bf16)
    assert gu == 2 * _packed(wq, 2, cfg.inter, cfg.d, cfg.group_gu) + lora_bytes + acts_gu
    acts_dn = (m * cfg.inter + 2 * m * cfg.d) * 2          # h in, residual in, y out
    assert dn == _packed(wq, 4, cfg.d, cfg.inter, cfg.group_down) + acts_dn
    gu4, _ = bench.algorithmic_bytes(cfg, m, bits_gu=4, lora=False)
    assert gu4 == 2 * _packed(wq, 4, cfg.inter, cfg.d, cfg.group_gu) + acts_gu


def test_qwen3_4b_figures(env):
    """The per-call figures quoted for the Qwen3-4B layer at one token."""
    bench, synth, _ = env
    cfg = synth.CONFIGS["qwen3_4b"]
    gu, dn = bench.algorithmic_bytes(cfg, 1)
    assert gu == 14_819_328 and dn == 13_259_776
    step = cfg.layers * (gu + dn)
    assert abs(step / 1e9 - 1.011) < 0.001
    gu4, _ = bench.algorithmic_bytes(cfg, 1, bits_gu=4, lora=False)
    assert abs(cfg.layers * (gu4 + dn) / 1e9 - 1.431) < 0.001


def test_prefill_flops(env):
    bench, synth, _ = env
    cfg = synth.CONFIGS["dense_14b"]
    m, d, i, r = 512, cfg.d, cfg.inter, cfg.r
    gu, dn = bench.prefill_flops(cfg, m)
    products = [(m, d, i), (m, d, i), (m, d, 2 * r), (m, r, i), (m, r, i)]  # gate, up, x A^T, t_g B_g^T, t_u B_u^T
    assert gu == sum(2 * a * b * c for a, b, c in products)
    assert dn == 2 * m * i * d
    unit = 2 * 128 ** 3
    adapters = 2 * m * d * 2 * r + 2 * 2 * m * r * i
    assert gu == 2 * (m // 128) * (i // 128) * (d // 128) * unit + adapters  # 2 x 4 x 136 x 40 units
    assert gu == 184_012_505_088 and abs((gu + dn) / 1e9 - 275.3) < 0.05


def test_traffic_record_tracks_the_sources(env):
    bench, _, _ = env
    with open(os.path.join(ROOT, "profiles", "dram_traffic.json")) as f:
        rec = json.load(f)
    for kernel, files in (("gateup_w2_lora", bench.GEMV_SOURCES), ("down_w4", bench.GEMV_SOURCES),
                          ("gemm_gateup_w2_m512", bench.GEMM_SOURCES), ("gemm_down_w4_m512", bench.GEMM_SOURCES)):
        e = rec[kernel]
        assert tuple(e["sources"]) == tuple(files)
        want = e["dram_bytes_per_launch"] if e["source_sha"] == bench.source_sha(files) else None
        assert bench.recorded_traffic(kernel, files) == want
        # the same record keyed to other sources is not used
        assert bench.recorded_traffic(kernel, ("wq_dense.cu",)) is None
    assert bench.recorded_traffic("no_such_kernel") is None
