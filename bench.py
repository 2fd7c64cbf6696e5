"""Decode MLP-stack benchmark of the W4/W2-GateUp block on GB300.

One step = one decode step of m tokens through the whole MLP stack of the
Qwen3-4B-shaped workload (36 layers, d=2560, inter=9728; 2-bit gate/up with
group 128 and LoRA rank 16 on both; 4-bit down with group 128; unit-weight
RMSNorm before each MLP), replayed from a CUDA graph of wq_mlp_forward.
Inputs are seeded synthetic draws of the paper's weight / activation shapes;
the packed weights (1.01 GB per step) are far larger than L2, so no flush is
needed between steps.

Reported besides the step rate: the fused 2-bit gate/up call and the 4-bit
down call timed on their own (36 distinct layers back to back, one graph) for
the HBM roofline, the uniform-W4 stack on the same GPU (speedup, Gain%), the
same stack with the adapters merged into the 2-bit codes, the bf16 down call
of the BF16/W2-GateUp configuration, the end-to-end rate through the C ABI with host buffers, SM clocks sampled during
the timed region, the CPU oracle on a bounded sample, and the prefill leg: a
512-token chunk through 14B-shaped layers (d=5120, inter=17408, LoRA rank 32),
which runs on the tcgen05 dequant-GEMM path, against the tensor roofline.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl wq|reference]
  python bench.py --leg prefill --eager --steps 2 --warmup 1   (launches only, for ncu)
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "decode MLP-stack tokens/s and fused W2 gate/up GEMV HBM GB/s (% of peak) at 1 GB300"
UNIT = "tokens/s"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=50)
    ap.add_argument("--impl", default="wq", choices=["wq", "reference"])
    ap.add_argument("--config", default="qwen3_4b")
    ap.add_argument("--m", type=int, default=1)
    ap.add_argument("--layers", type=int, default=0, help="0: the config's depth")
    ap.add_argument("--no-extras", action="store_true", help="skip the comparator / per-kernel / CPU legs")
    ap.add_argument("--eager", action="store_true",
                    help="profiling aid: run the stack with plain stream launches (no CUDA graph), print no JSON")
    ap.add_argument("--leg", default="decode", choices=["decode", "prefill", "moe", "decoder", "w3", "bf16down"],
                    help="with --eager: which stack to run (the decode stack, the prefill chunk, the MoE stack, "
                         "whole decoder layers at --context, the stack with 3-bit g32 gate/up, or with bf16 down)")
    ap.add_argument("--context", type=int, default=8192, help="with --eager --leg decoder: the KV-cache length")
    ap.add_argument("--prefill-layers", type=int, default=4, help="distinct 14B-shaped layers of the prefill leg")
    ap.add_argument("--sweep", action="store_true",
                    help="instead of the bench line: decode stacks of the 4B/8B/14B shapes over their token counts, "
                         "one JSON line")
    return ap.parse_args()


# --------------------------------------------------------------------------- helpers
def dist_setup(args):
    import torch
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if ws > 1:
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if backend == "nccl":
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
    return ws, rank, local


def barrier(ws):
    if ws > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(v, ws):
    if ws == 1:
        return v
    import torch
    import torch.distributed as dist
    t = torch.tensor([v], dtype=torch.float64, device="cuda" if torch.cuda.is_available() else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


def measured_tensor_peak():
    """Dense bf16 (= binary16) tensor TFLOP/s: the burst figure, for a kernel timed on its own."""
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["bf16_tflops"]), "measured"
    return 1900.0, "fallback"


class ClockSampler:
    """nvidia-smi samples of SM clock / throttle reasons during the timed region."""

    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.file = None

    def start(self):
        try:
            self.file = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.QUERY}",
                                          "--format=csv,noheader,nounits", "-lms", "50"],
                                         stdout=self.file, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"]}
        time.sleep(0.15)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.file.flush()
        rows = []
        with open(self.file.name) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.file.name)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        smax = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower().startswith("active")})
        return {"sm_mhz": float(np.median(sm)) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": reasons, "samples": len(rows)}


# --------------------------------------------------------------------------- byte model
def algorithmic_bytes(cfg, m, bits_gu=2, lora=True):
    """Bytes one decode step must move: packed codes, fp16 scales/zeros, LoRA
    factors, bf16 activations in and out (nothing else)."""
    d, inter, g = cfg.d, cfg.inter, cfg.group_gu
    codes_gu = 2 * inter * d * bits_gu / 8
    meta_gu = 2 * inter * (d // g) * 4
    lora_b = (2 * inter * cfg.r * 2) if lora else 0
    lora_a = (2 * cfg.r * d * 2) if lora else 0
    act_gu = m * d * 2 + m * inter * 2                       # x in, h out
    gateup = codes_gu + meta_gu + lora_a + lora_b + act_gu
    codes_d = d * inter * 4 / 8
    meta_d = d * (inter // cfg.group_down) * 4
    act_d = m * inter * 2 + 2 * m * d * 2                    # h in, residual in, y out
    down = codes_d + meta_d + act_d
    return gateup, down


PREFILL_CONFIG, PREFILL_M = "dense_14b", 512


def prefill_flops(cfg, m):
    """Algorithmic flops of one layer on m tokens: the gate and up products
    with their adapters (x A^T, then t B^T for both), and the down product."""
    gateup = 2 * 2 * m * cfg.d * cfg.inter + 2 * m * cfg.d * 2 * cfg.r + 2 * 2 * m * cfg.r * cfg.inter
    down = 2 * m * cfg.inter * cfg.d
    return gateup, down


GEMV_SOURCES = ("wq_gemv.cu", "wq_ptx.cuh", "wq_internal.h")
GEMM_SOURCES = ("wq_gemm.cu", "wq_ptx.cuh", "wq_internal.h")


def source_sha(files=GEMV_SOURCES):
    h = hashlib.sha256()
    for fn in files:
        with open(os.path.join(ROOT, "paper_2606_04238_gb300", "csrc", fn), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def recorded_traffic(kernel, files=GEMV_SOURCES):
    """DRAM bytes per launch from the committed ncu summary, if the kernel source is unchanged."""
    p = os.path.join(ROOT, "profiles", "dram_traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        d = json.load(f)
    e = d.get(kernel)
    if not e or e.get("source_sha") != source_sha(files):
        return None
    return e.get("dram_bytes_per_launch")


def stack_config(cfg, n_layers, m, ws_):
    """The workload description both arms report."""
    gu_bytes, dn_bytes = algorithmic_bytes(cfg, m)
    return {"workload": f"{cfg.name}_mlp_stack_{n_layers}L_m{m}", "model": f"{cfg.name}-shaped MLP stack",
            "d": cfg.d, "inter": cfg.inter, "layers": n_layers, "m": m, "global_batch": m * ws_,
            "seq_len": 1, "group": cfg.group_gu, "lora_r": cfg.r, "lora_scale": cfg.lora_scale,
            "prenorm": True, "parallelism": f"replicas x{ws_}",
            "l2": f"no flush: {n_layers * (gu_bytes + dn_bytes) / 1e9:.2f} GB of packed weights per step "
                  "(> 129 MB L2)"}


# --------------------------------------------------------------------------- GPU arm
def build_stack(wq, synth, cfg, n_layers, bits_gu, lora, dev):
    import torch
    layers = []
    for l in range(n_layers):
        wg, wu, wd = synth.layer_weights(cfg, l, device=dev)
        kw = {}
        if lora and bits_gu in (2, 3):
            a, bg, bu = synth.lora(cfg.d, cfg.inter, cfg.r, 10_000 + l, device=dev)
            kw = dict(lora_a=a, lora_b_gate=bg, lora_b_up=bu, lora_scale=cfg.lora_scale)
        layers.append(wq.MLPLayer(wq.pack(wg, cfg.group_gu, bits_gu), wq.pack(wu, cfg.group_gu, bits_gu),
                                  wq.pack(wd, cfg.group_down, 4), **kw))
        del wg, wu, wd
    torch.cuda.synchronize()
    return layers


def capture(fn):
    import torch
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        fn()
        fn()
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        fn()
    torch.cuda.synchronize()
    return g


def time_graph(g, steps, warmup, ws_=1, sampler=None, pre=None, post=None):
    """Device time of `steps` replays (CUDA events on the replay stream), max over ranks."""
    import torch
    stream = torch.cuda.current_stream()
    for _ in range(warmup):
        if pre:
            pre()
        g.replay()
        if post:
            post()
    torch.cuda.synchronize()
    barrier(ws_)
    torch.cuda.synchronize()
    if sampler:
        sampler.start()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(steps):
        if pre:
            pre()
        g.replay()
        if post:
            post()
    e1.record(stream)
    torch.cuda.synchronize()
    clocks = sampler.stop() if sampler else None
    barrier(ws_)
    ms = e0.elapsed_time(e1)
    return max_over_ranks(ms, ws_), clocks


def cpu_oracle_sample(cfg, m, target_s=12.0, max_layers=8):
    """The fp64 oracle on the host cores: time a bounded number of the stack's
    layers and scale to the stack's depth (tokens/s of the whole stack)."""
    import oracle as orc
    from paper_2606_04238_gb300 import synth
    x = synth.bf16_bits(synth.activations((m, cfg.d), 2024))
    elapsed, done = 0.0, 0
    for l in range(max_layers):
        wg, wu, wd = synth.layer_weights(cfg, l)
        qg = orc.quantize(wg.numpy(), cfg.group_gu, 2)[:3]
        qu = orc.quantize(wu.numpy(), cfg.group_gu, 2)[:3]
        qd = orc.quantize(wd.numpy(), cfg.group_down, 4)[:3]
        a, bg, bu = synth.lora(cfg.d, cfg.inter, cfg.r, 10_000 + l)
        t0 = time.perf_counter()
        _, hb = orc.gateup(x, qg, qu, cfg.group_gu, synth.bf16_bits(a), synth.bf16_bits(bg), synth.bf16_bits(bu),
                           cfg.lora_scale, prenorm=True)
        _, x = orc.down(hb, qd, cfg.group_down, x)
        elapsed += time.perf_counter() - t0
        done += 1
        if elapsed >= target_s:
            break
    per_layer = elapsed / done
    return {"value": m / (per_layer * cfg.layers), "unit": UNIT, "cores": orc.threads(), "kind": "oracle",
            "sample": f"{done} of {cfg.layers} layers at m={m} (fp64 C oracle, OpenMP), scaled to the full stack; "
                      f"{per_layer * 1e3:.1f} ms per layer"}


def run_gpu(args):
    import torch
    from paper_2606_04238_gb300 import synth, wq

    ws_, rank, local = dist_setup(args)
    import __graft_entry__
    if rank == 0 or not os.path.exists(wq.library_path()):
        __graft_entry__.build()
    barrier(ws_)
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    cfg = synth.CONFIGS[args.config]
    n_layers = args.layers or cfg.layers
    m = args.m
    steps, warmup = max(1, args.steps), max(3, args.warmup)
    if args.eager and args.leg == "prefill":
        run_prefill(wq, synth, dev, args.prefill_layers, steps, warmup, eager=True)
        return
    if args.eager and args.leg in ("moe", "decoder"):
        run_eager_leg(args, wq, synth, dev, steps, warmup)
        return
    if args.sweep:
        print(json.dumps(run_sweep(wq, synth, dev, min(steps, 200), warmup)))
        return

    if args.eager and args.leg == "w3":
        import dataclasses
        layers = build_stack(wq, synth, dataclasses.replace(cfg, group_gu=32), n_layers, 3, True, dev)
    else:
        layers = build_stack(wq, synth, cfg, n_layers, 2, True, dev)
    if args.eager and args.leg == "bf16down":
        layers = [wq.MLPLayer(L.gate, L.up, wq.dense_weight(synth.weights((cfg.d, cfg.inter), 3 * l + 2, device=dev)
                                                             .to(torch.bfloat16)),
                              lora_a=L.lora_a, lora_b_gate=L.lora_b_gate, lora_b_up=L.lora_b_up,
                              lora_scale=L.lora_scale) for l, L in enumerate(layers)]
    table = wq.LayerTable(layers)
    ws = wq.workspace(m, cfg.d, cfg.inter, cfg.r)
    x = synth.activations((m, cfg.d), 2024 + rank, device=dev)
    y = torch.empty_like(x)
    if args.eager:
        # for ncu: the same launches as one step, issued eagerly
        for _ in range(warmup + steps):
            wq.mlp_forward(x, layers, prenorm=True, y=y, ws=ws, table=table)
        torch.cuda.synchronize()
        assert wq.device_status() == 0
        print(f"eager: {warmup + steps} stack steps of {n_layers} layers done", flush=True)
        return
    g = capture(lambda: wq.mlp_forward(x, layers, prenorm=True, y=y, ws=ws, table=table))
    sampler = ClockSampler(local)
    ms, clocks = time_graph(g, steps, warmup, ws_, sampler)
    ms_step = ms / steps
    value = ws_ * m * steps / (ms / 1e3)
    launches_per_step = 2 * n_layers + 1  # first layer's input statistics, then gate/up and down per layer

    # end to end through the C ABI with host buffers: H2D of x, the stack, D2H of y
    xh = torch.empty((m, cfg.d), dtype=torch.bfloat16).pin_memory()
    xh.copy_(x.cpu())
    yh = torch.empty((m, cfg.d), dtype=torch.bfloat16).pin_memory()
    xd = torch.empty_like(x)

    def e2e_step():
        xd.copy_(xh, non_blocking=True)
        wq.mlp_forward(xd, layers, prenorm=True, y=y, ws=ws, table=table)
        yh.copy_(y, non_blocking=True)

    ge = capture(e2e_step)
    ms_e2e, _ = time_graph(ge, steps, warmup, ws_)
    e2e = {"value": ws_ * m * steps / (ms_e2e / 1e3), "unit": UNIT, "h2d_bytes_per_step": xh.numel() * 2,
           "d2h_bytes_per_step": yh.numel() * 2,
           "path": "pinned host x -> cudaMemcpyAsync -> wq_mlp_forward -> cudaMemcpyAsync -> pinned host y, "
                   "in one CUDA graph per step"}

    peak, peak_src = measured_peaks()
    gu_bytes, dn_bytes = algorithmic_bytes(cfg, m)
    out = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws_, "steps": steps, "warmup": warmup,
           "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
           "dtype": "w2/w4 codes x f16 mma, f32 accumulate, bf16 activations", "data": "synthetic",
           "config": stack_config(cfg, n_layers, m, ws_),
           "route": ("launch chain", "dequant-GEMM chain", "single-launch stack kernel")[
               wq.mlp_forward_info(m, layers, table=table)["route"]],
           "gpu_launches": launches_per_step * steps, "clocks": clocks, "e2e": e2e,
           "stack_gbs": n_layers * (gu_bytes + dn_bytes) / (ms_step / 1e3) / 1e9}

    if not args.no_extras and rank == 0:
        # per-kernel chains: 36 distinct layers back to back (PDL), for the roofline
        h = torch.empty((m, cfg.inter), dtype=torch.bfloat16, device=dev)
        yk = torch.empty_like(x)

        def gu_chain():
            for L in layers:
                wq.gateup_w2_lora(x, L.gate, L.up, L.lora_a, L.lora_b_gate, L.lora_b_up, L.lora_scale, prenorm=True,
                                  h=h, ws=ws)

        def dn_chain():
            for L in layers:
                wq.down_w4(h, L.down, residual=x, y=yk, ws=ws)

        ks = max(20, steps // 4)
        ms_gu, _ = time_graph(capture(gu_chain), ks, warmup)
        ms_dn, _ = time_graph(capture(dn_chain), ks, warmup)
        t_gu = ms_gu / ks / n_layers / 1e3
        t_dn = ms_dn / ks / n_layers / 1e3
        gu_gbs, dn_gbs = gu_bytes / t_gu / 1e9, dn_bytes / t_dn / 1e9
        tr = recorded_traffic("gateup_w2_lora")
        out["roofline"] = {"bound": "hbm", "achieved": gu_gbs, "peak": peak, "unit": "GB/s", "frac": gu_gbs / peak,
                           "traffic": tr, "kernel": "wq_gateup_w2_lora (first-layer tile-partials kernel + fused 2-bit gate/up GEMV)",
                           "algorithmic_bytes_per_launch": gu_bytes, "us_per_launch": t_gu * 1e6,
                           "peak_source": f"{peak_src} HBM copy bandwidth (MEASURED_PEAKS.json hbm_gbs)"}
        out["kernels"] = {
            "gateup_w2_lora": {"us": t_gu * 1e6, "gbs": gu_gbs, "frac": gu_gbs / peak, "bytes": gu_bytes},
            "down_w4": {"us": t_dn * 1e6, "gbs": dn_gbs, "frac": dn_gbs / peak, "bytes": dn_bytes,
                        "traffic": recorded_traffic("down_w4")},
        }

        # the bf16 down layer of the BF16/W2-GateUp configuration (Sec. 6.1), 36 distinct matrices back to back
        wdb = [synth.weights((cfg.d, cfg.inter), 3 * l + 2, device=dev).to(torch.bfloat16) for l in range(n_layers)]

        def bd_chain():
            for W in wdb:
                wq.down_bf16(h, W, residual=x, y=yk)

        ms_bd, _ = time_graph(capture(bd_chain), ks, warmup)
        t_bd = ms_bd / ks / n_layers / 1e3
        bd_bytes = cfg.d * cfg.inter * 2 + m * cfg.inter * 2 + 2 * m * cfg.d * 2
        out["kernels"]["down_bf16"] = {"us": t_bd * 1e6, "gbs": bd_bytes / t_bd / 1e9,
                                       "frac": bd_bytes / t_bd / 1e9 / peak, "bytes": bd_bytes,
                                       "note": "bf16 down of the BF16/W2-GateUp configuration (wq_down_bf16)"}
        del wdb
        # the uniform-W4 comparator stack (same workload, 4-bit gate/up, no adapter)
        del g, ge
        w4 = build_stack(wq, synth, cfg, n_layers, 4, False, dev)
        t4 = wq.LayerTable(w4)
        g4 = capture(lambda: wq.mlp_forward(x, w4, prenorm=True, y=y, ws=ws, table=t4))
        ms4, _ = time_graph(g4, steps, warmup)
        tps4 = m * steps / (ms4 / 1e3)
        tps = value / ws_
        out["w4_uniform"] = {"tokens_per_s": tps4, "ms_per_step": ms4 / steps,
                             "speedup_w4w2_over_w4": tps / tps4, "gain_pct": 100.0 * (tps - tps4) / tps4,
                             "paper_gain_pct_context": "7.5-23.3% whole-model TPS, LIFE roofline model on "
                                                       "Device A (50 TOPs, 100 GB/s) / Device B (200 GB/s)"}
        del w4, g4
        # the same stack with each layer's adapters merged into new 2-bit codes (wq_merge_lora; Sec. 4.2
        # and Sec. 7 step 5 allow either form): no adapter bytes and no LoRA stages on the decode path
        wm = torch.empty((cfg.inter, cfg.d), dtype=torch.float32, device=dev)
        merged = [wq.merge_layer(L, w_merged=wm) for L in layers]
        del wm
        tmg = wq.LayerTable(merged)
        gmg = capture(lambda: wq.mlp_forward(x, merged, prenorm=True, y=y, ws=ws, table=tmg))
        msm, _ = time_graph(gmg, steps, warmup)
        tpsm = m * steps / (msm / 1e3)
        out["merged_adapters"] = {"tokens_per_s": tpsm, "ms_per_step": msm / steps, "vs_unmerged": tpsm / tps,
                                  "algorithmic_gb_per_step": n_layers * sum(algorithmic_bytes(cfg, m, lora=False)) / 1e9,
                                  "note": "adapters merged into the 2-bit codes and requantized; r = 0 at decode"}
        del merged, tmg, gmg
        # the BF16/W2-GateUp configuration (Sec. 6.1): the same 2-bit gate/up and adapters, a dense bf16 down
        bdl = [wq.MLPLayer(L.gate, L.up, wq.dense_weight(synth.weights((cfg.d, cfg.inter), 3 * l + 2, device=dev)
                                                          .to(torch.bfloat16)),
                           lora_a=L.lora_a, lora_b_gate=L.lora_b_gate, lora_b_up=L.lora_b_up, lora_scale=L.lora_scale)
               for l, L in enumerate(layers)]
        tbd = wq.LayerTable(bdl)
        gbd = capture(lambda: wq.mlp_forward(x, bdl, prenorm=True, y=y, ws=ws, table=tbd))
        msb, _ = time_graph(gbd, steps, warmup)
        tpsb = m * steps / (msb / 1e3)
        bd_gb = n_layers * (gu_bytes + cfg.d * cfg.inter * 2 + m * cfg.inter * 2 + 2 * m * cfg.d * 2) / 1e9
        out["bf16_down_stack"] = {"tokens_per_s": tpsb, "ms_per_step": msb / steps, "vs_w4_down": tpsb / tps,
                                  "algorithmic_gb_per_step": bd_gb,
                                  "stack_gbs": bd_gb / (msb / steps / 1e3), "frac_of_hbm": bd_gb / (msb / steps / 1e3) / peak,
                                  "note": "BF16/W2-GateUp: 2-bit gate/up with the adapters, dense bf16 down "
                                          "(wq_mlp_forward with bits-16 down weights)"}
        del bdl, tbd, gbd
        torch.cuda.empty_cache()
        out["quant_settings"] = run_quant_settings(wq, synth, dev, cfg, n_layers, m, x, y, ws, steps, warmup, peak)
        torch.cuda.empty_cache()
        out["prefill"] = run_prefill(wq, synth, dev, args.prefill_layers, max(20, min(steps, 200)), warmup)
        torch.cuda.empty_cache()
        out["decoder_layer"] = run_decoder(wq, synth, dev, max(10, min(steps, 50)), warmup)
        out["sweep"] = run_sweep(wq, synth, dev, max(10, min(steps, 50)), warmup, BENCH_SWEEP)["rows"]
        torch.cuda.empty_cache()
        out["moe"] = run_moe(wq, synth, dev, max(10, min(steps, 50)), warmup, peak)
        out["cpu_baseline"] = cpu_oracle_sample(cfg, m)

    if rank == 0:
        print(json.dumps(out))
    barrier(ws_)


SWEEP = (("qwen3_4b", (1, 2, 4, 8, 16, 32, 64)), ("dense_8b", (1, 4, 16, 32, 64)), ("dense_14b", (1, 16, 64)))
# the decode token counts of the benchmark configurations (4B stack, 8B and 14B stacks), in the bench line
BENCH_SWEEP = (("qwen3_4b", (2, 4, 8, 16)), ("dense_8b", (1, 4, 16, 64)), ("dense_14b", (1, 16, 64)))


def run_sweep(wq, synth, dev, steps, warmup, sweep=SWEEP):
    """Decode MLP stacks of the 4B, 8B and 14B shapes (all layers, W2 gate/up
    + LoRA, W4 down, RMSNorm) at their token counts: tokens/s, µs per step and
    the stack's algorithmic bytes per step over the measured HBM bandwidth."""
    import torch
    peak, src = measured_peaks()
    out = {"metric": "decode MLP-stack tokens/s over token counts", "peak_gbs": peak, "peak_source": src,
           "data": "synthetic", "rows": []}
    for name, ms in sweep:
        cfg = synth.CONFIGS[name]
        layers = build_stack(wq, synth, cfg, cfg.layers, 2, True, dev)
        table = wq.LayerTable(layers)
        for m in ms:
            ws = wq.workspace(m, cfg.d, cfg.inter, cfg.r)
            x = synth.activations((m, cfg.d), 4096 + m, device=dev)
            y = torch.empty_like(x)
            g = capture(lambda: wq.mlp_forward(x, layers, prenorm=True, y=y, ws=ws, table=table))
            ms_tot, clocks = time_graph(g, steps, warmup, 1, ClockSampler(dev.index or 0))
            t_step = ms_tot / steps / 1e3
            gu, dn = algorithmic_bytes(cfg, m)
            gbs = cfg.layers * (gu + dn) / t_step / 1e9
            out["rows"].append({"config": name, "layers": cfg.layers, "m": m,
                                "route": ("launch chain", "dequant-GEMM chain", "single-launch stack kernel")[
                                    wq.mlp_forward_info(m, layers, table=table)["route"]],
                                "tokens_per_s": m / t_step,
                                "us_per_step": t_step * 1e6, "us_per_layer": t_step * 1e6 / cfg.layers,
                                "stack_gbs": gbs, "frac_of_hbm": gbs / peak, "clocks": clocks})
            assert wq.device_status() == 0
            del g, ws, x, y
        del layers, table
        torch.cuda.empty_cache()
    return out


def run_prefill(wq, synth, dev, n_layers, steps, warmup, eager=False):
    """A 512-token chunk through n_layers distinct 14B-shaped layers (the
    tcgen05 dequant-GEMM path): whole-stack rate, then the gate/up and the
    down calls timed on their own for the tensor roofline."""
    import torch
    cfg = synth.CONFIGS[PREFILL_CONFIG]
    m = PREFILL_M
    layers = build_stack(wq, synth, cfg, n_layers, 2, True, dev)
    ws = wq.workspace(m, cfg.d, cfg.inter, cfg.r)
    x = synth.activations((m, cfg.d), 512, device=dev)
    y = torch.empty_like(x)

    def stack():
        wq.mlp_forward(x, layers, prenorm=True, y=y, ws=ws)

    if eager:
        for _ in range(warmup + steps):
            stack()
        torch.cuda.synchronize()
        assert wq.device_status() == 0
        print(f"eager: {warmup + steps} prefill steps of {n_layers} layers done", flush=True)
        return None
    ms, clocks = time_graph(capture(stack), steps, warmup, 1, ClockSampler(dev.index or 0))
    h = torch.empty((m, cfg.inter), dtype=torch.bfloat16, device=dev)
    yk = torch.empty_like(x)

    def gu_chain():
        for L in layers:
            wq.gateup_w2_lora(x, L.gate, L.up, L.lora_a, L.lora_b_gate, L.lora_b_up, L.lora_scale, prenorm=True,
                              h=h, ws=ws)

    def dn_chain():
        for L in layers:
            wq.down_w4(h, L.down, residual=x, y=yk, ws=ws)

    ms_gu, _ = time_graph(capture(gu_chain), steps, warmup)
    ms_dn, _ = time_graph(capture(dn_chain), steps, warmup)
    assert wq.device_status() == 0
    f_gu, f_dn = prefill_flops(cfg, m)
    t_layer = ms / steps / n_layers / 1e3
    t_gu = ms_gu / steps / n_layers / 1e3
    t_dn = ms_dn / steps / n_layers / 1e3
    peak, src = measured_tensor_peak()
    gu_tf, dn_tf = f_gu / t_gu / 1e12, f_dn / t_dn / 1e12
    wbytes = sum(algorithmic_bytes(cfg, m)) - (m * cfg.d * 2 * 3 + m * cfg.inter * 2 * 2)
    return {
        "workload": f"{cfg.name}_prefill_stack_{n_layers}L_m{m}",
        "config": {"d": cfg.d, "inter": cfg.inter, "layers": n_layers, "m": m, "group": cfg.group_gu,
                   "lora_r": cfg.r, "prenorm": True,
                   "l2": f"no flush: {n_layers * wbytes / 1e9:.2f} GB of packed weights per step (> 129 MB L2)"},
        "tokens_per_s": m * steps / (ms / 1e3), "us_per_layer": t_layer * 1e6,
        "tflops": (f_gu + f_dn) / t_layer / 1e12, "flops_per_layer": f_gu + f_dn,
        "dtype": "binary16 x binary16 tcgen05.mma, fp32 TMEM accumulate (weights dequantized to binary16)",
        "clocks": clocks,
        "roofline": {"bound": "tensor", "achieved": gu_tf, "peak": peak, "unit": "TFLOP/s", "frac": gu_tf / peak,
                     "traffic": recorded_traffic("gemm_gateup_w2_m512", GEMM_SOURCES),
                     "kernel": "wq_gateup_w2_lora at m=512 (input kernel + tcgen05 dequant-GEMM)",
                     "algorithmic_flops_per_launch": f_gu, "us_per_launch": t_gu * 1e6,
                     "peak_source": f"{src} dense bf16 burst (MEASURED_PEAKS.json bf16_tflops)"},
        "kernels": {"gateup_w2_lora": {"us": t_gu * 1e6, "tflops": gu_tf, "frac": gu_tf / peak, "flops": f_gu},
                    "down_w4": {"us": t_dn * 1e6, "tflops": dn_tf, "frac": dn_tf / peak, "flops": f_dn,
                                "traffic": recorded_traffic("gemm_down_w4_m512", GEMM_SOURCES)}},
    }


DECODER_CONTEXTS = (1024, 8192, 32768)
DECODER_HEADS = (32, 8, 128)  # query heads, kv heads, head_dim of the Qwen3-4B attention


def run_decoder(wq, synth, dev, steps, warmup, n_layers=None, contexts=DECODER_CONTEXTS, batch=1):
    """One decode step through whole decoder layers of the Qwen3-4B shape
    (4-bit q/k/v/o projections, grouped-query attention over a bf16 KV cache,
    then the MLP block) at several context lengths, with the MLP at
    W4/W2-GateUp (2-bit gate/up + LoRA) and at uniform W4: the decode rate and
    the gain of the 2-bit gate/up over context (the attention's cache reads
    grow with the context while the MLP's bytes stay fixed)."""
    import torch
    cfg = synth.CONFIGS["qwen3_4b"]
    n_layers = n_layers or cfg.layers
    H, Hkv, hd = DECODER_HEADS
    max_ctx = max(contexts)
    attn, caches, mlps = [], [], {2: [], 4: []}
    for l in range(n_layers):
        wqkv = synth.weights(((H + 2 * Hkv) * hd, cfg.d), 7000 + 2 * l, device=dev)
        wo = synth.weights((cfg.d, H * hd), 7001 + 2 * l, device=dev)
        attn.append((wq.pack(wqkv, 128, 4), wq.pack(wo, 128, 4)))
        del wqkv, wo
        g = torch.Generator(device=dev)
        g.manual_seed(9000 + l)
        kc = torch.randn((batch, Hkv, max_ctx, hd), generator=g, device=dev).to(torch.bfloat16)
        vc = torch.randn((batch, Hkv, max_ctx, hd), generator=g, device=dev).to(torch.bfloat16)
        caches.append((kc, vc))
    for bits in (2, 4):
        mlps[bits] = build_stack(wq, synth, cfg, n_layers, bits, bits == 2, dev)
    wm = torch.empty((cfg.inter, cfg.d), dtype=torch.float32, device=dev)
    mlps["merged"] = [wq.merge_layer(L, w_merged=wm) for L in mlps[2]]  # 2-bit codes, adapters merged (r = 0)
    del wm
    x = synth.activations((batch, cfg.d), 77, device=dev)
    bufs = [torch.empty_like(x) for _ in range(2)]
    rows = []
    for ctx in contexts:
        lens = torch.full((batch,), ctx - 1, dtype=torch.int32, device=dev)
        row = {"context": ctx}
        for bits, name in ((4, "w4"), (2, "w4w2_gateup"), ("merged", "w4w2_gateup_merged")):
            layers = [wq.DecoderLayer(attn[l][0], attn[l][1], mlps[bits][l], H, Hkv, hd) for l in range(n_layers)]
            cls = [L.c() for L in layers]
            ws = wq.decoder_workspace(batch, layers[0], max_ctx)

            def step():
                cur = x
                for l in range(n_layers):
                    out = bufs[l & 1]
                    wq.decoder_layer_forward(cur, lens, layers[l], caches[l][0], caches[l][1], y=out, ws=ws, c_layer=cls[l])
                    cur = out

            ms, _ = time_graph(capture(step), steps, warmup)
            assert wq.device_status() == 0
            t = ms / steps / 1e3
            row[name] = {"tokens_per_s": batch / t, "us_per_layer": t * 1e6 / n_layers}
            del ws
        row["gain_pct"] = 100.0 * (row["w4w2_gateup"]["tokens_per_s"] / row["w4"]["tokens_per_s"] - 1.0)
        row["gain_pct_merged"] = 100.0 * (row["w4w2_gateup_merged"]["tokens_per_s"] / row["w4"]["tokens_per_s"] - 1.0)
        rows.append(row)
    del caches, mlps, attn
    torch.cuda.empty_cache()
    return {"workload": f"qwen3_4b_decoder_{n_layers}L_b{batch}", "heads": {"q": H, "kv": Hkv, "head_dim": hd},
            "kv_cache": "bf16, random N(0, 1) contents up to the context",
            "rows": rows,
            "note": "one decode step through whole decoder layers (attention projections 4-bit g128; the MLP as "
                    "standalone gate/up and down calls): uniform W4 (no adapter), W4/W2-GateUp with the unmerged "
                    "rank-16 adapter, and W4/W2-GateUp with the adapter merged into the 2-bit codes; gain_pct and "
                    "gain_pct_merged are the decode-rate gains of the last two over uniform W4"}


# gate/up quantization settings of the same stack: the headline W2 g128, the paper's W2 g32 (Sec. 4.1; its
# scales and zeros cost 1 bit a weight), App. B's W3 g32, and the uniform W4 g128 comparator
QUANT_SETTINGS = ((2, 128, True), (2, 32, True), (3, 32, True), (4, 128, False))


def run_quant_settings(wq, synth, dev, cfg, n_layers, m, x, y, ws, steps, warmup, peak):
    """The decode stack (same workload, 4-bit g128 down) with each gate/up setting: rate, bytes a step and the
    fraction of HBM bandwidth those bytes take at that rate."""
    import dataclasses

    import torch
    rows = []
    for bits, g, lora in QUANT_SETTINGS:
        c2 = dataclasses.replace(cfg, group_gu=g)
        layers = build_stack(wq, synth, c2, n_layers, bits, lora, dev)
        table = wq.LayerTable(layers)
        gr = capture(lambda: wq.mlp_forward(x, layers, prenorm=True, y=y, ws=ws, table=table))
        ms, _ = time_graph(gr, steps, warmup)
        assert wq.device_status() == 0
        gu, dn = algorithmic_bytes(c2, m, bits, lora)
        t = ms / steps / 1e3
        gb = n_layers * (gu + dn) / 1e9
        rows.append({"gate_up": f"W{bits} g{g}" + (" + LoRA r" + str(cfg.r) if lora else ""),
                     "tokens_per_s": m / t, "us_per_layer": t * 1e6 / n_layers, "gb_per_step": gb,
                     "frac_of_hbm": gb / t / peak,
                     "route": ("launch chain", "dequant-GEMM chain", "single-launch stack kernel")[
                         wq.mlp_forward_info(m, layers, table=table)["route"]]})
        del layers, table, gr
        torch.cuda.empty_cache()
    return {"workload": f"{cfg.name}_stack_{n_layers}L_m{m}", "down": f"W4 g{cfg.group_down}", "rows": rows}


# GPT-OSS-20B-shaped MoE MLP (Sec. 5's MoE model): hidden 2880, 32 experts of width 2880, top-4, 24 layers,
# groups of 64 (the paper's INT4 g64 setting for this model)
MOE_SHAPE = dict(d=2880, inter=2880, experts=32, top_k=4, layers=24, group=64, r=16, lora_scale=2.0)


def run_moe(wq, synth, dev, steps, warmup, peak, shape=MOE_SHAPE, m=1):
    """One decode step through a stack of MoE MLP blocks at W4/W2-GateUp (2-bit
    gate/up experts with rank-16 adapters, 4-bit down) and at uniform W4: the
    decode rate, the bytes the selected experts move per token, and the gain of
    the 2-bit gate/up when routing leaves most experts unread."""
    import torch
    d, inter, E, k, L, g, r = (shape[key] for key in ("d", "inter", "experts", "top_k", "layers", "group", "r"))
    x = synth.activations((m, d), 31, device=dev)
    logits = [synth.weights((m, E), 8000 + l, std=1.0, device=dev) for l in range(L)]
    out = {"workload": f"gpt_oss_20b_moe_{L}L_m{m}", "d": d, "expert_width": inter, "experts": E, "top_k": k,
           "group": g, "lora_rank": r,
           "routing": "fixed seeded N(0, 1) router logits per layer (top-4 of 32 experts)"}
    for bits, name in ((2, "w4w2_gateup"), (4, "w4")):
        blocks = []
        for l in range(L):
            wg = synth.weights((E * inter, d), 50_000 + 3 * l, device=dev)
            wu = synth.weights((E * inter, d), 50_001 + 3 * l, device=dev)
            wd = synth.weights((E * d, inter), 50_002 + 3 * l, device=dev)
            kw = {}
            if bits == 2:
                _, bg, bu = synth.lora(d, E * inter, r, 60_000 + l, device=dev)
                a = synth.weights((E * 2 * r, d), 61_000 + l, std=0.01, device=dev).to(torch.bfloat16)
                kw = dict(lora_a=a, lora_b_gate=bg, lora_b_up=bu, lora_scale=shape["lora_scale"])
            ex = wq.MLPLayer(wq.pack(wg, g, bits), wq.pack(wu, g, bits), wq.pack(wd, g, 4), **kw)
            blocks.append(wq.MoELayer(ex, E, k))
            del wg, wu, wd
        cls = [b.c() for b in blocks]
        ws = wq.moe_workspace(m, blocks[0])
        bufs = [torch.empty_like(x) for _ in range(2)]

        def step():
            cur = x
            for l in range(L):
                o = bufs[l & 1]
                wq.moe_forward(cur, logits[l], blocks[l], y=o, ws=ws, c_layer=cls[l])
                cur = o

        ms, _ = time_graph(capture(step), steps, warmup)
        assert wq.device_status() == 0
        t = ms / steps / 1e3
        # bytes of one expert: packed gate, up, down, the adapter's rows; times the experts a token selects
        ex0 = blocks[0].experts
        per_expert = (ex0.gate.nbytes + ex0.up.nbytes + ex0.down.nbytes) / E
        if bits == 2:
            per_expert += (2 * r * d + 2 * inter * r) * 2
        active = L * m * k * per_expert  # an upper bound when tokens share experts
        out[name] = {"tokens_per_s": m / t, "us_per_layer": t * 1e6 / L, "active_gb_per_step": active / 1e9,
                     "gbs": active / t / 1e9, "frac_of_hbm": active / t / 1e9 / peak,
                     "all_experts_gb": L * per_expert * E / 1e9}
        del blocks, cls, ws
        torch.cuda.empty_cache()
    out["gain_pct"] = 100.0 * (out["w4w2_gateup"]["tokens_per_s"] / out["w4"]["tokens_per_s"] - 1.0)
    out["byte_ratio_w4_over_w4w2"] = out["w4"]["active_gb_per_step"] / out["w4w2_gateup"]["active_gb_per_step"]
    out["note"] = ("wq_moe_forward per layer (routing + tile partials, gate/up and down over the selected "
                   "experts' slots, combine): only the k selected experts' weights are read")
    return out


def run_eager_leg(args, wq, synth, dev, steps, warmup):
    """Profiling aid (--eager): the MoE stack or whole decoder layers issued with plain stream launches."""
    import torch
    n = args.layers or 2
    m = args.m
    if args.leg == "moe":
        sh = MOE_SHAPE
        d, inter, E, k, g, r = (sh[key] for key in ("d", "inter", "experts", "top_k", "group", "r"))
        blocks = []
        for l in range(n):
            _, bg, bu = synth.lora(d, E * inter, r, 60_000 + l, device=dev)
            a = synth.weights((E * 2 * r, d), 61_000 + l, std=0.01, device=dev).to(torch.bfloat16)
            ex = wq.MLPLayer(wq.pack(synth.weights((E * inter, d), 50_000 + 3 * l, device=dev), g, 2),
                             wq.pack(synth.weights((E * inter, d), 50_001 + 3 * l, device=dev), g, 2),
                             wq.pack(synth.weights((E * d, inter), 50_002 + 3 * l, device=dev), g, 4),
                             lora_a=a, lora_b_gate=bg, lora_b_up=bu, lora_scale=sh["lora_scale"])
            blocks.append(wq.MoELayer(ex, E, k))
        logits = [synth.weights((m, E), 8000 + l, std=1.0, device=dev) for l in range(n)]
        x = synth.activations((m, d), 31, device=dev)
        ws = wq.moe_workspace(m, blocks[0])

        def step():
            cur = x
            for l in range(n):
                cur = wq.moe_forward(cur, logits[l], blocks[l], ws=ws)
    else:
        cfg = synth.CONFIGS["qwen3_4b"]
        H, Hkv, hd = DECODER_HEADS
        layers = build_stack(wq, synth, cfg, n, 2, True, dev)
        dl, caches = [], []
        for l in range(n):
            wqkv = synth.weights(((H + 2 * Hkv) * hd, cfg.d), 7000 + 2 * l, device=dev)
            wo = synth.weights((cfg.d, H * hd), 7001 + 2 * l, device=dev)
            dl.append(wq.DecoderLayer(wq.pack(wqkv, 128, 4), wq.pack(wo, 128, 4), layers[l], H, Hkv, hd))
            gen = torch.Generator(device=dev)
            gen.manual_seed(9000 + l)
            caches.append(tuple(torch.randn((m, Hkv, args.context, hd), generator=gen, device=dev)
                                .to(torch.bfloat16) for _ in range(2)))
        lens = torch.full((m,), args.context - 1, dtype=torch.int32, device=dev)
        x = synth.activations((m, cfg.d), 77, device=dev)
        ws = wq.decoder_workspace(m, dl[0], args.context)

        def step():
            cur = x
            for l in range(n):
                cur = wq.decoder_layer_forward(cur, lens, dl[l], caches[l][0], caches[l][1], ws=ws)
    for _ in range(warmup + steps):
        step()
    torch.cuda.synchronize()
    assert wq.device_status() == 0
    print(f"eager: {warmup + steps} {args.leg} steps of {n} layers done", flush=True)


# --------------------------------------------------------------------------- reference arm
def run_reference(args):
    """The oracle as it stands, on the host cores: each timed step is one layer
    of the stack (a bounded sample; ms_per_step is that measured time); the
    rate is the whole stack's, m / (layers x the time a step)."""
    ws_ = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    import oracle as orc
    from paper_2606_04238_gb300 import synth
    orc.build()
    cfg = synth.CONFIGS[args.config]
    m = args.m
    n_layers = args.layers or cfg.layers
    nprep = min(4, max(1, args.steps + args.warmup))
    prepared = []
    for l in range(nprep):
        wg, wu, wd = synth.layer_weights(cfg, l)
        a, bg, bu = synth.lora(cfg.d, cfg.inter, cfg.r, 10_000 + l)
        prepared.append((orc.quantize(wg.numpy(), cfg.group_gu, 2)[:3], orc.quantize(wu.numpy(), cfg.group_gu, 2)[:3],
                         orc.quantize(wd.numpy(), cfg.group_down, 4)[:3], synth.bf16_bits(a), synth.bf16_bits(bg),
                         synth.bf16_bits(bu)))
    x = synth.bf16_bits(synth.activations((m, cfg.d), 2024))

    def step(i, x):
        qg, qu, qd, a, bg, bu = prepared[i % nprep]
        _, hb = orc.gateup(x, qg, qu, cfg.group_gu, a, bg, bu, cfg.lora_scale, prenorm=True)
        return orc.down(hb, qd, cfg.group_down, x)[1]

    for i in range(max(0, args.warmup)):
        x = step(i, x)
    t0 = time.perf_counter()
    for i in range(args.steps):
        x = step(i, x)
    el = time.perf_counter() - t0
    per_layer = el / max(1, args.steps)
    value = m / (per_layer * n_layers)
    sample = (f"each timed step is 1 of the {n_layers} layers at m={m} (fp64 C oracle, OpenMP, {nprep} distinct "
              f"layers cycled); value = m / ({n_layers} x the measured time a step); {per_layer * 1e3:.1f} ms a step")
    print(json.dumps({"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws_,
                      "steps": args.steps, "warmup": args.warmup, "ms_per_step": per_layer * 1e3,
                      "step_unit": f"one layer of the {n_layers}-layer stack",
                      "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
                      "data": "synthetic", "config": stack_config(cfg, n_layers, m, ws_),
                      "cpu_baseline": {"value": value, "unit": UNIT, "cores": orc.threads(), "kind": "oracle",
                                       "sample": sample},
                      "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}))


def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
