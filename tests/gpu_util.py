"""Helpers of the GPU parity tests: upload oracle-packed weights, compare
bf16 / fp32 outputs with the oracle."""
import numpy as np
import torch

import oracle as orc
from paper_2606_04238_gb300 import synth, wq


def upload_packed(q, s, z, group, bits, dev="cuda"):
    """Oracle quantization -> oracle packing -> device QWeight (oracle to GPU only)."""
    codes, meta = orc.tile_pack(q, s, z, group, bits)
    n, k = q.shape
    return wq.QWeight(torch.from_numpy(codes.view(np.int32)).to(dev), torch.from_numpy(meta.view(np.int16)).to(dev),
                      n, k, group, bits)


def bits_of(t):
    return synth.bf16_bits(t)


def f64_of_bf16(t):
    return t.detach().float().cpu().numpy().astype(np.float64)


def check_bf16(got, ref, what, min_exact=0.97, depth=1):
    """bf16 device output vs fp64 oracle value.

    Bound: max|gpu - oracle| <= 2e-3 (max|oracle| + 1), plus the half-ulp
    rounding of the bf16 store itself (|v| 2^-8 bounds half a bf16 ulp), per
    element.  Also: at least `min_exact` of the elements equal the oracle's
    own bf16 rounding bit for bit (differences only where the fp32 and fp64
    sums straddle a rounding boundary).  `depth` > 1 compares the end of a
    chain of `depth` layers run on their own outputs: each layer's bf16
    rounding flips are carried into the next, so the bound is depth times the
    one-layer bound.
    """
    g = f64_of_bf16(got)
    ref = np.asarray(ref, np.float64)
    assert g.shape == ref.shape, (g.shape, ref.shape)
    if ref.size == 0:
        return
    tol = depth * (2e-3 * (np.abs(ref).max() + 1.0) + np.abs(ref) * 2.0 ** -8)
    err = np.abs(g - ref)
    bad = err > tol
    assert not bad.any(), f"{what}: {bad.sum()} elements out of bound, max err {err.max():.3e} " \
                          f"(tol at worst {tol.flat[np.argmax(err - tol)]:.3e})"
    exact = np.mean(bits_of(got) == orc.f64_to_bf16_bits(ref))
    assert exact >= min_exact, f"{what}: only {exact:.4f} of elements match the oracle's bf16 rounding"


def check_f32(got, ref, what, rel=1e-4):
    g = got.detach().cpu().numpy().astype(np.float64)
    ref = np.asarray(ref, np.float64)
    err = np.abs(g - ref).max() if ref.size else 0.0
    assert err <= rel * max(np.abs(ref).max(), 1e-30), f"{what}: max err {err:.3e} vs max|ref| {np.abs(ref).max():.3e}"
