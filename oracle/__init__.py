"""CPU oracle for the W4/W2-GateUp decode MLP path (plain C, fp64).

TEST INFRASTRUCTURE.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
package.  The product path (``paper_2606_04238_gb300``) never imports it and
shares no code with it.

What it computes (paper sections cited in ``wq_oracle.c``):
  * ``quantize``   Stage-1 group-wise asymmetric min-max RTN (Sec. 4.1), fp32,
                   bit-exact definition of codes / scales / zeros.
  * ``tile_pack``  the packed storage format (byte layout definition).
  * ``gateup``     g,u = x W^T + alpha (x A^T) B^T (Eq. 1) on the dequantized
                   gate/up weights, h = SiLU(g) * u (Sec. 3.3), fp64.
  * ``down``       y = residual + h Wd^T on the dequantized 4-bit down weights.
  * ``rms_scale``  unit-weight RMSNorm scale 1/sqrt(mean(x^2)+eps) per token.
  * ``down_bf16``  y = residual + h Wd^T with a bf16 Wd (the BF16/W2-GateUp
                   configuration of the accuracy experiments, Sec. 6.1), fp64.
  * ``rope`` / ``attn_decode``  rotary embedding and one decode step of
                   grouped-query attention over a bf16 KV cache (the rest of
                   a decoder layer around the MLP), fp64.
  * ``qproj``      unrounded fp64 inputs through a quantized matrix.
  * ``decoder``    (module) one decode step of a whole decoder layer composed
                   from the functions here; ``moe`` (module) a mixture-of-
                   experts MLP block composed from ``gateup`` and ``down``.
  * ``merge_lora`` the merged matrix deq(W) + alpha B A (Eq. 1; Sec. 4.2 lets
                   the adapters be merged after training), fp64 then one
                   rounding to fp32, ready to be quantized again.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "wq_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "liboracle.so")
_lock = threading.Lock()
_lib = None

RMS_EPS = 1e-6


def compile_source(src: str, out: str) -> str:
    """gcc with IEEE arithmetic (no fast-math, no FMA contraction) -> shared library ``out``."""
    tmp = out + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fopenmp", "-ffp-contract=off", "-fno-fast-math",
           "-fPIC", "-shared", "-o", tmp, src, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, out)
    return out


def build(force: bool = False) -> str:
    """Compile the oracle (see compile_source) unless the library is newer than its source."""
    os.makedirs(_BUILD_DIR, exist_ok=True)
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        compile_source(_SRC, _LIB_PATH)
    return _LIB_PATH


def _library_path() -> str:
    """The compiled oracle.  WQ_ORACLE_LIB names another build of this source
    instead: the mutation tests load copies with one planted mistake."""
    return os.environ.get("WQ_ORACLE_LIB") or build()


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(_library_path())
            P = ctypes.c_void_p
            I = ctypes.c_int
            D = ctypes.c_double
            S = ctypes.c_size_t
            sig = {
                "orc_quantize": (I, [P, I, I, I, I, P, P, P]),
                "orc_tile_pack": (I, [P, P, P, I, I, I, I, P, P]),
                "orc_tile_unpack": (I, [P, P, I, I, I, I, P, P, P]),
                "orc_dequant": (I, [P, P, P, I, I, I, P]),
                "orc_merge_lora": (I, [P, P, P, I, I, I, P, P, I, D, P]),
                "orc_rms_scale": (I, [P, I, I, D, P]),
                "orc_gateup": (I, [P, I, I, I, P, P, P, P, P, P, I, P, P, P, I, D, I, D, P, P]),
                "orc_down": (I, [P, I, I, I, P, P, P, I, P, P, P]),
                "orc_down_bf16": (I, [P, I, I, I, P, P, P, P]),
                "orc_rope": (I, [P, I, I, ctypes.c_long, D]),
                "orc_qproj": (I, [P, I, I, P, P, P, I, I, P]),
                "orc_attn_decode": (I, [P, P, P, P, I, I, I, I, I, P]),
                "orc_threads": (I, []),
                "orc_set_threads": (None, [I]),
                "orc_f32_to_f16_array": (None, [P, S, P]),
                "orc_f16_to_f64_array": (None, [P, S, P]),
                "orc_f64_to_bf16_array": (None, [P, S, P]),
                "orc_bf16_to_f64_array": (None, [P, S, P]),
            }
            for name, (res, args) in sig.items():
                fn = getattr(lib, name)
                fn.restype = res
                fn.argtypes = args
            _lib = lib
    return _lib


def _p(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


# ---------------------------------------------------------------- conversions
def f32_to_f16_bits(a) -> np.ndarray:
    a = _c(a, np.float32)
    out = np.empty(a.shape, np.uint16)
    _load().orc_f32_to_f16_array(_p(a), a.size, _p(out))
    return out


def f16_bits_to_f64(a) -> np.ndarray:
    a = _c(a, np.uint16)
    out = np.empty(a.shape, np.float64)
    _load().orc_f16_to_f64_array(_p(a), a.size, _p(out))
    return out


def f64_to_bf16_bits(a) -> np.ndarray:
    a = _c(a, np.float64)
    out = np.empty(a.shape, np.uint16)
    _load().orc_f64_to_bf16_array(_p(a), a.size, _p(out))
    return out


def bf16_bits_to_f64(a) -> np.ndarray:
    a = _c(a, np.uint16)
    out = np.empty(a.shape, np.float64)
    _load().orc_bf16_to_f64_array(_p(a), a.size, _p(out))
    return out


# --------------------------------------------------------------- quantization
def quantize(w, group: int, bits: int):
    """Stage-1 RTN quantization of an fp32 [n, k] matrix -> (q u8, s f16 bits, z f16 bits, nonfinite)."""
    w = _c(w, np.float32)
    n, k = w.shape
    q = np.empty((n, k), np.uint8)
    s = np.empty((n, k // group), np.uint16)
    z = np.empty((n, k // group), np.uint16)
    rc = _load().orc_quantize(_p(w), n, k, group, bits, _p(q), _p(s), _p(z))
    if rc < 0:
        raise ValueError("orc_quantize: bad arguments")
    return q, s, z, rc


def packed_sizes(n: int, k: int, group: int, bits: int):
    """(code words, meta halves) of the packed format for an [n, k] matrix."""
    rt, kb = (n + 15) // 16, (k + 127) // 128
    wpb = {2: 128, 3: 192, 4: 256}[bits]
    return rt * kb * wpb, rt * (kb * 128 // group) * 32


def tile_pack(q, s, z, group: int, bits: int):
    q = _c(q, np.uint8)
    s = _c(s, np.uint16)
    z = _c(z, np.uint16)
    n, k = q.shape
    nw, nm = packed_sizes(n, k, group, bits)
    codes = np.empty(nw, np.uint32)
    meta = np.empty(nm, np.uint16)
    if _load().orc_tile_pack(_p(q), _p(s), _p(z), n, k, group, bits, _p(codes), _p(meta)) < 0:
        raise ValueError("orc_tile_pack: bad arguments")
    return codes, meta


def tile_unpack(codes, meta, n: int, k: int, group: int, bits: int):
    codes = _c(codes, np.uint32)
    meta = _c(meta, np.uint16)
    q = np.empty((n, k), np.uint8)
    s = np.empty((n, k // group), np.uint16)
    z = np.empty((n, k // group), np.uint16)
    if _load().orc_tile_unpack(_p(codes), _p(meta), n, k, group, bits, _p(q), _p(s), _p(z)) < 0:
        raise ValueError("orc_tile_unpack: bad arguments")
    return q, s, z


def dequant(q, s, z, group: int) -> np.ndarray:
    q = _c(q, np.uint8)
    s = _c(s, np.uint16)
    z = _c(z, np.uint16)
    n, k = q.shape
    w = np.empty((n, k), np.float64)
    if _load().orc_dequant(_p(q), _p(s), _p(z), n, k, group, _p(w)) < 0:
        raise ValueError("orc_dequant: bad arguments")
    return w


def merge_lora(q, s, z, group: int, lora_b, lora_a, lora_scale: float) -> np.ndarray:
    """fp32 [n, k] matrix deq(W) + alpha B A (B bf16 bits [n, r], A bf16 bits [r, k]).

    alpha is taken as the fp32 value the library receives (``float`` in its C ABI).
    """
    q = _c(q, np.uint8)
    s = _c(s, np.uint16)
    z = _c(z, np.uint16)
    n, k = q.shape
    lb = _c(lora_b, np.uint16).reshape(n, -1)
    r = lb.shape[1]
    la = _c(lora_a, np.uint16).reshape(r, k) if r else np.zeros(1, np.uint16)
    out = np.empty((n, k), np.float32)
    rc = _load().orc_merge_lora(_p(q), _p(s), _p(z), n, k, group, _p(lb if r else np.zeros(1, np.uint16)),
                                _p(la), r, float(np.float32(lora_scale)), _p(out))
    if rc < 0:
        raise ValueError("orc_merge_lora: bad arguments")
    return out


# -------------------------------------------------------------------- forward
def rms_scale(x_bits, eps: float = RMS_EPS) -> np.ndarray:
    """rs[t] = 1 / sqrt(mean(x[t]^2) + eps) in fp64; prenorm multiplies x by it, unrounded."""
    x = _c(x_bits, np.uint16)
    m, d = x.shape
    out = np.empty(m, np.float64)
    _load().orc_rms_scale(_p(x), m, d, eps, _p(out))
    return out


def gateup(x_bits, gate, up, group: int, lora_a=None, lora_bg=None, lora_bu=None,
           lora_scale: float = 0.0, prenorm: bool = False, eps: float = RMS_EPS):
    """h = SiLU(g) * u with unmerged LoRA.  gate / up are (q, s, z) tuples.

    Returns (h_f64 [m, inter], h_bf16_bits [m, inter]).
    """
    x = _c(x_bits, np.uint16)
    m, d = x.shape
    qg, sg, zg = (_c(gate[0], np.uint8), _c(gate[1], np.uint16), _c(gate[2], np.uint16))
    qu, su, zu = (_c(up[0], np.uint8), _c(up[1], np.uint16), _c(up[2], np.uint16))
    inter = qg.shape[0]
    if lora_a is None:
        r = 0
        la = lbg = lbu = np.zeros(1, np.uint16)
    else:
        la, lbg, lbu = _c(lora_a, np.uint16), _c(lora_bg, np.uint16), _c(lora_bu, np.uint16)
        r = lbg.shape[1]
    h = np.empty((m, inter), np.float64)
    hb = np.empty((m, inter), np.uint16)
    rc = _load().orc_gateup(_p(x), m, d, inter, _p(qg), _p(sg), _p(zg), _p(qu), _p(su), _p(zu),
                            group, _p(la), _p(lbg), _p(lbu), r, float(lora_scale), int(bool(prenorm)),
                            float(eps), _p(h), _p(hb))
    if rc < 0:
        raise ValueError("orc_gateup: bad arguments")
    return h, hb


def down(h_bits, wd, group: int, residual_bits=None):
    """y = residual + h deq(Wd)^T.  wd is a (q, s, z) tuple.  Returns (y_f64, y_bf16_bits)."""
    h = _c(h_bits, np.uint16)
    m, inter = h.shape
    q, s, z = (_c(wd[0], np.uint8), _c(wd[1], np.uint16), _c(wd[2], np.uint16))
    d = q.shape[0]
    res = None if residual_bits is None else _c(residual_bits, np.uint16)
    y = np.empty((m, d), np.float64)
    yb = np.empty((m, d), np.uint16)
    rc = _load().orc_down(_p(h), m, inter, d, _p(q), _p(s), _p(z), group, _p(res), _p(y), _p(yb))
    if rc < 0:
        raise ValueError("orc_down: bad arguments")
    return y, yb


def down_bf16(h_bits, wd_bits, residual_bits=None):
    """y = residual + h Wd^T with Wd bf16 bits [d, inter].  Returns (y_f64, y_bf16_bits)."""
    h = _c(h_bits, np.uint16)
    m, inter = h.shape
    wd = _c(wd_bits, np.uint16)
    d = wd.shape[0]
    assert wd.shape == (d, inter)
    res = None if residual_bits is None else _c(residual_bits, np.uint16)
    y = np.empty((m, d), np.float64)
    yb = np.empty((m, d), np.uint16)
    if _load().orc_down_bf16(_p(h), m, inter, d, _p(wd), _p(res), _p(y), _p(yb)) < 0:
        raise ValueError("orc_down_bf16: bad arguments")
    return y, yb


def rope(x, pos: int, theta: float) -> np.ndarray:
    """Rotary embedding of fp64 heads x [n_heads, hd] at position pos (returns a rotated copy)."""
    out = np.array(x, dtype=np.float64, order="C", copy=True)
    n_heads, hd = out.shape
    if _load().orc_rope(_p(out), n_heads, hd, int(pos), float(theta)) < 0:
        raise ValueError("orc_rope: bad arguments")
    return out


def attn_decode(q, k_bits, v_bits, lens) -> np.ndarray:
    """o [B, H, hd] from fp64 q [B, H, hd] over bf16-bit caches [B, Hkv, L, hd] and lengths [B]."""
    q = _c(q, np.float64)
    kc, vc = _c(k_bits, np.uint16), _c(v_bits, np.uint16)
    b, h, hd = q.shape
    _, hkv, lmax, hd2 = kc.shape
    assert hd2 == hd and vc.shape == kc.shape and kc.shape[0] == b
    ln = _c(lens, np.int32)
    o = np.empty((b, h, hd), np.float64)
    if _load().orc_attn_decode(_p(q), _p(kc), _p(vc), _p(ln), b, h, hkv, hd, lmax, _p(o)) < 0:
        raise ValueError("orc_attn_decode: bad arguments")
    return o


def qproj(x, w, group: int) -> np.ndarray:
    """out = x deq(W)^T for unrounded fp64 x [m, k]; w is a (q, s, z) tuple of an [n, k] matrix."""
    x = _c(x, np.float64)
    q, s, z = (_c(w[0], np.uint8), _c(w[1], np.uint16), _c(w[2], np.uint16))
    m, k = x.shape
    n = q.shape[0]
    assert q.shape[1] == k
    out = np.empty((m, n), np.float64)
    if _load().orc_qproj(_p(x), m, k, _p(q), _p(s), _p(z), n, group, _p(out)) < 0:
        raise ValueError("orc_qproj: bad arguments")
    return out


def threads() -> int:
    return _load().orc_threads()


def set_threads(n: int) -> None:
    _load().orc_set_threads(int(n))
