"""Python binding of libwq.so (include/wq.h): argument marshalling only.

Every function here converts torch tensors to device pointers and sizes,
calls the C ABI of the same name on the current CUDA stream, and raises
``WQError`` on a non-zero status.  All arithmetic runs in the CUDA kernels;
there is no fallback: if the library is missing or no GPU is present the
calls raise.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import torch

from . import _build

WQ_PRENORM = 1
WQ_LAUNCH_CHAIN = 2
WQ_LAUNCH_STACK = 4
WQ_BF16 = 0
WQ_F32 = 1

_STATUS = {0: "WQ_OK", -1: "WQ_ERR_ARG", -2: "WQ_ERR_SHAPE", -3: "WQ_ERR_ALIGN", -4: "WQ_ERR_UNSUPPORTED",
           -5: "WQ_ERR_CUDA", -6: "WQ_ERR_TIMEOUT", -7: "WQ_ERR_WORKSPACE"}


class WQError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{_STATUS.get(status, status)}: {message}")
        self.status = status


class _QWeight(ctypes.Structure):
    _fields_ = [("codes", ctypes.c_void_p), ("meta", ctypes.c_void_p), ("n", ctypes.c_int32),
                ("k", ctypes.c_int32), ("group", ctypes.c_int32), ("bits", ctypes.c_int32)]


class _MLPLayer(ctypes.Structure):
    _fields_ = [("gate", _QWeight), ("up", _QWeight), ("down", _QWeight), ("lora_a", ctypes.c_void_p),
                ("lora_b_gate", ctypes.c_void_p), ("lora_b_up", ctypes.c_void_p), ("r", ctypes.c_int32),
                ("lora_scale", ctypes.c_float)]


class _DecoderLayer(ctypes.Structure):
    _fields_ = [("qkv", _QWeight), ("o", _QWeight), ("mlp", _MLPLayer), ("n_heads", ctypes.c_int32),
                ("n_kv", ctypes.c_int32), ("head_dim", ctypes.c_int32), ("rope_theta", ctypes.c_float)]


class _MoELayer(ctypes.Structure):
    _fields_ = [("experts", _MLPLayer), ("n_experts", ctypes.c_int32), ("top_k", ctypes.c_int32)]


_lib = None


def library_path() -> str:
    """libwq.so, or the bounds-checking debug build when WQ_DEBUG_LIB=1."""
    return _build.DEBUG_LIB_PATH if os.environ.get("WQ_DEBUG_LIB") == "1" else _build.LIB_PATH


def lib():
    """The loaded libwq.so; raises if it has not been built."""
    global _lib
    if _lib is None:
        path = library_path()
        if not os.path.exists(path):
            raise RuntimeError(f"libwq.so not found at {path}: run __graft_entry__.build() first")
        L = ctypes.CDLL(path)
        P, I, S, F, U = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t, ctypes.c_float, ctypes.c_uint
        QP = ctypes.POINTER(_QWeight)
        sig = {
            "wq_packed_sizes": (I, [I, I, I, I, ctypes.POINTER(S), ctypes.POINTER(S)]),
            "wq_pack": (I, [P, I, I, I, I, QP, P, P]),
            "wq_pack_w2": (I, [P, I, I, I, QP, P, P]),
            "wq_pack_w4": (I, [P, I, I, I, QP, P, P]),
            "wq_merge_lora": (I, [QP, P, P, I, F, P, QP, P, P]),
            "wq_workspace_bytes": (S, [I, I, I, I]),
            "wq_workspace_init": (I, [P, S, P]),
            "wq_gateup_w2_lora": (I, [P, I, QP, QP, P, P, P, I, F, U, P, P, S, P]),
            "wq_gateup_w2_lora_noalloc": (I, [P, I, QP, QP, P, P, P, I, F, U, P, P]),
            "wq_gateup_w3_lora": (I, [P, I, QP, QP, P, P, P, I, F, U, P, P, S, P]),
            "wq_gateup_w4": (I, [P, I, QP, QP, U, P, P, S, P]),
            "wq_down_w4": (I, [P, I, QP, P, P, I, P, S, P]),
            "wq_down_bf16": (I, [P, I, P, I, I, P, P, I, P]),
            "wq_mlp_forward": (I, [P, I, ctypes.POINTER(_MLPLayer), I, U, P, P, S, P]),
            "wq_mlp_forward_states": (I, [P, I, ctypes.POINTER(_MLPLayer), I, U, P, P, P, P, S, P]),
            "wq_mlp_forward_info": (I, [I, ctypes.POINTER(_MLPLayer), I, U, ctypes.POINTER(ctypes.c_int64)]),
            "wq_plan_info": (I, [I, I, I, I, I, I, ctypes.POINTER(ctypes.c_int64)]),
            "wq_attn_workspace_bytes": (S, [I, I, I, I, I]),
            "wq_attn_decode": (I, [P, P, P, I, I, I, I, I, F, P, P, I, P, P, S, P]),
            "wq_decoder_workspace_bytes": (S, [I, ctypes.POINTER(_DecoderLayer), I]),
            "wq_decoder_layer_forward": (I, [P, I, P, ctypes.POINTER(_DecoderLayer), P, P, I, U, P, P, S, P]),
            "wq_moe_workspace_bytes": (S, [I, ctypes.POINTER(_MoELayer), U]),
            "wq_moe_forward": (I, [P, I, P, ctypes.POINTER(_MoELayer), U, P, P, P, P, P, P, S, P]),
            "wq_wait_check": (I, [P]),
            "wq_last_error": (ctypes.c_char_p, []),
            "wq_device_status": (I, [ctypes.POINTER(I)]),
            "wq_version": (ctypes.c_char_p, []),
            "wq_debug_record": (I, [ctypes.POINTER(ctypes.c_longlong)]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


def _check(status: int):
    if status != 0:
        raise WQError(status, lib().wq_last_error().decode())


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream():
    return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)


@dataclass
class QWeight:
    """A packed group-quantized matrix [n, k] held in two device tensors."""
    codes: torch.Tensor   # int32 words
    meta: torch.Tensor    # int16 (binary16 bit patterns)
    n: int
    k: int
    group: int
    bits: int

    def c(self) -> _QWeight:
        return _QWeight(self.codes.data_ptr(), self.meta.data_ptr(), self.n, self.k, self.group, self.bits)

    @property
    def nbytes(self) -> int:
        return self.codes.numel() * 4 + self.meta.numel() * 2


def dense_weight(w: torch.Tensor) -> QWeight:
    """A dense bf16 [n, k] matrix as a down weight of wq_mlp_forward (bits 16;
    the BF16/W2-GateUp configuration)."""
    assert w.dtype == torch.bfloat16 and w.is_cuda and w.is_contiguous()
    n, k = w.shape
    return QWeight(w.view(torch.int16).view(-1), torch.zeros(8, dtype=torch.int16, device=w.device), n, k, 0, 16)


def packed_sizes(bits: int, n: int, k: int, group: int):
    cb, mb = ctypes.c_size_t(), ctypes.c_size_t()
    _check(lib().wq_packed_sizes(bits, n, k, group, ctypes.byref(cb), ctypes.byref(mb)))
    return cb.value, mb.value


def empty_qweight(n: int, k: int, group: int, bits: int, device="cuda") -> QWeight:
    cb, mb = packed_sizes(bits, n, k, group)
    return QWeight(torch.empty(cb // 4, dtype=torch.int32, device=device),
                   torch.empty(mb // 2, dtype=torch.int16, device=device), n, k, group, bits)


def pack(w: torch.Tensor, group: int, bits: int, nonfinite: torch.Tensor | None = None,
         out: QWeight | None = None) -> QWeight:
    """Quantize and pack an fp32 [n, k] device matrix (wq_pack)."""
    assert w.dtype == torch.float32 and w.is_cuda and w.is_contiguous()
    n, k = w.shape
    q = out if out is not None else empty_qweight(n, k, group, bits, device=w.device)
    cq = q.c()
    _check(lib().wq_pack(_ptr(w), n, k, group, bits, ctypes.byref(cq), _ptr(nonfinite), _stream()))
    return q


def pack_w2(w, group, nonfinite=None):
    return pack(w, group, 2, nonfinite)


def pack_w4(w, group, nonfinite=None):
    return pack(w, group, 4, nonfinite)


def merge_lora(src: QWeight, lora_b: torch.Tensor | None, lora_a: torch.Tensor | None, lora_scale: float,
               out: QWeight | None = None, w_merged: torch.Tensor | None = None,
               nonfinite: torch.Tensor | None = None) -> QWeight:
    """Merge an adapter into a packed matrix and quantize it again (wq_merge_lora).

    lora_b is bf16 [n, r] and lora_a bf16 [r, k], contiguous on the device (None
    for r = 0).  ``out=src`` merges in place; ``w_merged`` (fp32 [n, k]) receives
    the merged matrix before quantization.
    """
    r = 0 if lora_b is None else lora_b.shape[1]
    if r:
        assert lora_b.dtype == torch.bfloat16 and lora_a.dtype == torch.bfloat16
        assert lora_b.is_contiguous() and lora_a.is_contiguous()
        assert tuple(lora_b.shape) == (src.n, r) and tuple(lora_a.shape) == (r, src.k)
    if w_merged is None:
        w_merged = torch.empty(src.n, src.k, dtype=torch.float32, device=src.codes.device)
    q = out if out is not None else empty_qweight(src.n, src.k, src.group, src.bits, device=src.codes.device)
    cs, cq = src.c(), q.c()
    _check(lib().wq_merge_lora(ctypes.byref(cs), _ptr(lora_b) if r else None, _ptr(lora_a) if r else None, r,
                               float(lora_scale), _ptr(w_merged), ctypes.byref(cq), _ptr(nonfinite), _stream()))
    return q


def workspace_bytes(m: int, d: int, inter: int, r: int = 0) -> int:
    return int(lib().wq_workspace_bytes(m, d, inter, r))


def workspace(m: int, d: int, inter: int, r: int = 0, device="cuda") -> torch.Tensor:
    """A zero-initialised workspace tensor for up to m tokens of a (d, inter) layer."""
    nb = workspace_bytes(m, d, inter, r)
    if nb == 0:
        raise WQError(-2, f"no workspace size for m={m}, d={d}, inter={inter}")
    ws = torch.empty(nb, dtype=torch.uint8, device=device)
    _check(lib().wq_workspace_init(_ptr(ws), nb, _stream()))
    return ws


def gateup_w2_lora(x, gate: QWeight, up: QWeight, lora_a=None, lora_b_gate=None, lora_b_up=None,
                   lora_scale: float = 0.0, prenorm: bool = False, h=None, ws=None):
    m, d = x.shape
    r = 0 if lora_b_gate is None else lora_b_gate.shape[1]
    if h is None:
        h = torch.empty((m, gate.n), dtype=torch.bfloat16, device=x.device)
    if ws is None:
        ws = workspace(max(m, 1), d, gate.n, r, device=x.device)
    cg, cu = gate.c(), up.c()
    _check(lib().wq_gateup_w2_lora(_ptr(x), m, ctypes.byref(cg), ctypes.byref(cu), _ptr(lora_a), _ptr(lora_b_gate),
                                   _ptr(lora_b_up), r, float(lora_scale), WQ_PRENORM if prenorm else 0, _ptr(h),
                                   _ptr(ws), ws.numel(), _stream()))
    return h


def gateup_w3_lora(x, gate: QWeight, up: QWeight, lora_a=None, lora_b_gate=None, lora_b_up=None,
                   lora_scale: float = 0.0, prenorm: bool = False, h=None, ws=None):
    """wq_gateup_w3_lora: gateup_w2_lora with 3-bit gate/up codes (App. B)."""
    m, d = x.shape
    r = 0 if lora_b_gate is None else lora_b_gate.shape[1]
    if h is None:
        h = torch.empty((m, gate.n), dtype=torch.bfloat16, device=x.device)
    if ws is None:
        ws = workspace(max(m, 1), d, gate.n, r, device=x.device)
    cg, cu = gate.c(), up.c()
    _check(lib().wq_gateup_w3_lora(_ptr(x), m, ctypes.byref(cg), ctypes.byref(cu), _ptr(lora_a), _ptr(lora_b_gate),
                                   _ptr(lora_b_up), r, float(lora_scale), WQ_PRENORM if prenorm else 0, _ptr(h),
                                   _ptr(ws), ws.numel(), _stream()))
    return h


def gateup_w2_lora_noalloc(x, gate: QWeight, up: QWeight, lora_a=None, lora_b_gate=None, lora_b_up=None,
                           lora_scale: float = 0.0, prenorm: bool = False, h=None):
    """wq_gateup_w2_lora_noalloc: the same call with the library's built-in scratch.

    For callers that cannot allocate device memory; ``h`` may be passed in so
    that nothing is allocated on the Python side either.
    """
    m, d = x.shape
    r = 0 if lora_b_gate is None else lora_b_gate.shape[1]
    if h is None:
        h = torch.empty((m, gate.n), dtype=torch.bfloat16, device=x.device)
    cg, cu = gate.c(), up.c()
    _check(lib().wq_gateup_w2_lora_noalloc(_ptr(x), m, ctypes.byref(cg), ctypes.byref(cu), _ptr(lora_a),
                                           _ptr(lora_b_gate), _ptr(lora_b_up), r, float(lora_scale),
                                           WQ_PRENORM if prenorm else 0, _ptr(h), _stream()))
    return h


def gateup_w4(x, gate: QWeight, up: QWeight, prenorm: bool = False, h=None, ws=None):
    m, d = x.shape
    if h is None:
        h = torch.empty((m, gate.n), dtype=torch.bfloat16, device=x.device)
    if ws is None:
        ws = workspace(max(m, 1), d, gate.n, 0, device=x.device)
    cg, cu = gate.c(), up.c()
    _check(lib().wq_gateup_w4(_ptr(x), m, ctypes.byref(cg), ctypes.byref(cu), WQ_PRENORM if prenorm else 0, _ptr(h),
                              _ptr(ws), ws.numel(), _stream()))
    return h


def down_w4(h, down: QWeight, residual=None, out_f32: bool = False, y=None, ws=None):
    m, inter = h.shape
    if y is None:
        y = torch.empty((m, down.n), dtype=torch.float32 if out_f32 else torch.bfloat16, device=h.device)
    if ws is None:
        ws = workspace(max(m, 1), down.n, inter, 0, device=h.device)
    cd = down.c()
    _check(lib().wq_down_w4(_ptr(h), m, ctypes.byref(cd), _ptr(residual), _ptr(y), WQ_F32 if out_f32 else WQ_BF16,
                            _ptr(ws), ws.numel(), _stream()))
    return y


def down_bf16(h, wd, residual=None, out_f32: bool = False, y=None):
    """y = residual + h Wd^T with a bf16 Wd [d, inter] (wq_down_bf16)."""
    assert h.dtype == torch.bfloat16 and wd.dtype == torch.bfloat16 and h.is_contiguous() and wd.is_contiguous()
    m, inter = h.shape
    d = wd.shape[0]
    assert wd.shape[1] == inter
    if y is None:
        y = torch.empty((m, d), dtype=torch.float32 if out_f32 else torch.bfloat16, device=h.device)
    _check(lib().wq_down_bf16(_ptr(h), m, _ptr(wd), d, inter, _ptr(residual), _ptr(y), WQ_F32 if out_f32 else WQ_BF16,
                              _stream()))
    return y


@dataclass
class MLPLayer:
    gate: QWeight
    up: QWeight
    down: QWeight
    lora_a: torch.Tensor | None = None
    lora_b_gate: torch.Tensor | None = None
    lora_b_up: torch.Tensor | None = None
    lora_scale: float = 0.0

    @property
    def r(self) -> int:
        return 0 if self.lora_b_gate is None else self.lora_b_gate.shape[1]

    def c(self) -> _MLPLayer:
        return _MLPLayer(self.gate.c(), self.up.c(), self.down.c(),
                         None if self.lora_a is None else self.lora_a.data_ptr(),
                         None if self.lora_b_gate is None else self.lora_b_gate.data_ptr(),
                         None if self.lora_b_up is None else self.lora_b_up.data_ptr(),
                         self.r, float(self.lora_scale))


def merge_layer(layer: MLPLayer, w_merged: torch.Tensor | None = None) -> MLPLayer:
    """The layer with its gate and up adapters merged into new 2-bit codes
    (wq_merge_lora on each); the merged layer carries no adapter (r = 0)."""
    r = layer.r
    if r == 0:
        return MLPLayer(layer.gate, layer.up, layer.down)
    a = layer.lora_a
    gate = merge_lora(layer.gate, layer.lora_b_gate, a[:r], layer.lora_scale, w_merged=w_merged)
    up = merge_lora(layer.up, layer.lora_b_up, a[r:], layer.lora_scale, w_merged=w_merged)
    return MLPLayer(gate, up, layer.down)


class LayerTable:
    """The C array of wq_mlp_layer for a stack (kept alive for graph replays)."""

    def __init__(self, layers):
        self.layers = list(layers)
        self.array = (_MLPLayer * max(1, len(self.layers)))(*[l.c() for l in self.layers])


def _stack_flags(prenorm: bool, chain: bool, stack: bool = False) -> int:
    return (WQ_PRENORM if prenorm else 0) | (WQ_LAUNCH_CHAIN if chain else 0) | (WQ_LAUNCH_STACK if stack else 0)


def mlp_forward(x, layers, prenorm: bool = True, y=None, ws=None, table: LayerTable | None = None,
                chain: bool = False, stack: bool = False):
    """Stack of gated-MLP layers (wq_mlp_forward) on the current stream; chain=True
    asks for the per-layer launch chain (WQ_LAUNCH_CHAIN), stack=True for the
    single-launch stack kernel (WQ_LAUNCH_STACK)."""
    m, d = x.shape
    if table is None:
        table = LayerTable(layers)
    if y is None:
        y = torch.empty_like(x)
    if ws is None:
        l0 = table.layers[0]
        ws = workspace(max(m, 1), d, l0.gate.n, l0.r, device=x.device)
    _check(lib().wq_mlp_forward(_ptr(x), m, table.array, len(table.layers), _stack_flags(prenorm, chain, stack), _ptr(y),
                                _ptr(ws), ws.numel(), _stream()))
    return y


def mlp_forward_states(x, layers, prenorm: bool = True, states=None, h_states=None, y=None, ws=None,
                       table: LayerTable | None = None, chain: bool = False, with_h: bool = False,
                       stack: bool = False):
    """wq_mlp_forward_states: the stack plus every layer's output, bf16 [n_layers, m, d], and with
    with_h=True every layer's h, bf16 [n_layers, m, inter].  Returns (y, states, h_states)."""
    m, d = x.shape
    if table is None:
        table = LayerTable(layers)
    n = len(table.layers)
    inter = table.layers[0].gate.n
    if states is None:
        states = torch.empty((n, m, d), dtype=torch.bfloat16, device=x.device)
    if h_states is None and with_h:
        h_states = torch.empty((n, m, inter), dtype=torch.bfloat16, device=x.device)
    if y is None:
        y = torch.empty_like(x)
    if ws is None:
        l0 = table.layers[0]
        ws = workspace(max(m, 1), d, l0.gate.n, l0.r, device=x.device)
    _check(lib().wq_mlp_forward_states(_ptr(x), m, table.array, n, _stack_flags(prenorm, chain, stack), _ptr(y),
                                       _ptr(states), _ptr(h_states), _ptr(ws), ws.numel(), _stream()))
    return y, states, h_states


ROUTE_GEMV_CHAIN, ROUTE_GEMM_CHAIN, ROUTE_STACK = 0, 1, 2
_STEP_FIELDS = ("rb", "kp", "wk", "tpw", "panels", "ctas")


def mlp_forward_info(m: int, layers, prenorm: bool = True, table: LayerTable | None = None,
                     chain: bool = False, stack: bool = False) -> dict:
    """How wq_mlp_forward would run this stack (wq_mlp_forward_info)."""
    if table is None:
        table = LayerTable(layers)
    arr = (ctypes.c_int64 * 16)()
    _check(lib().wq_mlp_forward_info(m, table.array, len(table.layers), _stack_flags(prenorm, chain, stack), arr))
    v = list(arr)
    out = {"route": v[0]}
    if v[0] == ROUTE_STACK:
        out["stack"] = dict(zip(("ctas", "stages", "stage_bytes", "h_barrier", "warps_per_tile", "tiles_per_cta",
                                 "smem"), v[1:8]))
    if v[0] == ROUTE_GEMV_CHAIN:
        out["gateup"] = dict(zip(_STEP_FIELDS, v[1:7]))
        out["down"] = dict(zip(_STEP_FIELDS, v[7:13]))
        out["panel"] = bool(v[13])
    return out


PLAN_FIELDS = ("row_tiles", "kblocks", "rb", "kp", "wk", "panels", "ctas", "threads", "smem", "tok_chunk")
KIND_GATEUP_W2, KIND_GATEUP_W4, KIND_DOWN_W4, KIND_GATEUP_W3 = 0, 1, 2, 3


def plan_info(kind: int, n: int, k: int, m: int, group: int, r: int = 0) -> dict:
    """The launch decomposition the library would use on the current device."""
    arr = (ctypes.c_int64 * 10)()
    _check(lib().wq_plan_info(kind, n, k, m, group, r, arr))
    return dict(zip(PLAN_FIELDS, list(arr)))


def attn_workspace(batch: int, n_heads: int, n_kv: int, head_dim: int, max_len: int, device="cuda") -> torch.Tensor:
    nb = int(lib().wq_attn_workspace_bytes(batch, n_heads, n_kv, head_dim, max_len))
    if nb == 0:
        raise WQError(-2, "no attention workspace for these sizes")
    return torch.empty(nb, dtype=torch.uint8, device=device)


def attn_decode(qkv, x, lens, k_cache, v_cache, n_heads: int, n_kv: int, theta: float, o=None, ws=None):
    """wq_attn_decode: one decode step of grouped-query attention; the caches
    (bf16 [B, n_kv, max_len, head_dim]) gain position lens[b]."""
    b, d = x.shape
    _, hkv, max_len, hd = k_cache.shape
    assert hkv == n_kv and lens.dtype == torch.int32
    if o is None:
        o = torch.empty((b, n_heads * hd), dtype=torch.bfloat16, device=x.device)
    if ws is None:
        ws = attn_workspace(b, n_heads, n_kv, hd, max_len, device=x.device)
    _check(lib().wq_attn_decode(_ptr(qkv), _ptr(x), _ptr(lens), b, d, n_heads, n_kv, hd, float(theta), _ptr(k_cache),
                                _ptr(v_cache), max_len, _ptr(o), _ptr(ws), ws.numel(), _stream()))
    return o


@dataclass
class DecoderLayer:
    """A decoder layer: 4-bit qkv (rows of Wq, Wk, Wv) and o projections around an MLPLayer."""
    qkv: QWeight
    o: QWeight
    mlp: MLPLayer
    n_heads: int
    n_kv: int
    head_dim: int
    rope_theta: float = 1e6

    def c(self) -> _DecoderLayer:
        return _DecoderLayer(self.qkv.c(), self.o.c(), self.mlp.c(), self.n_heads, self.n_kv, self.head_dim,
                             float(self.rope_theta))


def decoder_workspace(batch: int, layer: DecoderLayer, max_len: int, device="cuda") -> torch.Tensor:
    cl = layer.c()
    nb = int(lib().wq_decoder_workspace_bytes(batch, ctypes.byref(cl), max_len))
    if nb == 0:
        raise WQError(-2, "no decoder workspace for these sizes")
    ws = torch.empty(nb, dtype=torch.uint8, device=device)
    _check(lib().wq_workspace_init(_ptr(ws), nb, _stream()))
    return ws


def decoder_layer_forward(x, lens, layer: DecoderLayer, k_cache, v_cache, prenorm: bool = True, y=None, ws=None,
                          c_layer=None):
    """wq_decoder_layer_forward: one decode step of the layer for x bf16 [B, d]."""
    b, d = x.shape
    max_len = k_cache.shape[2]
    if y is None:
        y = torch.empty_like(x)
    if ws is None:
        ws = decoder_workspace(b, layer, max_len, device=x.device)
    cl = c_layer if c_layer is not None else layer.c()
    _check(lib().wq_decoder_layer_forward(_ptr(x), b, _ptr(lens), ctypes.byref(cl), _ptr(k_cache), _ptr(v_cache),
                                          max_len, WQ_PRENORM if prenorm else 0, _ptr(y), _ptr(ws), ws.numel(),
                                          _stream()))
    return y


@dataclass
class MoELayer:
    """A mixture-of-experts block: the experts' matrices stacked row-wise in one
    MLPLayer (gate/up [E*inter, d], down [E*d, inter], lora_a [E*2r, d],
    lora_b_* [E*inter, r]), n_experts experts, top_k of them per token."""
    experts: MLPLayer
    n_experts: int
    top_k: int

    def c(self) -> _MoELayer:
        return _MoELayer(self.experts.c(), self.n_experts, self.top_k)


def moe_workspace(m: int, layer: MoELayer, prenorm: bool = True, device="cuda") -> torch.Tensor:
    cl = layer.c()
    nb = int(lib().wq_moe_workspace_bytes(m, ctypes.byref(cl), WQ_PRENORM if prenorm else 0))
    if nb == 0:
        raise WQError(-2, "no MoE workspace for these sizes")
    ws = torch.empty(nb, dtype=torch.uint8, device=device)
    _check(lib().wq_workspace_init(_ptr(ws), nb, _stream()))
    return ws


def moe_forward(x, logits, layer: MoELayer, prenorm: bool = True, y=None, ws=None, with_slots: bool = False,
                c_layer=None):
    """wq_moe_forward for x bf16 [m, d] and router logits fp32 [m, E].  Returns y,
    or with with_slots (y, expert_idx [m, k], expert_w [m, k], h [m*k, inter], y_slots [m*k, d])."""
    m, d = x.shape
    k = layer.top_k
    inter = layer.experts.gate.n // layer.n_experts
    if y is None:
        y = torch.empty_like(x)
    if ws is None:
        ws = moe_workspace(m, layer, prenorm, device=x.device)
    idx = wt = hs = ys = None
    if with_slots:
        idx = torch.empty((m, k), dtype=torch.int32, device=x.device)
        wt = torch.empty((m, k), dtype=torch.float32, device=x.device)
        hs = torch.empty((m * k, inter), dtype=torch.bfloat16, device=x.device)
        ys = torch.empty((m * k, d), dtype=torch.float32, device=x.device)
    cl = c_layer if c_layer is not None else layer.c()
    _check(lib().wq_moe_forward(_ptr(x), m, _ptr(logits), ctypes.byref(cl), WQ_PRENORM if prenorm else 0, _ptr(y),
                                _ptr(idx), _ptr(wt), _ptr(hs), _ptr(ys), _ptr(ws), ws.numel(), _stream()))
    return (y, idx, wt, hs, ys) if with_slots else y


def wait_check():
    """wq_wait_check: a launch whose bounded waits run out (WQ_ERR_TIMEOUT in the device status)."""
    _check(lib().wq_wait_check(_stream()))


def device_status() -> int:
    v = ctypes.c_int(0)
    _check(lib().wq_device_status(ctypes.byref(v)))
    return v.value


def debug_record():
    """Debug build: (site, line, value, count) of the first failed in-kernel check."""
    rec = (ctypes.c_longlong * 4)()
    _check(lib().wq_debug_record(rec))
    return tuple(rec)


def version() -> str:
    return lib().wq_version().decode()
