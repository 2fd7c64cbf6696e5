"""The C ABI library: it loads on a machine without a GPU, exports every
function include/wq.h declares, and rejects bad arguments on the host before
touching the device."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def wq():
    from paper_2606_04238_gb300 import _build
    _build.build()
    from paper_2606_04238_gb300 import wq as mod
    mod.lib()
    return mod


def _declared_functions():
    names = set()
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            text = open(os.path.join(ROOT, "include", fn)).read()
            text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
            names |= set(re.findall(r"\b(wq_[a-z0-9_]+)\s*\(", text))
    return sorted(names)


def test_exports_every_declared_function(wq):
    declared = _declared_functions()
    assert len(declared) >= 13
    lib = ctypes.CDLL(wq.library_path())
    for name in declared:
        assert hasattr(lib, name), f"{name} declared in include/ but not exported"


def test_version(wq):
    assert "sm_103a" in wq.version()


def test_packed_sizes(wq):
    # Qwen3-4B gate: 608 row tiles x 20 blocks x 512 B; 608 x 20 groups x 64 B
    assert wq.packed_sizes(2, 9728, 2560, 128) == (608 * 20 * 512, 608 * 20 * 64)
    # ragged rows and features pad to 16 x 128
    assert wq.packed_sizes(4, 21, 160, 32) == (2 * 2 * 1024, 2 * 8 * 64)
    # 3-bit codes (two planes): 192 words a block
    assert wq.packed_sizes(3, 40, 256, 32) == (3 * 2 * 768, 3 * 8 * 64)
    for bad in ((5, 16, 128, 64), (1, 16, 128, 64), (2, 16, 128, 48), (2, 16, 100, 64), (4, 16, 128, 256)):
        with pytest.raises(wq.WQError) as e:
            wq.packed_sizes(*bad)
        assert e.value.status == -2


def _qw(wq, n, k, group, bits, codes=16, meta=16):
    return wq._QWeight(codes, meta, n, k, group, bits)


def test_gateup_host_validation(wq):
    L = wq.lib()
    ok_g = _qw(wq, 64, 256, 64, 2)
    ok_u = _qw(wq, 64, 256, 64, 2)
    x = ctypes.c_void_p(16)

    def call(x, m, g, u, a=None, bg=None, bu=None, r=0, flags=0, h=16):
        return L.wq_gateup_w2_lora(x, m, ctypes.byref(g), ctypes.byref(u), a, bg, bu, r, 2.0, flags,
                                   ctypes.c_void_p(h), ctypes.c_void_p(16), 1 << 20, None)

    assert call(x, -1, ok_g, ok_u) == -1                                   # negative m
    assert call(x, 16385, ok_g, ok_u) == -4                                # beyond the token limit
    assert call(x, 1, _qw(wq, 64, 256, 64, 4), ok_u) == -2                 # wrong bit width
    assert L.wq_gateup_w3_lora(x, 65, ctypes.byref(_qw(wq, 64, 256, 64, 3)), ctypes.byref(_qw(wq, 64, 256, 64, 3)),
                               None, None, None, 0, 0.0, 0, ctypes.c_void_p(16), ctypes.c_void_p(16), 1 << 20,
                               None) == -4                                  # 3-bit codes above 64 tokens
    assert call(x, 1, ok_g, _qw(wq, 32, 256, 64, 2)) == -2                 # gate / up differ
    assert call(x, 1, _qw(wq, 64, 200, 64, 2), _qw(wq, 64, 200, 64, 2)) == -2  # k % group
    assert call(x, 1, _qw(wq, 64, 256, 48, 2), _qw(wq, 64, 256, 48, 2)) == -2  # group
    assert call(x, 1, _qw(wq, 64, 256, 64, 2, codes=8), ok_u) == -3        # misaligned codes
    assert call(x, 1, _qw(wq, 64, 256, 64, 2, codes=0), ok_u) == -1       # null codes
    assert call(x, 1, ok_g, ok_u, r=12, a=16, bg=16, bu=16) == -2         # rank not a multiple of 8
    assert call(x, 1, ok_g, ok_u, r=8) == -1                               # rank without pointers
    assert call(x, 1, ok_g, ok_u, flags=4) == -1                           # unknown flag
    assert call(x, 0, ok_g, ok_u) == 0                                     # empty batch: no-op
    assert call(ctypes.c_void_p(0), 1, ok_g, ok_u) == -1                   # null x
    assert call(ctypes.c_void_p(24), 1, ok_g, ok_u) == -3                  # misaligned x
    assert "aligned" in wq.lib().wq_last_error().decode()


def test_down_and_stack_host_validation(wq):
    L = wq.lib()
    dn = _qw(wq, 256, 64, 64, 4)
    assert L.wq_down_w4(ctypes.c_void_p(16), 1, ctypes.byref(_qw(wq, 256, 64, 64, 2)), None, ctypes.c_void_p(16), 0,
                        ctypes.c_void_p(16), 1 << 20, None) == -2
    assert L.wq_down_w4(ctypes.c_void_p(16), 1, ctypes.byref(dn), None, ctypes.c_void_p(16), 7,
                        ctypes.c_void_p(16), 1 << 20, None) == -1
    assert L.wq_down_w4(ctypes.c_void_p(16), 0, ctypes.byref(dn), None, ctypes.c_void_p(16), 0,
                        ctypes.c_void_p(16), 1 << 20, None) == 0
    layer = wq._MLPLayer(_qw(wq, 64, 256, 64, 2), _qw(wq, 64, 256, 64, 2), _qw(wq, 256, 128, 64, 4), None, None, None,
                         0, 0.0)
    arr = (wq._MLPLayer * 1)(layer)
    # down [256 x 128] does not match gate/up [64 x 256]
    assert L.wq_mlp_forward(ctypes.c_void_p(16), 1, arr, 1, 1, ctypes.c_void_p(16), ctypes.c_void_p(16), 1 << 20,
                            None) == -2
    assert "layer 0" in L.wq_last_error().decode()


def test_pack_host_validation(wq):
    L = wq.lib()
    q = _qw(wq, 0, 0, 0, 0, codes=0, meta=0)
    assert L.wq_pack(ctypes.c_void_p(16), 16, 128, 64, 5, ctypes.byref(q), None, None) == -2
    assert L.wq_pack(ctypes.c_void_p(16), 16, 96, 64, 2, ctypes.byref(q), None, None) == -2
    assert L.wq_pack(ctypes.c_void_p(16), 16, 128, 64, 2, ctypes.byref(q), None, None) == -1   # null codes
    q2 = _qw(wq, 0, 0, 0, 0, codes=16, meta=40)
    assert L.wq_pack(ctypes.c_void_p(16), 16, 128, 64, 2, ctypes.byref(q2), None, None) == -3  # misaligned meta


def test_merge_host_validation(wq):
    L = wq.lib()
    src = _qw(wq, 64, 256, 64, 2)
    out = _qw(wq, 0, 0, 0, 0)

    def call(src, b=16, a=16, r=8, scale=2.0, wm=16, out=out):
        return L.wq_merge_lora(None if src is None else ctypes.byref(src), ctypes.c_void_p(b), ctypes.c_void_p(a), r,
                               scale, ctypes.c_void_p(wm), None if out is None else ctypes.byref(out), None, None)

    assert call(None) == -1                                         # null source
    assert call(_qw(wq, 64, 256, 64, 5)) == -2                      # bits
    assert call(_qw(wq, 64, 256, 48, 2)) == -2                      # group
    assert call(_qw(wq, 64, 256, 64, 2, meta=8)) == -3              # misaligned meta
    assert call(src, r=65) == -2                                    # rank above 64
    assert call(src, a=0) == -1                                     # rank without A
    assert call(src, b=17) == -3                                    # odd B pointer
    assert call(src, scale=float("inf")) == -1                      # non-finite alpha
    assert call(src, out=None) == -1                                # null output
    assert call(src, wm=0) == -1                                    # null scratch
    assert call(src, wm=20) == -3                                   # misaligned scratch
    assert call(src, r=0, a=0, b=0, out=_qw(wq, 0, 0, 0, 0, codes=0)) == -1  # null output codes


def test_down_bf16_host_validation(wq):
    L = wq.lib()

    def call(h=16, m=1, wd=16, d=64, inter=128, res=None, y=16, dtype=0):
        return L.wq_down_bf16(ctypes.c_void_p(h), m, ctypes.c_void_p(wd), d, inter,
                              None if res is None else ctypes.c_void_p(res), ctypes.c_void_p(y), dtype, None)

    assert call(m=-1) == -1                                         # negative m
    assert call(m=16385) == -4                                      # beyond the token limit
    assert call(inter=80) == -2                                     # features not a multiple of 32
    assert call(d=0) == -2                                          # no rows
    assert call(dtype=5) == -1                                      # output type
    assert call(m=0, h=0) == 0                                      # empty batch: no-op
    assert call(h=0) == -1                                          # null h
    assert call(wd=8) == -3                                         # misaligned weights
    assert call(res=40) == -3                                       # misaligned residual


def test_product_path_has_no_oracle_import():
    pkg = os.path.join(ROOT, "paper_2606_04238_gb300")
    for dirpath, _, files in os.walk(pkg):
        for fn in files:
            if fn.endswith((".py", ".cu", ".cuh", ".h", ".cpp")):
                text = open(os.path.join(dirpath, fn)).read()
                assert "import oracle" not in text and "from oracle" not in text, fn
                assert "wq_oracle" not in text, fn


def test_moe_host_validation(wq):
    L = wq.lib()
    ex = wq._MLPLayer(_qw(wq, 4 * 64, 256, 64, 2), _qw(wq, 4 * 64, 256, 64, 2), _qw(wq, 4 * 256, 64, 64, 4), None,
                      None, None, 0, 0.0)

    def call(E=4, k=2, m=1, flags=1, x=16, experts=ex):
        layer = wq._MoELayer(experts, E, k)
        return L.wq_moe_forward(ctypes.c_void_p(x), m, ctypes.c_void_p(16), ctypes.byref(layer), flags,
                                ctypes.c_void_p(16), None, None, None, None, ctypes.c_void_p(16), 1 << 20, None)

    assert call(k=0) == -2                                           # no expert selected
    assert call(k=5) == -2                                           # more than the experts
    assert call(E=3) == -2                                           # rows not a multiple of the experts
    assert call(E=300, k=2) == -2                                    # above 256 experts
    assert call(m=65) == -2                                          # above 64 tokens
    assert call(flags=2) == -1                                       # unknown flag
    assert call(m=0) == 0                                            # empty batch: no-op
    assert call(x=0) == -1                                           # null x
    assert call(x=24) == -3                                          # misaligned x
    bad_down = wq._MLPLayer(ex.gate, ex.up, _qw(wq, 4 * 256, 128, 64, 4), None, None, None, 0, 0.0)
    assert call(experts=bad_down) == -2                              # down [E d x inter] mismatch
    with_lora = wq._MLPLayer(ex.gate, ex.up, ex.down, None, None, None, 8, 2.0)
    assert call(experts=with_lora) == -1                             # rank without pointers
