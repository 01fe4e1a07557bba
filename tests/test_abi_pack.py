"""C ABI (host side, no GPU): exported symbols, validation errors, and bit-exact parity of every
pp_pack section with the oracle's projection (§4.3 Eq. 6), connectivity pruning (§4.4) and
layout (§3.4) over the workloads' layer shapes and adversarial ties."""
import ctypes
import os
import re

import numpy as np
import pytest

from conftest import ROOT
from oracle import layout as OL
from oracle import patterns as OP
from oracle import project as OPR
from paper_2003_06513_gb300 import api
from paper_2003_06513_gb300 import workloads as WL

PP_ERR = {"NULL": -1, "SHAPE": -2, "PATTERN": -3, "KEEP": -4, "NONFINITE": -5, "ALIGN": -6,
          "DTYPE": -7, "NOT_BOUND": -8, "BUFFER": -9, "CUDA": -10, "ARG": -11}


def _declared_symbols():
    names = set()
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            with open(os.path.join(ROOT, "include", fn)) as f:
                src = f.read()
            names |= set(re.findall(r"^\s*(?:int|const char\*)\s+(pp_\w+)\s*\(", src, re.M))
    return names


def test_library_exports_every_declared_symbol(lib):
    names = _declared_symbols()
    assert {"pp_pack", "pp_conv", "pp_bind_device", "pp_export", "pp_query", "pp_destroy",
            "pp_status_string", "pp_default_patterns", "pp_maxpool2x2"} <= names
    for n in names:
        assert hasattr(lib, n), f"{n} declared in include/ but not exported"


def test_status_strings(lib):
    for code in [0] + list(PP_ERR.values()) + [-99]:
        assert isinstance(lib.pp_status_string(code), bytes)


def test_default_patterns_equal_oracle_library(lib):
    buf = (ctypes.c_uint16 * 8)()
    assert lib.pp_default_patterns(buf, 8) == 8
    assert list(buf) == OP.default8()


def _pack_raw(lib, W, cout, cin, groups=1, stride=1, masks=None, keep=0.5):
    masks = OP.default8() if masks is None else masks
    m = (ctypes.c_uint16 * max(1, len(masks)))(*masks)
    h = ctypes.c_void_p()
    Wc = np.ascontiguousarray(W, dtype=np.float32) if W is not None else None
    wp = Wc.ctypes.data_as(ctypes.POINTER(ctypes.c_float)) if Wc is not None else None
    st = lib.pp_pack(wp, cout, cin, groups, stride, m, len(masks), keep, ctypes.byref(h))
    return st, h


def test_pack_validation(lib):
    W = np.random.default_rng(0).standard_normal((4, 3, 3, 3)).astype(np.float32)
    assert _pack_raw(lib, None, 4, 3)[0] == PP_ERR["NULL"]
    assert _pack_raw(lib, W, 0, 3)[0] == PP_ERR["SHAPE"]
    assert _pack_raw(lib, W, 4, 0)[0] == PP_ERR["SHAPE"]
    assert _pack_raw(lib, W, 4, 3, groups=2)[0] == PP_ERR["SHAPE"]
    assert _pack_raw(lib, W, 4, 3, stride=3)[0] == PP_ERR["SHAPE"]
    assert _pack_raw(lib, W, 4, 3, masks=[0x1F])[0] == PP_ERR["PATTERN"]        # 5 taps
    assert _pack_raw(lib, W, 4, 3, masks=[0x17, 0x17])[0] == PP_ERR["PATTERN"]  # duplicate
    assert _pack_raw(lib, W, 4, 3, masks=list(range(15, 15 + 9)))[0] == PP_ERR["PATTERN"]
    assert _pack_raw(lib, W, 4, 3, masks=[0x217])[0] == PP_ERR["PATTERN"]       # bit 9
    for keep in (0.0, -1.0, 1.0000001, float("nan")):
        assert _pack_raw(lib, W, 4, 3, keep=keep)[0] == PP_ERR["KEEP"]
    for bad in (np.nan, np.inf, -np.inf):
        Wb = W.copy()
        Wb[2, 1, 0, 2] = bad
        assert _pack_raw(lib, Wb, 4, 3)[0] == PP_ERR["NONFINITE"]
    st, h = _pack_raw(lib, W, 4, 3)
    assert st == 0
    v = ctypes.c_int64()
    assert lib.pp_query(h, 999, ctypes.byref(v)) == PP_ERR["ARG"]
    assert lib.pp_export(h, 42, None, 0) == PP_ERR["ARG"]
    assert lib.pp_export(h, 0, ctypes.c_void_p(1), 3) == PP_ERR["BUFFER"]
    # pp_conv / pp_bind_device arguments rejected before any CUDA call
    assert lib.pp_conv(None, None, 0, 1, 4, 4, None, 0, None, None) == PP_ERR["NULL"]
    assert lib.pp_conv(h, ctypes.c_void_p(256), 0, 1, 4, 4, None, 0, ctypes.c_void_p(4096),
                       None) == PP_ERR["NOT_BOUND"]
    assert lib.pp_bind_device(h, None, 1 << 20, None) == PP_ERR["NULL"]
    assert lib.pp_bind_device(h, ctypes.c_void_p(1024 + 16), 1 << 20, None) == PP_ERR["ALIGN"]
    assert lib.pp_bind_device(h, ctypes.c_void_p(1024), 1, None) == PP_ERR["BUFFER"]
    assert lib.pp_maxpool2x2(None, 5, 1, 1, 4, 4, None, None) == PP_ERR["DTYPE"]
    assert lib.pp_maxpool2x2(None, 0, 1, 1, 1, 4, None, None) == PP_ERR["SHAPE"]
    assert lib.pp_destroy(h) == 0
    assert lib.pp_destroy(None) == 0


SECTIONS = ["header", "pid", "perm", "desc", "kofs", "vals", "dense", "image"]


def _compare(W, keep, groups=1, stride=1, masks=None):
    from paper_2003_06513_gb300 import api
    masks = OP.default8() if masks is None else masks
    layer = api.pp_pack(W, masks, keep, groups, stride)
    r = OPR.project(W, masks, keep)
    ref = OL.build(W, r["pid"], masks, groups, stride, r["beta"])
    assert layer.beta == r["beta"]
    for name in SECTIONS:
        got = layer.export(name)
        exp = ref[name].reshape(-1)
        if name == "header":
            exp = ref["header"]
        assert got.dtype == exp.dtype, name
        assert got.tobytes() == exp.tobytes(), f"section {name} differs from the oracle"
    return layer, r


@pytest.mark.parametrize("cout,cin,keep,seed", [(64, 64, 0.5, 0), (13, 5, 0.3, 1), (8, 1, 1.0, 2),
                                                (1, 1, 1.0, 3), (17, 9, 0.01, 4), (64, 3, 1.0, 5),
                                                (40, 24, 0.140625, 6), (9, 33, 0.75, 7)])
def test_pack_bit_exact_random(cout, cin, keep, seed):
    W = np.random.default_rng(seed).standard_normal((cout, cin, 3, 3)).astype(np.float32)
    _compare(W, keep)


def test_pack_bit_exact_single_layer_workload():
    L = WL.single_layer()
    _compare(WL.weights(L), L.keep)


@pytest.mark.parametrize("idx", [0, 1, 2, 4, 8, 12])
def test_pack_bit_exact_vgg_layers(idx):
    L = WL.vgg16()[idx]
    _compare(WL.weights(L), L.keep)


@pytest.mark.parametrize("idx", [0, 3, 7, 13])
def test_pack_bit_exact_resnet_layers(idx):
    L = WL.resnet50_3x3()[idx]
    _compare(WL.weights(L), L.keep, stride=L.stride)


@pytest.mark.parametrize("idx", [0, 1, 16])
def test_pack_bit_exact_mobilenet_depthwise(idx):
    L = WL.mobilenet_v2_dw()[idx]
    _compare(WL.weights(L), L.keep, groups=L.cin, stride=L.stride)


def test_pack_bit_exact_adversarial_ties():
    """Integer-valued weights with many zeros and repeated magnitudes: ties in the pattern
    argmax, in the connectivity ranking and in the filter order."""
    rng = np.random.default_rng(21)
    W = rng.integers(-2, 3, size=(24, 16, 3, 3)).astype(np.float32)
    W[3] = 0.0                      # an all-zero filter
    W[5, :, 1, 1] = 7.0             # centre-only kernels
    W[7] = W[6]                     # identical filters
    W[9, 2] = -0.0
    for keep in (1.0, 0.5, 0.3, 0.05):
        _compare(W, keep)


def test_pack_other_library_bit_exact():
    """A 6-pattern library (§4.2 allows m = 6-8) different from the compiled one."""
    masks = [OP.mask_of(t) for t in ([0, 4, 5, 8], [1, 4, 6, 7], [2, 3, 4, 8], [0, 1, 4, 7],
                                     [3, 4, 7, 8], [1, 2, 4, 6])]
    W = np.random.default_rng(3).standard_normal((20, 12, 3, 3)).astype(np.float32)
    layer, _ = _compare(W, 0.4, masks=masks)
    assert layer.query("fast_path") == 0


def test_pack_counts_and_compression():
    W = np.random.default_rng(4).standard_normal((64, 64, 3, 3)).astype(np.float32)
    from paper_2003_06513_gb300 import api
    for keep, rate in ((1.0, 2.25), (0.28125, 8.0), (0.1875, 12.0), (0.140625, 16.0)):
        layer = api.pp_pack(W, None, keep)
        dense = layer.export("dense")
        assert np.count_nonzero(dense) == 4 * layer.beta
        assert 9 * 64 * 64 / np.count_nonzero(dense) == rate


def test_conv_pool_rejections_without_gpu(lib):
    """pp_conv_pool_ws refuses layers whose kernel has no fused pooling (depthwise, other
    libraries) and unbound handles, before touching the GPU."""
    rng = np.random.default_rng(3)
    Wd = rng.standard_normal((8, 1, 3, 3)).astype(np.float32)
    dw = api.pp_pack(Wd, None, 1.0, 8, 1)
    assert lib.pp_conv_pool_ws(dw._h, None, 0, 1, 8, 8, None, 1, None, None, 0, None) == -14
    assert b"fusion" in lib.pp_status_string(-14)
    Wt = rng.standard_normal((8, 4, 3, 3)).astype(np.float32)
    dense = api.pp_pack(Wt, None, 0.5)
    assert lib.pp_conv_pool_ws(dense._h, None, 0, 1, 8, 8, None, 1, None, None, 0, None) == -8   # not bound


def test_design_patterns_matches_oracle(lib):
    """pp_design_patterns equals the oracle's heuristic on random kernels and on VGG-16's."""
    rng = np.random.default_rng(8)
    cases = [rng.standard_normal((500, 9)).astype(np.float32),
             rng.integers(-2, 3, size=(400, 9)).astype(np.float32)]          # many magnitude ties
    cases.append(np.concatenate([WL.weights(L).reshape(-1, 9) for L in WL.vgg16()[:4]]))
    for K in cases:
        for m in (1, 6, 8):
            assert api.design_patterns([K], m) == OP.design_library(K, m)


def test_design_patterns_validation(lib):
    K = np.zeros((2, 9), np.float32)
    masks = (ctypes.c_uint16 * 8)()
    n = ctypes.c_int()
    ptr = K.ctypes.data_as(ctypes.POINTER(ctypes.c_float))
    assert lib.pp_design_patterns(ptr, 2, 0, masks, ctypes.byref(n)) == -2
    assert lib.pp_design_patterns(ptr, 2, 9, masks, ctypes.byref(n)) == -2
    assert lib.pp_design_patterns(ptr, 0, 8, masks, ctypes.byref(n)) == -2
    K[1, 3] = np.nan
    assert lib.pp_design_patterns(ptr, 2, 8, masks, ctypes.byref(n)) == -5
