"""GPU parity of pp_conv / pp_maxpool2x2 with the float64 oracle (§4.1 Eq. 1 over the projected
weights of §4.3 Eq. 6 and §4.4).

Error metric: |y_gpu - y_ref| / (sum |W_hat| |x| + |b| + 2^-1000) per output, max over outputs;
bar 1e-4 for fp32 I/O and 2e-3 for fp16 I/O.  The oracle projects the weights itself: nothing
it uses comes from the CUDA path.
"""
import ctypes

import numpy as np
import pytest
import torch

from oracle import conv as OC
from oracle import patterns as OP
from oracle import project as OPR
from paper_2003_06513_gb300 import _lib, api
from paper_2003_06513_gb300 import workloads as WL

pytestmark = pytest.mark.gpu

TOL = {torch.float32: 1e-4, torch.float16: 2e-3}


@pytest.fixture(autouse=True)
def _no_pipeline_timeout():
    """After every test: no kernel of the test recorded a pipeline wait that ran out (the status
    word of the conv kernels, read and cleared through pp_device_status)."""
    yield
    torch.cuda.synchronize()
    st = ctypes.c_uint(0)
    assert _lib.load().pp_device_status(1, ctypes.byref(st)) == 0
    assert st.value == 0, f"a conv kernel recorded pipeline timeout bits {st.value:#x}"


SPLIT_CAP = 32 << 20   # a workspace below the balanced schedule's (39 MB): the input-channel split


def _sms():
    return torch.cuda.get_device_properties(0).multi_processor_count


def _np_dt(dt):
    return np.float32 if dt == torch.float32 else np.float16


def run_gpu(W, x, b, keep, stride=1, relu=True, depthwise=False, dtype=torch.float32, masks=None,
            guard=0, to_host=True, ws=False, ws_bytes=None):
    """Pack + bind + pp_conv; x host array; returns the output (host float64 unless
    ``to_host=False``) and the layer."""
    layer = api.pp_pack(W, masks, keep, W.shape[0] if depthwise else 1, stride)
    dev = torch.device("cuda")
    layer.bind(dev)
    xt = torch.from_numpy(np.ascontiguousarray(x)).to(dev)
    bt = None if b is None else torch.from_numpy(b).to(dev)
    shape = layer.out_shape(x.shape)
    n = int(np.prod(shape))
    if guard:
        buf = torch.full((n + 2 * guard,), float("nan"), dtype=dtype, device=dev)
        y = buf[guard:guard + n].view(shape)
    else:
        y = torch.empty(shape, dtype=dtype, device=dev)
    wt = None
    if ws:
        nb = layer.workspace_bytes(x.shape) if ws_bytes is None else ws_bytes
        if nb:
            wt = torch.full((nb // 4,), float("nan"), dtype=torch.float32, device=dev)
    layer.conv(xt, bt, relu, y, workspace=wt)
    torch.cuda.synchronize()
    if guard:
        g = torch.cat([buf[:guard], buf[guard + n:]])
        assert torch.isnan(g).all(), "pp_conv wrote outside its output tensor"
    return (y.double().cpu().numpy() if to_host else y), layer


def oracle(W, x, b, keep, stride=1, relu=True, depthwise=False, masks=None):
    masks = OP.default8() if masks is None else masks
    Wh = OPR.project(W, masks, keep)["W_hat"]
    ref = OC.conv_ref(x.astype(np.float64), Wh, b, stride, relu, depthwise)
    den = OC.denominator(x.astype(np.float64), Wh, b, stride, depthwise)
    return ref, den


def check(W, x, b, keep, stride=1, relu=True, depthwise=False, dtype=torch.float32, masks=None,
          guard=64):
    y, layer = run_gpu(W, x, b, keep, stride, relu, depthwise, dtype, masks, guard)
    ref, den = oracle(W, x, b, keep, stride, relu, depthwise, masks)
    err = OC.max_norm_err(y, ref, den)
    assert err <= TOL[dtype], f"normalised error {err:.3e} > {TOL[dtype]}"
    return y, err


def rnd(shape, seed, relu=False, dtype=np.float32):
    return WL.activations(shape, seed, relu=relu, dtype=dtype)


# --------------------------------------------------------------------------- single layer

def test_single_layer_workload():
    L = WL.single_layer()
    x = WL.layer_input(L, 1)
    check(WL.weights(L), x, WL.bias(L), L.keep)


@pytest.mark.parametrize("N,Cin,Cout,H,W,keep,stride", [
    (1, 3, 5, 7, 7, 1.0, 1), (2, 16, 13, 13, 11, 0.5, 1), (1, 1, 1, 1, 1, 1.0, 1),
    (3, 5, 9, 1, 9, 0.7, 1), (1, 64, 24, 9, 13, 0.3, 1), (2, 8, 8, 15, 15, 0.5, 2),
    (1, 20, 17, 14, 14, 0.4, 2), (1, 3, 64, 2, 2, 1.0, 2), (4, 33, 40, 6, 5, 0.25, 1),
    (1, 130, 16, 8, 8, 0.6, 1), (2, 48, 72, 28, 28, 0.3, 1), (1, 16, 16, 17, 31, 0.5, 2)])
def test_shapes_fp32(N, Cin, Cout, H, W, keep, stride):
    rng = np.random.default_rng(N * 1000 + Cin * 10 + H)
    Wt = (rng.standard_normal((Cout, Cin, 3, 3)) * np.sqrt(2 / (9 * Cin))).astype(np.float32)
    x = rnd((N, Cin, H, W), Cin + H)
    b = (rng.standard_normal(Cout) * 0.1).astype(np.float32)
    check(Wt, x, b, keep, stride)


@pytest.mark.parametrize("ws", [False, True])
@pytest.mark.parametrize("N,Cin,Cout,H,W,keep,stride", [
    (1, 8, 8, 3, 1000, 0.5, 1),      # rows wider than any tile: several tiles along x
    (1, 8, 8, 3, 1001, 0.5, 2),
    (1, 16, 8, 5, 2100, 0.5, 1),
    (2, 4, 8, 300, 3, 1.0, 1),       # tall and narrow
    (1, 2048, 16, 2, 2, 0.2, 1),     # many input channels on a tiny image: 32+ stages per unit
    (1, 4096, 8, 1, 1, 0.1, 1)])     # a 1 x 1 image: every tap but the centre reads padding
def test_extreme_shapes(N, Cin, Cout, H, W, keep, stride, ws):
    rng = np.random.default_rng(Cin + W)
    Wt = (rng.standard_normal((Cout, Cin, 3, 3)) * np.sqrt(2 / (9 * Cin))).astype(np.float32)
    x = rnd((N, Cin, H, W), Cin + H)
    b = (rng.standard_normal(Cout) * 0.1).astype(np.float32)
    y, layer = run_gpu(Wt, x, b, keep, stride, guard=64, ws=ws)
    if ws:
        assert layer.plan(x.shape, layer.workspace_bytes(x.shape))["splits"] >= 1
    ref, den = oracle(Wt, x, b, keep, stride)
    err = OC.max_norm_err(y, ref, den)
    assert err <= TOL[torch.float32], f"normalised error {err:.3e}"


@pytest.mark.parametrize("dtype", [torch.float32, torch.float16])
@pytest.mark.parametrize("stride", [1, 2])
def test_input_one_element_off_alignment(dtype, stride):
    """x one element past a 16-byte boundary (even rows): the copy fallback must not pair
    elements across a misaligned address."""
    rng = np.random.default_rng(41)
    Wt = (rng.standard_normal((16, 12, 3, 3)) * np.sqrt(2 / 108)).astype(np.float32)
    x = rnd((2, 12, 10, 16), 43, dtype=_np_dt(dtype))
    b = (rng.standard_normal(16) * 0.1).astype(np.float32)
    layer = api.pp_pack(Wt, None, 0.5, 1, stride).bind("cuda")
    flat = torch.empty(x.size + 1, dtype=dtype, device="cuda")
    xt = flat[1:].view(x.shape)
    xt.copy_(torch.from_numpy(x))
    y = layer.conv(xt, torch.from_numpy(b).cuda(), True)
    ref, den = oracle(Wt, x, b, 0.5, stride)
    err = OC.max_norm_err(y.double().cpu().numpy(), ref, den)
    assert err <= TOL[dtype], f"normalised error {err:.3e}"


@pytest.mark.parametrize("stride", [1, 2])
def test_fp16_io(stride):
    rng = np.random.default_rng(5)
    Wt = (rng.standard_normal((24, 40, 3, 3)) * np.sqrt(2 / 360)).astype(np.float32)
    x = rnd((2, 40, 18, 20), 6, dtype=np.float16)
    b = (rng.standard_normal(24) * 0.1).astype(np.float32)
    check(Wt, x, b, 0.5, stride, dtype=torch.float16)


def test_no_bias_no_relu_and_degenerate_keep():
    rng = np.random.default_rng(8)
    Wt = rng.standard_normal((12, 10, 3, 3)).astype(np.float32)
    x = rnd((2, 10, 9, 9), 9)
    check(Wt, x, None, 0.5, relu=False)
    # beta = 1: a single kernel survives; every other filter outputs ReLU(bias)
    b = (rng.standard_normal(12) * 0.1).astype(np.float32)
    y, _ = check(Wt, x, b, 1e-9)
    r = OPR.project(Wt, OP.default8(), 1e-9)
    for co in range(12):
        if (r["pid"][co] < 0).all():
            assert np.all(y[:, co] == max(float(b[co]), 0.0))


def test_other_pattern_library_generic_path():
    masks = [OP.mask_of(t) for t in ([0, 4, 5, 8], [1, 4, 6, 7], [2, 3, 4, 8], [0, 1, 4, 7],
                                     [3, 4, 7, 8], [1, 2, 4, 6])]
    rng = np.random.default_rng(10)
    Wt = rng.standard_normal((11, 7, 3, 3)).astype(np.float32)
    x = rnd((2, 7, 10, 9), 11)
    b = rng.standard_normal(11).astype(np.float32)
    for stride in (1, 2):
        check(Wt, x, b, 0.6, stride, masks=masks)
    Wd = rng.standard_normal((9, 1, 3, 3)).astype(np.float32)
    check(Wd, rnd((2, 9, 8, 8), 12), b[:9], 1.0, 1, depthwise=True, masks=masks)


@pytest.mark.parametrize("dtype", [torch.float32, torch.float16])
@pytest.mark.parametrize("stride", [1, 2])
def test_depthwise(dtype, stride):
    rng = np.random.default_rng(13)
    C = 21
    Wd = (rng.standard_normal((C, 1, 3, 3)) * np.sqrt(2 / 9)).astype(np.float32)
    x = rnd((3, C, 13, 12), 14, dtype=_np_dt(dtype))
    b = (rng.standard_normal(C) * 0.1).astype(np.float32)
    check(Wd, x, b, 1.0, stride, depthwise=True, dtype=dtype)
    check(Wd, x, b, 0.5, stride, depthwise=True, dtype=dtype)     # pruned channels -> sigma(b)


@pytest.mark.parametrize("dtype", [torch.float32, torch.float16])
@pytest.mark.parametrize("N,C,H,W,stride", [(1, 8, 160, 160, 1),    # one plane over two CTAs
                                            (1, 8, 160, 160, 2),
                                            (2, 16, 32, 48, 1),     # 16-byte rows in both dtypes
                                            (2, 16, 32, 48, 2),
                                            (3, 40, 7, 7, 1),       # many small planes per CTA
                                            (2, 24, 14, 14, 2),
                                            (2, 24, 14, 14, 1),     # whole-row items, 14 wide
                                            (2, 16, 28, 28, 1),     # 28-wide rows in 2 pieces (fp16)
                                            (2, 16, 28, 28, 2),
                                            (1, 4, 9, 2100, 1),     # rows too wide to stage whole
                                            (1, 4, 9, 2100, 2)])
def test_depthwise_vector_and_tiled(dtype, N, C, H, W, stride):
    rng = np.random.default_rng(C * 7 + H)
    Wd = (rng.standard_normal((C, 1, 3, 3)) * np.sqrt(2 / 9)).astype(np.float32)
    x = rnd((N, C, H, W), H + W, dtype=_np_dt(dtype))
    b = (rng.standard_normal(C) * 0.1).astype(np.float32)
    check(Wd, x, b, 1.0, stride, depthwise=True, dtype=dtype, guard=64)
    check(Wd, x, b, 0.7, stride, relu=False, depthwise=True, dtype=dtype, guard=64)


@pytest.mark.parametrize("dtype", [torch.float32, torch.float16])
@pytest.mark.parametrize("H,stride", [(7, 1), (14, 1), (14, 2)])
def test_depthwise_other_library(dtype, H, stride):
    """A library other than the compiled one: the depthwise kernels take the taps from the masks
    (the default library's pattern-specialised row bodies do not apply)."""
    rng = np.random.default_rng(41 + H)
    C = 40
    masks = [OP.mask_of(t) for t in ([0, 4, 5, 8], [1, 4, 6, 7], [2, 3, 4, 8])]
    Wd = (rng.standard_normal((C, 1, 3, 3)) * np.sqrt(2 / 9)).astype(np.float32)
    x = rnd((3, C, H, H), 50 + H, dtype=_np_dt(dtype))
    b = (rng.standard_normal(C) * 0.1).astype(np.float32)
    check(Wd, x, b, 1.0, stride, depthwise=True, dtype=dtype, masks=masks)
    check(Wd, x, b, 0.6, stride, depthwise=True, dtype=dtype, masks=masks)


@pytest.mark.parametrize("dtype", [torch.float32, torch.float16])
def test_depthwise_unaligned_input(dtype):
    """x 8 bytes off a 16-byte boundary: the direct (unstaged) depthwise kernel."""
    rng = np.random.default_rng(31)
    C, H, W = 12, 20, 24
    Wd = (rng.standard_normal((C, 1, 3, 3)) * np.sqrt(2 / 9)).astype(np.float32)
    x = rnd((2, C, H, W), 32, dtype=_np_dt(dtype))
    b = (rng.standard_normal(C) * 0.1).astype(np.float32)
    layer = api.pp_pack(Wd, None, 1.0, C, 1).bind("cuda")
    off = 8 // x.itemsize
    flat = torch.empty(x.size + off, dtype=dtype, device="cuda")
    xt = flat[off:].view(x.shape)
    xt.copy_(torch.from_numpy(x))
    assert xt.data_ptr() % 16 == 8
    y = layer.conv(xt, torch.from_numpy(b).cuda(), True)
    ref, den = oracle(Wd, x, b, 1.0, 1, True, True)
    assert OC.max_norm_err(y.double().cpu().numpy(), ref, den) <= TOL[dtype]


@pytest.mark.parametrize("shape,stride,dtype,kernel", [
    ((3, 21, 13, 12), 1, torch.float32, 1),    # rows mode, one band
    ((2, 10, 37, 64), 1, torch.float16, 1),    # rows mode: two lane row-sets, a short last band
    ((2, 12, 33, 64), 2, torch.float16, 1),    # rows mode, stride 2, odd height (zero rows below)
    ((2, 8, 40, 48), 2, torch.float32, 1),     # rows mode, stride 2, five lane row-sets
    ((3, 21, 13, 12), 1, torch.float16, 3),    # planes, two columns a lane; x ends inside a 16-byte block
    ((3, 21, 13, 12), 2, torch.float32, 2),    # planes, stride 2; y ends inside a 16-byte block
    ((2, 24, 9, 9), 1, torch.float16, 4),      # planes, odd width
    ((1, 13, 7, 7), 1, torch.float16, 5),      # tiles of 7x7: 13 planes, a short last chunk
    ((3, 40, 7, 7), 1, torch.float32, 5),      # tiles of 7x7, fp32
    ((5, 40, 14, 14), 2, torch.float16, 7),    # tiles at stride 2, 14x14 to 7x7
    ((3, 21, 14, 14), 1, torch.float16, 6),    # tiles of 7 rows x 14 columns, two bands a plane
    ((2, 11, 28, 28), 1, torch.float16, 6),    # tiles: two column pieces x four bands a plane
    ((2, 11, 28, 28), 1, torch.float32, 1),    # fp32: 112-byte rows, rows mode
    ((2, 24, 28, 28), 2, torch.float16, 7),    # tiles at stride 2: two column pieces x two bands
    ((3, 21, 13, 12), 2, torch.float16, 2),    # 6 output columns at stride 2: column lanes
])
def test_streamed_depthwise(shape, stride, dtype, kernel):
    """The streamed depthwise kernel in each of its modes (asserted through the plan), with the
    chunk tails its bulk copies leave to plain loads and stores, against the oracle; NaN guard
    regions around y catch stray writes."""
    N, C, H, W = shape
    rng = np.random.default_rng(C * 3 + H + stride)
    Wd = (rng.standard_normal((C, 1, 3, 3)) * np.sqrt(2 / 9)).astype(np.float32)
    x = rnd(shape, 7 * H + W, dtype=_np_dt(dtype))
    b = (rng.standard_normal(C) * 0.1).astype(np.float32)
    lay = api.pp_pack(Wd, None, 1.0, C, stride)
    assert lay.plan(shape, 0, dtype=dtype)["dw_kernel"] == kernel
    check(Wd, x, b, 1.0, stride, depthwise=True, dtype=dtype, guard=64)
    check(Wd, x, b, 0.6, stride, relu=False, depthwise=True, dtype=dtype, guard=64)


@pytest.mark.parametrize("dtype", [torch.float32, torch.float16])
@pytest.mark.parametrize("stride", [1, 2])
def test_streamed_depthwise_rows_other_library(dtype, stride):
    """Rows mode with a library other than the compiled one: its masks match none of the row
    loops compiled per pattern, so every channel takes the nine-tap loop."""
    rng = np.random.default_rng(77 + stride)
    C, H, W = 12, 18, 64
    masks = [OP.mask_of(t) for t in ([0, 4, 5, 8], [1, 4, 6, 7], [2, 3, 4, 8])]
    Wd = (rng.standard_normal((C, 1, 3, 3)) * np.sqrt(2 / 9)).astype(np.float32)
    x = rnd((2, C, H, W), 60 + stride, dtype=_np_dt(dtype))
    b = (rng.standard_normal(C) * 0.1).astype(np.float32)
    lay = api.pp_pack(Wd, masks, 1.0, C, stride)
    assert lay.plan((2, C, H, W), 0, dtype=dtype)["dw_kernel"] == 1
    check(Wd, x, b, 1.0, stride, depthwise=True, dtype=dtype, masks=masks)
    check(Wd, x, b, 0.6, stride, depthwise=True, dtype=dtype, masks=masks)


@pytest.mark.parametrize("m", [6, 8])
def test_designed_library_end_to_end(m):
    """A library designed from the layer's own kernels (§4.2 heuristic) packs and runs through
    the same entry points; checked against the oracle projected with that library."""
    L = WL.vgg16()[2]                                           # 64 -> 128
    W, b = WL.weights(L), WL.bias(L)
    masks = api.design_patterns([W], m)
    assert masks == OP.design_library(W.reshape(-1, 9), m) and len(masks) == m
    x = WL.layer_input(L, 1)[:, :, :20, :18].copy()
    check(W, x, b, L.keep, 1, masks=masks)
    check(W, x, b, L.keep, 2, masks=masks)


def test_deterministic_and_zero_batch():
    L = WL.single_layer()
    x = WL.layer_input(L, 2)
    y1, layer = run_gpu(WL.weights(L), x, WL.bias(L), L.keep)
    y2, _ = run_gpu(WL.weights(L), x, WL.bias(L), L.keep)
    assert np.array_equal(y1, y2)
    xt = torch.empty((0, 64, 32, 32), device="cuda")
    out = layer.conv(xt, None, True)
    assert out.shape == (0, 64, 32, 32)


@pytest.mark.parametrize("dtype", [torch.float32, torch.float16])
def test_maxpool_exact(dtype):
    x = rnd((3, 5, 14, 15), 15, dtype=_np_dt(dtype))
    y = api.pp_maxpool2x2(torch.from_numpy(x).cuda())
    assert np.array_equal(y.cpu().numpy(), OC.maxpool2x2(x))


# --------------------------------------------------------------------------- workloads

def _sampled_check(L, n, dtype=torch.float32, samples=(0, -1), ws=True):
    """Full-batch launch with the workspace the benchmark gives it (its launch configuration),
    oracle on sampled images."""
    x = WL.layer_input(L, n, relu=not L.depthwise, dtype=_np_dt(dtype))
    W, b = WL.weights(L), WL.bias(L)
    y, _ = run_gpu(W, x, b, L.keep, L.stride, True, L.depthwise, dtype, guard=256, to_host=False,
                   ws=ws)
    assert bool(torch.isfinite(y).all())
    idx = [s % n for s in samples]
    ref, den = oracle(W, x[idx], b, L.keep, L.stride, True, L.depthwise)
    err = OC.max_norm_err(y[idx].double().cpu().numpy(), ref, den)
    assert err <= TOL[dtype], f"{L.name}: normalised error {err:.3e}"


@pytest.mark.parametrize("idx", range(13))
def test_vgg16_layer_batch32(idx):
    _sampled_check(WL.vgg16()[idx], 32)


@pytest.mark.parametrize("idx", range(16))
def test_resnet50_layer_batch64(idx):
    _sampled_check(WL.resnet50_3x3()[idx], 64)


@pytest.mark.parametrize("idx", range(17))
def test_mobilenet_dw_layer_batch128_fp16(idx):
    _sampled_check(WL.mobilenet_v2_dw()[idx], 128, torch.float16)


def test_vgg16_chained_network():
    """The whole 13-layer stack with the library's max-pool between blocks, batch 2; every
    layer is checked on the exact input the GPU layer received."""
    layers = WL.vgg16()
    x = torch.from_numpy(WL.vgg16_image(2)).cuda()
    for L in layers:
        W, b = WL.weights(L), WL.bias(L)
        layer = api.pp_pack(W, None, L.keep).bind("cuda")
        y = layer.conv(x, torch.from_numpy(b).cuda(), True)
        torch.cuda.synchronize()
        xin = x.cpu().numpy()
        ref, den = oracle(W, xin, b, L.keep)
        err = OC.max_norm_err(y.double().cpu().numpy(), ref, den)
        assert err <= 1e-4, f"{L.name}: {err:.3e}"
        if L.pool_after:
            p = api.pp_maxpool2x2(y)
            assert np.array_equal(p.cpu().numpy(), OC.maxpool2x2(y.cpu().numpy()))
            y = p
        x = y


# --------------------------------------------------------------------------- fused max-pool

def _pool_ref(W, x, b, keep, stride, relu):
    """Oracle conv, then the oracle's 2x2/2 max-pool; the denominator of a pooled output is the
    largest denominator in its window (max is 1-Lipschitz in the max norm)."""
    ref, den = oracle(W, x, b, keep, stride, relu)
    return OC.maxpool2x2(ref), OC.maxpool2x2(den)


@pytest.mark.parametrize("dtype", [torch.float32, torch.float16])
@pytest.mark.parametrize("N,Cin,Cout,H,W,stride,relu", [(2, 16, 24, 16, 16, 1, True),
                                                        (1, 8, 13, 15, 13, 1, True),     # odd: floor
                                                        (2, 8, 16, 17, 18, 2, False),
                                                        (3, 5, 9, 6, 34, 1, False)])
def test_conv_pool_fused(dtype, N, Cin, Cout, H, W, stride, relu):
    rng = np.random.default_rng(Cin * 11 + H)
    Wt = (rng.standard_normal((Cout, Cin, 3, 3)) * np.sqrt(2 / (9 * Cin))).astype(np.float32)
    x = rnd((N, Cin, H, W), H * 3 + W, dtype=_np_dt(dtype))
    b = (rng.standard_normal(Cout) * 0.1).astype(np.float32)
    layer = api.pp_pack(Wt, None, 0.5, 1, stride).bind("cuda")
    y = layer.conv(torch.from_numpy(x).cuda(), torch.from_numpy(b).cuda(), relu, pool2x2=True)
    ref, den = _pool_ref(Wt, x, b, 0.5, stride, relu)
    assert tuple(y.shape) == ref.shape
    assert OC.max_norm_err(y.double().cpu().numpy(), ref, den) <= TOL[dtype]


def test_conv_pool_fused_with_split_equals_unfused_pool():
    """Small images with a workspace: the split path pools in its reduction; the result matches
    pp_conv_ws followed by the library's max-pool (the two calls may plan different splits, so
    their fp32 sums differ only in rounding order) and the oracle."""
    L = WL.vgg16()[12]                                     # 512 -> 512 at 14x14, pooled
    W, b = WL.weights(L), WL.bias(L)
    x = torch.from_numpy(WL.layer_input(L, 16)).cuda()
    bt = torch.from_numpy(b).cuda()
    layer = api.pp_pack(W, None, L.keep).bind("cuda")
    nb = min(max(layer.workspace_bytes(x.shape, pool2x2=True), layer.workspace_bytes(x.shape)), SPLIT_CAP)
    assert layer.plan(x.shape, nb, pool2x2=True)["splits"] > 1
    ws = torch.full((nb // 4,), float("nan"), device="cuda")
    fused = layer.conv(x, bt, True, workspace=ws, pool2x2=True)
    plain = api.pp_maxpool2x2(layer.conv(x, bt, True, workspace=ws))
    ref, den = _pool_ref(W, x[:2].cpu().numpy(), b, L.keep, 1, True)
    assert OC.max_norm_err(fused[:2].double().cpu().numpy(), plain[:2].double().cpu().numpy(), den) <= 1e-5
    assert OC.max_norm_err(fused[:2].double().cpu().numpy(), ref, den) <= 1e-4


@pytest.mark.parametrize("idx", [i for i, L in enumerate(WL.vgg16()) if L.pool_after])
def test_vgg16_pool_layer_fused_batch32(idx):
    """The benchmark's launch configuration of each VGG-16 block end: batch 32, workspace,
    fused pooling; oracle on two sampled images."""
    L = WL.vgg16()[idx]
    x = WL.layer_input(L, 32)
    W, b = WL.weights(L), WL.bias(L)
    layer = api.pp_pack(W, None, L.keep).bind("cuda")
    xt = torch.from_numpy(x).cuda()
    nb = layer.workspace_bytes(xt.shape, pool2x2=True)
    ws = torch.empty(max(nb // 4, 1), device="cuda") if nb else None
    y = layer.conv(xt, torch.from_numpy(b).cuda(), True, workspace=ws, pool2x2=True)
    ref, den = _pool_ref(W, x[[0, 31]], b, L.keep, 1, True)
    assert OC.max_norm_err(y[[0, 31]].double().cpu().numpy(), ref, den) <= 1e-4


def test_vgg16_chained_network_fused_pool():
    """The 13-layer stack with the pooling fused into each block's last conv, batch 2."""
    x = torch.from_numpy(WL.vgg16_image(2)).cuda()
    for L in WL.vgg16():
        W, b = WL.weights(L), WL.bias(L)
        layer = api.pp_pack(W, None, L.keep).bind("cuda")
        y = layer.conv(x, torch.from_numpy(b).cuda(), True, pool2x2=L.pool_after)
        torch.cuda.synchronize()
        xin = x.cpu().numpy()
        if L.pool_after:
            ref, den = _pool_ref(W, xin, b, L.keep, 1, True)
        else:
            ref, den = oracle(W, xin, b, L.keep)
        err = OC.max_norm_err(y.double().cpu().numpy(), ref, den)
        assert err <= 1e-4, f"{L.name}: {err:.3e}"
        x = y
    assert tuple(x.shape) == (2, 512, 7, 7)


@pytest.mark.parametrize("dtype", [torch.float32, torch.float16])
def test_back_to_back_layers_match_layers_run_one_at_a_time(dtype):
    """Layers launched one after another on one stream with no synchronisation (each kernel may
    start its set-up while the previous one finishes) read exactly what the previous layer wrote:
    ping-pong buffers (so a layer overwrites what the layer before it read), one workspace shared
    by the split layers, a fused pool, a stride-2 layer and a depthwise layer; the chain, run three
    times over, must equal the same layers run one at a time with a synchronisation after each."""
    dev = torch.device("cuda")
    N = 2
    specs = [  # (Cin, Cout, H, stride, keep, depthwise, pool, input-channel split)
        (8, 32, 28, 1, 0.5, False, False, False),
        (32, 64, 28, 1, 0.3, False, True, True),
        (64, 64, 14, 1, 0.3, False, False, False),
        (64, 64, 14, 1, 0.3, False, False, True),
        (64, 128, 14, 2, 0.4, False, False, True),
        (128, 128, 7, 1, 1.0, True, False, False),
        (128, 128, 7, 1, 0.3, False, False, True),
    ]
    layers, biases, in_shapes, out_shapes = [], [], [], []
    for i, (ci, co, h, st, keep, dw, pool, _) in enumerate(specs):
        L = WL.ConvLayer(f"b2b{i}", ci, co, h, h, st, dw, keep, w_seed=900 + i, b_seed=950 + i)
        layers.append(api.pp_pack(WL.weights(L), None, keep, co if dw else 1, st).bind(dev))
        biases.append(torch.from_numpy(WL.bias(L)).to(dev))
        in_shapes.append((N, ci, h, h))
        o = layers[-1].out_shape(in_shapes[-1])
        out_shapes.append((o[0], o[1], o[2] // 2, o[3] // 2) if pool else o)
    x0 = torch.from_numpy(rnd(in_shapes[0], 990, dtype=_np_dt(dtype))).to(dev)
    ws = api.workspace_for(layers, in_shapes, dev)
    splits = [lay.plan(s, ws.numel() * 4 if sp[7] else 0)["splits"] for lay, s, sp in zip(layers, in_shapes, specs)]
    assert splits == [1, 32, 1, 32, 32, 0, 32], splits     # 0: the depthwise kernel

    ref = x0
    for lay, b, sp in zip(layers, biases, specs):
        ref = lay.conv(ref.clone(), b, True, workspace=ws if sp[7] else None, pool2x2=sp[6])
        torch.cuda.synchronize()

    big = max(int(np.prod(s)) for s in out_shapes)
    bufs = [torch.full((big,), float("nan"), dtype=dtype, device=dev) for _ in range(2)]
    for _ in range(3):
        cur = x0
        for i, (lay, b, sp) in enumerate(zip(layers, biases, specs)):
            y = bufs[i % 2].narrow(0, 0, int(np.prod(out_shapes[i]))).view(out_shapes[i])
            lay.conv(cur, b, True, y, workspace=ws if sp[7] else None, pool2x2=sp[6])
            cur = y
    torch.cuda.synchronize()
    assert torch.equal(cur, ref)


# --------------------------------------------------------------------------- channel split

def _split_case():
    L = WL.vgg16()[10]                                    # 512 -> 512 at 14x14
    return L, WL.weights(L), WL.bias(L), WL.layer_input(L, 32)


def test_split_is_planned_for_small_images():
    """14x14 maps leave SMs idle with whole units (64 units of two whole images on 152 SMs; their
    56-byte fp32 rows take the copy fallback): with the full workspace the balanced schedule over
    persistent CTAs, with less than it needs the input-channel split, without one a single pass."""
    L, W, b, x = _split_case()
    lay = api.pp_pack(W, None, L.keep)
    plan = lay.plan(x.shape, lay.workspace_bytes(x.shape))
    assert plan["path"] == 1 and plan["splits"] == 1 and plan["streamk"] == 1 and plan["ctas"] == _sms()
    plan = lay.plan(x.shape, SPLIT_CAP)
    assert plan["splits"] > 1 and plan["streamk"] == 0
    assert lay.plan(x.shape, 0)["splits"] == 1
    big = api.pp_pack(WL.weights(WL.vgg16()[1]), None, 0.3)
    assert big.plan((32, 64, 224, 224), 1 << 34)["splits"] == 1


def test_split_matches_oracle_single_pass_and_is_deterministic():
    L, W, b, x = _split_case()
    y_split, lay = run_gpu(W, x, b, L.keep, ws=True, ws_bytes=SPLIT_CAP)
    y_split2, _ = run_gpu(W, x, b, L.keep, ws=True, ws_bytes=SPLIT_CAP)
    y_one, _ = run_gpu(W, x, b, L.keep, ws=False)
    assert np.array_equal(y_split, y_split2)
    ref, den = oracle(W, x[[0, 31]], b, L.keep)
    assert OC.max_norm_err(y_split[[0, 31]], ref, den) <= 1e-4
    d = np.abs(y_split - y_one) / np.maximum(np.abs(y_one), 1e-3)
    assert float(np.max(d)) < 1e-3                       # only fp32 summation order differs


def test_balanced_schedule_copy_fallback_whole_images():
    """The same 14x14 layer with the full workspace: persistent CTAs over the copy fallback's
    stages (the zero halo of whole-image tiles is the same for every unit) and the balanced
    schedule; deterministic, within the oracle's tolerance, and equal to the single pass up to
    fp32 summation order."""
    L, W, b, x = _split_case()
    lay = api.pp_pack(W, None, L.keep)
    assert lay.plan(x.shape, lay.workspace_bytes(x.shape))["streamk"] == 1
    y1, _ = run_gpu(W, x, b, L.keep, ws=True)
    y2, _ = run_gpu(W, x, b, L.keep, ws=True)
    y0, _ = run_gpu(W, x, b, L.keep, ws=False)
    assert np.array_equal(y1, y2)
    ref, den = oracle(W, x[[0, 31]], b, L.keep)
    assert OC.max_norm_err(y1[[0, 31]], ref, den) <= 1e-4
    d = np.abs(y1 - y0) / np.maximum(np.abs(y0), 1e-3)
    assert float(np.max(d)) < 1e-3


def test_balanced_schedule_matches_oracle_and_is_deterministic():
    """VGG-16 layer 9 at batch 32 (bands of one block row of 4 images on the balanced schedule):
    the same result on every run (the head of a cut unit adds its parts in chunk order), the
    oracle's within tolerance, and the whole-unit schedule's up to fp32 summation order (the
    schedule off: no workspace)."""
    L = WL.vgg16()[8]
    W, b, x = WL.weights(L), WL.bias(L), WL.layer_input(L, 32)
    lay = api.pp_pack(W, None, L.keep)
    pl = lay.plan(x.shape, lay.workspace_bytes(x.shape))
    assert pl["streamk"] == 1 and (pl["tile_by"], pl["tile_nb"]) == (1, 4)
    y1, _ = run_gpu(W, x, b, L.keep, ws=True)
    y2, _ = run_gpu(W, x, b, L.keep, ws=True)
    y0, _ = run_gpu(W, x, b, L.keep, ws=False)
    assert np.array_equal(y1, y2)
    ref, den = oracle(W, x[[0, 31]], b, L.keep)
    assert OC.max_norm_err(y1[[0, 31]], ref, den) <= 1e-4
    full_den = OC.denominator(x[[7]].astype(np.float64), OPR.project(W, OP.default8(), L.keep)["W_hat"], b, 1)
    assert OC.max_norm_err(y1[[7]], y0[[7]], full_den) <= 1e-5


def test_split_with_small_workspace_and_fp16():
    L, W, b, x = _split_case()
    lay = api.pp_pack(W, None, L.keep)
    need = lay.workspace_bytes(x.shape)
    out_bytes = 32 * 512 * 14 * 14 * 4
    assert need >= 2 * out_bytes
    # room for two splits only: still correct
    y2, _ = run_gpu(W, x, b, L.keep, ws=True, ws_bytes=2 * out_bytes)
    ref, den = oracle(W, x[[5]], b, L.keep)
    assert OC.max_norm_err(y2[[5]], ref, den) <= 1e-4
    # too small for any split: single pass
    y1, _ = run_gpu(W, x, b, L.keep, ws=True, ws_bytes=out_bytes)
    assert OC.max_norm_err(y1[[5]], ref, den) <= 1e-4
    xh = x.astype(np.float16)
    yh, _ = run_gpu(W, xh, b, L.keep, ws=True, dtype=torch.float16)
    ref, den = oracle(W, xh[[3]], b, L.keep)
    assert OC.max_norm_err(yh[[3]], ref, den) <= 2e-3


@pytest.mark.parametrize("idx", [13, 14, 15])
def test_resnet50_split_layers_without_workspace(idx):
    _sampled_check(WL.resnet50_3x3()[idx], 64, ws=False)
