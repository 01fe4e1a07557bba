"""pp_conv_static_scratch: the entry point for callers that may not allocate device memory.

Such callers (code inside a host runtime that owns every device allocation, plugins that must
not allocate while serving) still pass x, y and bias, and the split of the input channels keeps
its partial sums in the library's own static device array instead of a caller workspace.  The
test calls the entry point through the C ABI.  It first fills the array with wrong partial sums
(the same layer on the negated input), then runs the checked call twice in a row and compares
both results with the workspace entry point pp_conv_ws and with the oracle on two sampled
images, within the tolerance of the other conv tests: a call that read a partial sum it did not
write would fail.  The file sorts last so that a run stopping at the first failure has already
run every other test.
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

PP_ERR_NULL = -1
PP_ERR_ARG = -11
PP_ERR_SCRATCH = -13


def _call_static(lib, layer, x, b, y, relu=1):
    N, _, H, W = x.shape if x is not None else y.shape
    xp = ctypes.c_void_p(x.data_ptr()) if x is not None else None
    return lib.pp_conv_static_scratch(layer._h, xp, 0, N, H, W, ctypes.c_void_p(b.data_ptr()), relu,
                                      ctypes.c_void_p(y.data_ptr()), None)


def test_static_scratch_entry_point_matches_workspace_entry_point():
    lib = _lib.load()
    cap = ctypes.c_size_t()
    assert lib.pp_static_scratch_bytes(ctypes.byref(cap)) == 0 and cap.value == 32 << 20

    L = WL.vgg16()[10]                                # 512 -> 512 at 14x14: split input channels
    W, bias = WL.weights(L), WL.bias(L)
    x_np = WL.layer_input(L, 16)
    layer = api.pp_pack(W, None, L.keep).bind("cuda")
    x = torch.from_numpy(x_np).cuda()
    b = torch.from_numpy(bias).cuda()
    plan = layer.plan(x.shape, cap.value)             # the split the static call runs
    need = plan["workspace_bytes"]
    assert plan["splits"] > 1 and 0 < need <= cap.value

    ws = torch.empty(need // 4, dtype=torch.float32, device="cuda")
    ref = layer.conv(x, b, True, workspace=ws)
    torch.cuda.synchronize()

    # leave wrong partial sums in the array: same layer and split on the negated input
    junk = torch.empty_like(ref)
    assert _call_static(lib, layer, -x, b, junk, relu=0) == 0
    torch.cuda.synchronize()
    assert (junk - ref).abs().max().item() > 0.1

    Wh = OPR.project(W, OP.default8(), L.keep)["W_hat"]
    idx = [0, 15]
    oracle = OC.conv_ref(x_np[idx].astype(np.float64), Wh, bias, 1, True)
    den = OC.denominator(x_np.astype(np.float64), Wh, bias, 1)
    ref_h = ref.double().cpu().numpy()
    for _ in range(2):                                # two calls in a row share the array
        y = torch.full_like(ref, float("nan"))
        assert _call_static(lib, layer, x, b, y) == 0
        torch.cuda.synchronize()
        y_h = y.double().cpu().numpy()
        err = OC.max_norm_err(y_h, ref_h, den)
        assert err <= 1e-4, f"static-scratch result differs from pp_conv_ws: {err:.3e}"
        err = OC.max_norm_err(y_h[idx], oracle, den[idx])
        assert err <= 1e-4, f"static-scratch result differs from the oracle: {err:.3e}"


def test_static_scratch_rejects_calls_beyond_its_size():
    lib = _lib.load()
    # a wide layer on small images: few CTAs, so the plan splits the input channels, and for
    # some batch the partial sums of that split outgrow the 32 MiB array (calls below that batch
    # run normally on zero inputs)
    C = 1024
    W = np.random.default_rng(0).standard_normal((C, C, 3, 3)).astype(np.float32)
    layer = api.pp_pack(W, None, 0.25).bind("cuda")
    b = torch.zeros(C, device="cuda")
    shape = None
    for n in (16, 32, 64, 96, 128):
        x = torch.zeros((n, C, 7, 7), device="cuda")
        y = torch.zeros((n, C, 7, 7), device="cuda")
        rc = _call_static(lib, layer, x, b, y)
        torch.cuda.synchronize()
        if rc == PP_ERR_SCRATCH:
            shape = (n, C, 7, 7)
            break
        assert rc == 0 and torch.count_nonzero(y).item() == 0
    assert shape is not None, "no call shape needs more scratch than the static array"
    # argument errors come before the size check
    assert _call_static(lib, layer, None, b, y) == PP_ERR_NULL
    assert _call_static(lib, layer, x, b, y, relu=2) == PP_ERR_ARG
    assert b"static scratch" in lib.pp_status_string(PP_ERR_SCRATCH)
