"""Failure detection of the dense kernel's pipeline, in the form this hardware allows: a wait
that runs out records a status bit and the kernel returns, so the context stays usable.

pp_debug_inject_timeout makes the next launch issue none of its stage copies and wait only about
10 us for them (the barrier it waits on is one that nothing arrives on).  No fault, trap or hang
is involved: every wait is bounded and nothing is in flight when the kernel exits.
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

FULL_TIMEOUT = 1     # status bit: a stage's data never arrived


def _status(clear):
    st = ctypes.c_uint(0)
    assert _lib.load().pp_device_status(1 if clear else 0, ctypes.byref(st)) == 0
    return st.value


@pytest.mark.parametrize("dtype", [torch.float32, torch.float16])
def test_pipeline_wait_runs_out_then_next_call_is_correct(dtype):
    lib = _lib.load()
    torch.cuda.synchronize()
    assert _status(True) == 0
    rng = np.random.default_rng(5)
    W = (rng.standard_normal((64, 48, 3, 3)) * np.sqrt(2 / (9 * 48))).astype(np.float32)
    x_np = WL.activations((2, 48, 40, 36), 9, relu=True,
                          dtype=np.float32 if dtype == torch.float32 else np.float16)
    b_np = (rng.standard_normal(64) * 0.1).astype(np.float32)
    layer = api.pp_pack(W, None, 0.5).bind("cuda")
    x = torch.from_numpy(x_np).cuda()
    b = torch.from_numpy(b_np).cuda()
    assert layer.plan(x.shape, 0)["splits"] == 1

    y = torch.full((2, 64, 40, 36), float("nan"), dtype=dtype, device="cuda")
    assert lib.pp_debug_inject_timeout() == 0
    layer.conv(x, b, True, out=y)                 # the launch itself succeeds
    torch.cuda.synchronize()
    assert _status(True) & FULL_TIMEOUT
    assert torch.isnan(y).all()                   # the timed-out kernel wrote nothing

    y = layer.conv(x, b, True)                    # the next call runs normally
    torch.cuda.synchronize()
    assert _status(True) == 0
    Wh = OPR.project(W, OP.default8(), 0.5)["W_hat"]
    ref = OC.conv_ref(x_np.astype(np.float64), Wh, b_np, 1, True)
    den = OC.denominator(x_np.astype(np.float64), Wh, b_np, 1)
    tol = 1e-4 if dtype == torch.float32 else 2e-3
    assert OC.max_norm_err(y.double().cpu().numpy(), ref, den) <= tol
