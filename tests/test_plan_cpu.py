"""Launch planner of the pattern-sparse kernel (pp_conv_plan and pp_conv_workspace_size, host
only, no GPU): invariants every plan must keep, over random call shapes and the workloads.

The planner assumes 148 SMs when no GPU is present; the invariants do not depend on that."""
import numpy as np
import pytest

from oracle import patterns as OP
from paper_2003_06513_gb300 import api
from paper_2003_06513_gb300 import workloads as WL

SMEM_MAX = 227 * 1024
MAX_CHUNKS = 256      # input-channel stages one unit may walk


def _check(layer, shape, ws):
    pl = layer.plan(shape, ws)
    assert pl["path"] == 1
    assert pl["splits"] >= 1 and pl["units"] >= 1 and pl["ctas"] >= 1
    assert 1 <= pl["channels_per_stage"] <= 64
    assert pl["tile_by"] >= 1 and pl["tile_bx"] >= 1 and pl["tile_nb"] >= 1
    assert pl["filter_groups"] * pl["spatial_warps"] == 16
    assert 0 < pl["smem_bytes"] <= SMEM_MAX
    assert 1 <= pl["chunks_per_unit"] <= MAX_CHUNKS
    # a split needs its workspace, and never more than the caller gave
    out_bytes = 4 * shape[0] * layer.cout * ((shape[2] - 1) // layer.stride + 1) * ((shape[3] - 1) // layer.stride + 1)
    if pl["splits"] == 1:
        assert pl["workspace_bytes"] == 0
    else:
        assert pl["workspace_bytes"] == pl["splits"] * out_bytes <= ws
    # every split gets whole stages of channels and covers the input channels once
    cin = shape[1]
    per_split = pl["chunks_per_unit"] * pl["channels_per_stage"]
    assert per_split * pl["splits"] >= cin > per_split * (pl["splits"] - 1)
    # units: tiles x filter chunks x splits; persistent CTAs never exceed the units
    assert pl["units"] % pl["splits"] == 0
    assert pl["ctas"] <= pl["units"]
    return pl


@pytest.mark.parametrize("seed", range(40))
def test_random_shapes(seed):
    rng = np.random.default_rng(seed)
    cin = int(rng.choice([1, 3, 7, 16, 33, 64, 130, 256, 512, 1024]))
    cout = int(rng.choice([1, 5, 8, 24, 64, 129, 256, 512]))
    n = int(rng.choice([1, 2, 5, 16, 32, 64]))
    h, w = int(rng.integers(1, 80)), int(rng.integers(1, 300))
    stride = int(rng.choice([1, 2]))
    keep = float(rng.choice([1.0, 0.5, 0.3, 0.1]))
    W = rng.standard_normal((cout, cin, 3, 3)).astype(np.float32)
    layer = api.pp_pack(W, None, keep, 1, stride)
    shape = (n, cin, h, w)
    full = layer.workspace_bytes(shape)
    _check(layer, shape, 0)
    pl = _check(layer, shape, full)
    assert pl["workspace_bytes"] == full      # the query reports what the launch would use


@pytest.mark.parametrize("which", ["vgg16", "resnet50"])
def test_workload_plans(which):
    layers = WL.vgg16() if which == "vgg16" else WL.resnet50_3x3()
    n = 32 if which == "vgg16" else 64
    for L in layers:
        layer = api.pp_pack(WL.weights(L), None, L.keep, 1, L.stride)
        shape = (n, L.cin, L.h, L.w)
        for ws in (0, layer.workspace_bytes(shape), 1 << 20):
            _check(layer, shape, ws)


def test_other_paths_report_no_plan():
    rng = np.random.default_rng(3)
    dw = api.pp_pack(rng.standard_normal((16, 1, 3, 3)).astype(np.float32), None, 1.0, 16, 1)
    assert dw.plan((2, 16, 20, 20), 0)["path"] == 2
    masks = [OP.mask_of(t) for t in ([0, 4, 5, 8], [1, 4, 6, 7], [2, 3, 4, 8])]
    gen = api.pp_pack(rng.standard_normal((8, 4, 3, 3)).astype(np.float32), masks, 0.5)
    assert gen.plan((1, 4, 9, 9), 0)["path"] == 3
    assert gen.workspace_bytes((1, 4, 9, 9)) == 0
