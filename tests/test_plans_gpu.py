"""GPU parity of every launch plan the planner can choose, and of the single-layer sweep at its
full batch.

Each case states the plan outcome it exercises and asserts it through layer.plan (the same plan
the launch uses): linear tiles, rectangles of several whole images, bands of block rows of
several images, the bank-group lane order,
blocks shifted to start at output columns 4j - 1 (4j - 2 under the fp32 fused pool), the copy
fallback for rows that are not a multiple of 16 bytes, fp16 stages through TMA without the fused
pool, input-channel splits up to 32 ways, the balanced schedule, more units than one persistent
CTA per SM can hold in its table, and the fused pool.
Outputs are compared with the float64 oracle (§4.1 Eq. 1 over the projection of §4.3-4.4) on
two sampled images of the full batch; the bar is 1e-4 of sum|W_hat||x| for fp32 I/O and 2e-3 for
fp16 I/O.  Inputs come from the seeded generators only."""
import numpy as np
import pytest
import torch

from oracle import conv as OC
from oracle import patterns as OP
from oracle import project as OPR
from paper_2003_06513_gb300 import api
from paper_2003_06513_gb300 import workloads as WL

pytestmark = pytest.mark.gpu

TOL = {"f32": 1e-4, "f16": 2e-3}
SMS_TABLE = 64        # units one persistent CTA holds in its table


CAP = 32 << 20        # a workspace below the balanced schedule's (39 MB): the channel split


def _run(cout, cin, n, h, w, keep, io, pool=False, stride=1, seed=0, relu_in=True, ws_cap=None):
    rng = np.random.default_rng(seed)
    W = (rng.standard_normal((cout, cin, 3, 3)) * np.sqrt(2 / (9 * cin))).astype(np.float32)
    b = (rng.standard_normal(cout) * 0.1).astype(np.float32)
    x = WL.activations((n, cin, h, w), seed + 17, relu=relu_in,
                       dtype=np.float32 if io == "f32" else np.float16)
    layer = api.pp_pack(W, None, keep, 1, stride).bind("cuda")
    xt = torch.from_numpy(x).cuda()
    nb = layer.workspace_bytes(xt.shape, pool, xt.dtype)
    if ws_cap is not None:
        nb = min(nb, ws_cap)
    ws = torch.empty(max(nb // 4, 1), device="cuda") if nb else None
    plan = layer.plan(xt.shape, nb, pool, xt.dtype)
    y = layer.conv(xt, torch.from_numpy(b).cuda(), True, workspace=ws, pool2x2=pool)
    idx = [0, n - 1] if n > 1 else [0]
    Wh = OPR.project(W, OP.default8(), keep)["W_hat"]
    xs = x[idx].astype(np.float64)
    ref = OC.conv_ref(xs, Wh, b, stride, True)
    den = OC.denominator(xs, Wh, b, stride)
    if pool:
        ref, den = OC.maxpool2x2(ref), OC.maxpool2x2(den)
    err = OC.max_norm_err(y[idx].double().cpu().numpy(), ref, den)
    assert err <= TOL[io], f"max normalised error {err:.3e}"
    return plan, y


def _sms():
    return torch.cuda.get_device_properties(0).multi_processor_count


def test_units_overflow_the_persistent_table():
    """VGG-16 layer 1 shape at batch 256: more units than one CTA per SM holds, so the launch
    takes ceil(units / 64) persistent CTAs."""
    plan, _ = _run(64, 3, 256, 224, 224, 1.0, "f32", seed=1)
    assert plan["units"] > SMS_TABLE * _sms()
    assert plan["ctas"] == -(-plan["units"] // SMS_TABLE) > _sms()


@pytest.mark.parametrize("pool", [False, True])
def test_linear_tile(pool):
    """28x28 maps at keep 1.0: lanes take consecutive blocks across image boundaries (whole
    images staged, several per tile), with a split."""
    plan, _ = _run(128, 128, 64, 28, 28, 1.0, "f32", pool=pool, seed=2)
    nb_rect = max(1, 32 * plan["spatial_warps"] // (plan["tile_by"] * plan["tile_bx"]))
    assert (plan["tile_by"], plan["tile_bx"]) == (7, 7) and plan["tile_nb"] > nb_rect   # linear
    assert plan["shift"] == 0 and plan["splits"] > 1 and plan["streamk"] == 0


@pytest.mark.parametrize("case", [
    # cout, cin, n, h, keep, io, pool, stride, workspace cap (None: what the plan asks for)
    (256, 256, 8, 28, 0.3, "f32", False, 1, None),     # bands and a channel split
    (256, 256, 8, 28, 0.3, "f32", False, 1, 0),        # bands alone
    (256, 256, 8, 28, 0.3, "f32", True, 1, None),      # fused pool, blocks at 4j - 2
    (64, 64, 16, 56, 0.4, "f16", False, 1, None),      # fp16 stages (56 halves: TMA rows)
    (256, 256, 32, 28, 0.3, "f32", False, 1, None),    # balanced schedule (VGG-16 28x28 shape)
    (256, 256, 30, 28, 0.3, "f32", False, 1, 0),       # a last band of 2 images (30 = 7 x 4 + 2)
    (64, 64, 16, 56, 0.4, "f32", False, 1, None),      # two spatial warps, bank-group lane order
    (128, 128, 8, 56, 0.4, "f32", False, 2, None),     # stride 2, two filter groups per warp
    (128, 128, 8, 56, 0.4, "f16", False, 2, 0),
])
def test_band_tiles(case):
    """Bands: full-width rectangles of whole block rows of several images side by side in one
    stage (28x28 outputs: one block row of 4 images; 56x56: one block row of 4 images over two
    spatial warps), so no output row is computed past the image."""
    cout, cin, n, h, keep, io, pool, stride, cap = case
    plan, _ = _run(cout, cin, n, h, h, keep, io, pool=pool, stride=stride, seed=40 + h + n, ws_cap=cap)
    ho = (h - 1) // stride + 1
    nby, nbx = -(-ho // 4), (ho + plan["shift"] + 3) // 4
    assert plan["tile_bx"] == nbx and plan["tile_by"] < nby and nby % plan["tile_by"] == 0
    assert plan["tile_nb"] > 1 and plan["tile_by"] * nbx * plan["tile_nb"] <= 32 * plan["spatial_warps"]
    if n == 32:
        assert plan["streamk"] == 1
    if stride == 2:
        assert plan["groups_per_warp"] == 2
    if cap == 0:
        assert plan["splits"] == 1 and plan["streamk"] == 0


@pytest.mark.parametrize("pool", [False, True])
def test_bank_group_lane_order(pool):
    """56x56 maps at keep 0.3: rows of 15 shifted blocks, each warp's blocks dealt to lanes by
    shared-memory bank group; blocks at 4j - 1 without the pool, at 4j - 2 with it."""
    plan, _ = _run(128, 128, 16, 56, 56, 0.3, "f32", pool=pool, seed=3)
    assert plan["lane_sort"] == 1 and plan["shift"] == (2 if pool else 1)


@pytest.mark.parametrize("split", [False, True])
@pytest.mark.parametrize("h,w", [(14, 28), (14, 26), (13, 27), (12, 30), (9, 13)])
def test_pool_blocks_at_4j_minus_2(h, w, split):
    """fp32 fused pool with blocks at output columns 4j - 2: widths 0, 1, 2 and 3 (mod 4), so a
    row's first block pools columns -2..1 (pooled column -1 is not stored) and its last one may
    hang over the edge; rows through TMA (28 floats) and the copy fallback (26, 27, 30, 13);
    without a workspace and with a 32-way split (pooled in the split's reduction)."""
    plan, _ = _run(64, 64, 8, h, w, 0.3, "f32", pool=True, seed=20 + w, ws_cap=None if split else 0)
    assert plan["shift"] == 2 and (plan["splits"] > 1) == split


def test_multi_image_rectangles_with_split():
    """7x7 maps: rectangles of 8 whole images (2x2 blocks each) and an 8-way split (a workspace
    too small for the balanced schedule)."""
    plan, _ = _run(256, 256, 64, 7, 7, 0.5, "f32", seed=4, ws_cap=CAP)
    assert plan["tile_nb"] == 8 and plan["splits"] > 1 and plan["streamk"] == 0


@pytest.mark.parametrize("pool", [False, True])
def test_balanced_schedule(pool):
    """VGG-16 layer 9's shape (512 -> 512, 28x28, keep 0.3, batch 32, fp32): 256 whole units
    would take 1.7 waves; the balanced schedule spreads their chunks over 152 CTAs and every
    unit cut between two CTAs is summed by its head CTA."""
    plan, _ = _run(512, 512, 32, 28, 28, 0.3, "f32", pool=pool, seed=11)
    assert plan["streamk"] == 1 and plan["splits"] == 1 and plan["ctas"] == _sms()
    assert plan["units"] % _sms() != 0


def test_balanced_schedule_fp16():
    """fp16 rows of 56 elements (112 bytes, through TMA), 154 units (just over one wave) on 152
    CTAs: almost every CTA holds a head of one unit and a part of the next."""
    plan, _ = _run(256, 256, 11, 56, 56, 0.3, "f16", seed=12)
    assert plan["streamk"] == 1 and _sms() < plan["units"] < 2 * _sms()


def test_no_balanced_schedule_without_tma_rows():
    """fp16 rows of 28 elements (56 bytes: the copy fallback, one CTA per unit): the planner
    keeps whole units (and the channel split) there."""
    plan, _ = _run(512, 512, 32, 28, 28, 0.3, "f16", seed=13)
    assert plan["streamk"] == 0


@pytest.mark.parametrize("cout,cin,n,h,io,groups", [
    (128, 64, 16, 56, "f32", 2),    # ResNet-50's first stage head, at a smaller batch
    (40, 24, 3, 30, "f32", 2),      # 5 filter groups: one warp's second group missing, one warp idle
    (256, 128, 8, 28, "f16", 2),    # fp16 stages
    (64, 32, 4, 29, "f32", 2),      # odd map: the copy fallback, a ragged last block row and column
    (8, 16, 2, 20, "f32", 1),       # a single filter group: one group per warp
])
def test_stride2_two_groups_per_warp(cout, cin, n, h, io, groups):
    """Stride-2 launches give each warp two filter groups (8 warps of 16 slots, one input window
    per lane serving both groups' kept kernels) wherever a unit holds two groups or more."""
    plan, _ = _run(cout, cin, n, h, h, 0.4, io, stride=2, seed=30 + h)
    assert plan["groups_per_warp"] == groups


def test_stride2_balanced_schedule():
    """512 input channels, 128 whole units at stride 2: the balanced schedule over 152 CTAs with
    two filter groups per warp (a part's 16 slots per warp go to its workspace slot)."""
    plan, _ = _run(256, 512, 32, 56, 56, 0.4, "f32", stride=2, seed=41)
    assert plan["streamk"] == 1 and plan["groups_per_warp"] == 2 and plan["ctas"] == _sms()


@pytest.mark.parametrize("shape", [(5, 64, 1, 13, 13), (5, 64, 3, 13, 11), (24, 96, 1, 7, 7),
                                   (64, 64, 1, 75, 75), (128, 64, 1, 55, 55)])
def test_split_reduction_element_counts(shape):
    """The split reduction takes 4 outputs per thread (16-byte loads of every split) where the
    output count is a multiple of 4 and large (360 000 and 387 200 here, planes of 5625 and 3025
    outputs, so quads cross from one output plane into the next and take each element's own
    bias), else one output per thread (845, 2145 and 1176)."""
    cout, cin, n, h, w = shape
    plan, _ = _run(cout, cin, n, h, w, 0.5, "f32", seed=50 + h + n)
    assert plan["splits"] > 8


def test_batch_one_split_32_ways():
    plan, _ = _run(256, 256, 1, 14, 14, 0.25, "f32", seed=5)
    assert plan["splits"] == 32 and plan["shift"] == 1


@pytest.mark.parametrize("io", ["f32", "f16"])
def test_copy_fallback_rows(io):
    """Rows of 30 elements (120 / 60 bytes: no tensor copy), shifted blocks, split."""
    plan, _ = _run(64, 32, 4, 20, 30, 0.5, io, seed=6)
    assert plan["shift"] == 1 and plan["splits"] > 1


@pytest.mark.parametrize("pool", [False, True])
def test_fp16_through_tma(pool):
    """fp16 rows of 56 elements (112 bytes): fp16 stages through TMA, with and without the pool."""
    plan, _ = _run(128, 128, 16, 56, 56, 0.3, "f16", pool=pool, seed=7)
    assert plan["shift"] == (0 if pool else 1)


@pytest.mark.parametrize("io", ["f32", "f16"])
def test_stride2_heads(io):
    """Stride 2 with two filter groups per warp over bands of 4 images: fp32 deals each warp's
    blocks to lanes by shared-memory bank group (window column 0 from the left block's lane by an
    indexed shuffle); fp16 keeps the raster order."""
    plan, _ = _run(128, 128, 16, 56, 56, 0.4, io, stride=2, seed=8)
    assert plan["shift"] == 0 and plan["groups_per_warp"] == 2 and plan["tile_nb"] > 1
    assert plan["lane_sort"] == (1 if io == "f32" else 0)


# the single-layer sweep (C = Cin = Cout, H = W, batch, keep, io) at full batch
SWEEP = [(128, 56, 64, 1.0, "f32"), (256, 28, 256, 0.25, "f16"), (512, 14, 256, 0.5, "f32"),
         (512, 7, 256, 0.25, "f16"), (256, 56, 16, 0.25, "f16"), (128, 28, 64, 1.0, "f16"),
         (256, 14, 1, 1.0, "f32"), (512, 28, 16, 0.5, "f32"), (128, 7, 16, 1.0, "f32")]


@pytest.mark.parametrize("c,hw,n,keep,io", SWEEP)
def test_sweep_point_full_batch(c, hw, n, keep, io):
    """Points of the 288-point sweep at their full batch, with the sweep's own seeds (weights,
    bias) and N(0,1) inputs as the sweep draws them."""
    pts = [(L, nn, dt) for L, nn, dt in WL.sweep() if (L.cin, L.h, nn, L.keep, dt) == (c, hw, n, keep, io)]
    assert len(pts) == 1
    L, _, _ = pts[0]
    W, b = WL.weights(L), WL.bias(L)
    x = WL.activations((n, c, hw, hw), L.x_seed, dtype=np.float32 if io == "f32" else np.float16)
    layer = api.pp_pack(W, None, keep).bind("cuda")
    xt = torch.from_numpy(x).cuda()
    nb = layer.workspace_bytes(xt.shape, dtype=xt.dtype)
    ws = torch.empty(max(nb // 4, 1), device="cuda") if nb else None
    y = layer.conv(xt, torch.from_numpy(b).cuda(), True, workspace=ws)
    idx = [0, n - 1] if n > 1 else [0]
    Wh = OPR.project(W, OP.default8(), keep)["W_hat"]
    xs = x[idx].astype(np.float64)
    err = OC.max_norm_err(y[idx].double().cpu().numpy(), OC.conv_ref(xs, Wh, b, 1, True),
                          OC.denominator(xs, Wh, b, 1))
    assert err <= TOL[io], f"max normalised error {err:.3e}"
