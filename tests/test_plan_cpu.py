"""Launch planner of the pattern-sparse kernel (pp_conv_plan and pp_conv_workspace_size, host
only, no GPU): invariants every plan must keep, over random call shapes and the workloads.

The planner assumes 152 SMs (a GB300) when no GPU is present; the invariants do not depend on that."""
import numpy as np
import pytest
import torch

from oracle import patterns as OP
from paper_2003_06513_gb300 import _lib, api
from paper_2003_06513_gb300 import workloads as WL

SMEM_MAX = 227 * 1024
MAX_CHUNKS = 256      # input-channel stages one unit may walk
SMS = 152             # the planner's SM count without a GPU (a GB300)
# balanced schedule: a slot of 16 warps x 8 slots x 16 x 32 fp32 accumulators per CTA, then a flag
# per (CTA, warp)
STREAMK_BYTES = SMS * 16 * 8 * 16 * 32 * 4 + SMS * 16 * 4


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
    if pl["streamk"]:
        assert pl["splits"] == 1 and pl["ctas"] == SMS
        assert pl["workspace_bytes"] == STREAMK_BYTES <= ws
        assert pl["chunks_per_unit"] * pl["units"] >= 2 * SMS
    elif pl["splits"] == 1:
        assert pl["workspace_bytes"] == 0
    else:
        assert pl["workspace_bytes"] == pl["splits"] * out_bytes <= ws
    # every split gets whole stages of channels and covers the input channels once
    cin = shape[1]
    per_split = pl["chunks_per_unit"] * pl["channels_per_stage"]
    assert per_split * pl["splits"] >= cin > per_split * (pl["splits"] - 1)
    # units: tiles x filter chunks x splits; persistent CTAs never exceed the units
    assert pl["units"] % pl["splits"] == 0
    assert pl["ctas"] <= pl["units"] or pl["streamk"]
    # lanes by bank group: stride 1, or stride 2 with two filter groups per warp
    assert pl["lane_sort"] in (0, 1) and (layer.stride == 1 or pl["lane_sort"] == 0 or pl["groups_per_warp"] == 2)
    assert pl["shift"] in (0, 1, 2) and (layer.stride == 1 or pl["shift"] == 0)
    assert pl["streamk"] in (0, 1)
    # bands (several images, fewer block rows than an image): full-width rows of block rows that
    # divide the image's, within the lanes, only for inputs through TMA (fp32 rows of a multiple
    # of 4) and below 6 kept kernels per (input channel, filter group)
    ho, wo = (shape[2] - 1) // layer.stride + 1, (shape[3] - 1) // layer.stride + 1
    nby = (ho + 3) // 4
    if pl["tile_nb"] > 1 and pl["tile_by"] < nby:
        BANDS_SEEN.append(shape)
        assert pl["tile_bx"] == _nbx(pl, wo) and nby % pl["tile_by"] == 0
        assert pl["tile_by"] * pl["tile_bx"] * pl["tile_nb"] <= 32 * pl["spatial_warps"]
        assert shape[3] % 4 == 0
        assert layer.beta / (-(-layer.cout // 8) * shape[1]) < 6
    return pl


BANDS_SEEN = []


def _nbx(pl, wo):
    """Blocks per output row: 4 columns each, starting at column 0, or at -1 or -2 when shifted."""
    return (wo + pl["shift"] + 3) // 4


def _stage_geometry(pl, stride):
    """Staged rows per (image, channel) and their width in floats, as the planner lays them out."""
    by, bx = pl["tile_by"], pl["tile_bx"]
    ih = 4 * by + 2 if stride == 1 else 8 * by + 1
    bw = 4 * bx + 8 if stride == 1 else 8 * bx + 4
    return ih, bw + 4 if bw % 8 == 0 else bw


def _is_linear(pl, shape, stride):
    """Whether the plan's tile is the linear one (None where its shape does not tell)."""
    n = shape[0]
    ho, wo = (shape[2] - 1) // stride + 1, (shape[3] - 1) // stride + 1
    nby, nbx = (ho + 3) // 4, _nbx(pl, wo)
    if (pl["tile_by"], pl["tile_bx"]) != (nby, nbx) or pl["tile_nb"] == 1:
        return False
    bpi, lanes = nby * nbx, 32 * pl["spatial_warps"]
    rect_nb = min(n, 256, max(1, lanes // bpi))
    lin_nb = min(n, (lanes - 1) // bpi + 2)
    if rect_nb == lin_nb or (bpi < lanes and lanes % bpi == 0):
        return None if rect_nb == lin_nb and not (bpi < lanes and lanes % bpi == 0) else False
    return pl["tile_nb"] == lin_nb


def _window_wavefronts(pl, shape, stride, t, dealt):
    """Wavefronts of warp 0's 16-byte window loads in tile t: 4 phases of 8 lanes, each costing
    the most lanes on one of the 8 bank groups; lanes in raster order or dealt by
    (rank within bank group, bank group) with idle lanes last.  A block's window starts 4 * stride
    elements right of its left neighbour's and 4 * stride rows below the block above."""
    n = shape[0]
    by_t, bx_t, nb = pl["tile_by"], pl["tile_bx"], pl["tile_nb"]
    lanes = 32 * pl["spatial_warps"]
    linear = bool(_is_linear(pl, shape, stride))
    ih, bw = _stage_geometry(pl, stride)
    grp = []
    for lane in range(32):
        if linear:
            b = t * lanes + lane
            img, rem = b // (by_t * bx_t) - (t * lanes) // (by_t * bx_t), b % (by_t * bx_t)
            active = b // (by_t * bx_t) < n and img < nb
        else:
            img, rem = divmod(lane, by_t * bx_t)
            active = img < nb
        off = img * pl["channels_per_stage"] * ih * bw + (rem // bx_t) * 4 * stride * bw + (rem % bx_t) * 4 * stride
        grp.append((off // 4) % 8 if active else None)
    order = list(range(32))
    if dealt:
        seen, keys = {}, []
        for lane, g in enumerate(grp):
            if g is None:
                keys.append((1 << 20) + lane)
            else:
                keys.append(16 * seen.get(g, 0) + g)
                seen[g] = seen.get(g, 0) + 1
        order = sorted(range(32), key=lambda lane: keys[lane])
    w = 0
    for ph in range(4):
        gs = [grp[lane] for lane in order[8 * ph:8 * ph + 8] if grp[lane] is not None]
        w += max([gs.count(g) for g in set(gs)] or [0])
    return w


@pytest.mark.parametrize("which", ["vgg16", "resnet50"])
def test_lane_order_by_bank_group(which):
    """The planner deals blocks to lanes by bank group exactly where that lowers the modelled
    wavefronts of the window loads (stride 1, and stride 2 with two filter groups per warp): on
    VGG-16 the 56x56 layers (rows of 14 blocks), not the others; on ResNet-50 the stride-2 heads
    (a row's blocks 32 bytes apart, on every other bank group; images in between on the others)."""
    layers = WL.vgg16() if which == "vgg16" else WL.resnet50_3x3()
    n = 32 if which == "vgg16" else 64
    got = {}
    for L in layers:
        layer = api.pp_pack(WL.weights(L), None, L.keep, 1, L.stride)
        shape = (n, L.cin, L.h, L.w)
        pl = layer.plan(shape, layer.workspace_bytes(shape))
        got[L.name] = pl["lane_sort"]
        if L.stride != 1 and pl["groups_per_warp"] != 2:
            assert pl["lane_sort"] == 0
            continue
        tiles = 1
        ho, wo = L.ho, L.wo
        nby, nbx = (ho + 3) // 4, _nbx(pl, wo)
        if _is_linear(pl, shape, L.stride):
            tiles = min(64, (n * nby * nbx + 31) // 32)
        raster = sum(_window_wavefronts(pl, shape, L.stride, t, False) for t in range(tiles))
        dealt = sum(_window_wavefronts(pl, shape, L.stride, t, True) for t in range(tiles))
        assert pl["lane_sort"] == (1 if dealt < raster else 0), (L.name, raster, dealt)
    if which == "vgg16":
        assert [got[f"vgg{i}"] for i in range(1, 14)] == [0, 0, 0, 0, 1, 1, 1, 0, 0, 0, 0, 0, 0]
    else:   # the stride-2 heads: several images a tile, an odd image stride in bank groups
        assert [got[L.name] for L in layers if L.stride == 2] == [1, 1, 1]


def test_multi_image_stages_are_not_bank_aligned():
    """Where an 8-lane phase of the window loads holds blocks of several images (fewer than 8
    blocks per image, stride 1), the image stride in the stage is no multiple of 32 floats, which
    would put every image's windows on the same banks (ResNet-50's 7x7 layers: 2x2 blocks)."""
    seen = 0
    for which, n in (("vgg16", 32), ("resnet50", 64)):
        layers = WL.vgg16() if which == "vgg16" else WL.resnet50_3x3()
        for L in layers:
            layer = api.pp_pack(WL.weights(L), None, L.keep, 1, L.stride)
            shape = (n, L.cin, L.h, L.w)
            pl = layer.plan(shape, layer.workspace_bytes(shape))
            if (L.stride == 1 and pl["tile_nb"] > 1 and pl["tile_by"] * pl["tile_bx"] < 8
                    and pl["channels_per_stage"] > 1):
                ih, bw = _stage_geometry(pl, L.stride)
                assert (pl["channels_per_stage"] * ih * bw) % 32 != 0, L.name
                seen += 1
    assert seen == 2


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
    before = len(BANDS_SEEN)
    for L in layers:
        layer = api.pp_pack(WL.weights(L), None, L.keep, 1, L.stride)
        shape = (n, L.cin, L.h, L.w)
        for ws in (0, layer.workspace_bytes(shape), 1 << 20):
            _check(layer, shape, ws)
    assert len(BANDS_SEEN) > before       # the 28x28 (and ResNet-50's 56x56) layers take bands


def test_other_paths_report_no_plan():
    rng = np.random.default_rng(3)
    dw = api.pp_pack(rng.standard_normal((16, 1, 3, 3)).astype(np.float32), None, 1.0, 16, 1)
    assert dw.plan((2, 16, 20, 20), 0)["path"] == 2
    masks = [OP.mask_of(t) for t in ([0, 4, 5, 8], [1, 4, 6, 7], [2, 3, 4, 8])]
    gen = api.pp_pack(rng.standard_normal((8, 4, 3, 3)).astype(np.float32), masks, 0.5)
    assert gen.plan((1, 4, 9, 9), 0)["path"] == 3
    assert gen.workspace_bytes((1, 4, 9, 9)) == 0


def test_linear_tile_weighed_by_density():
    """28x28 maps with blocks at columns 4j (7 blocks a row, the fp16 fused-pool layout, rows
    through the copy fallback): at VGG-16's keep 0.3 the planner takes 4x7 rectangles without a
    split; at keep 1.0 the linear tile (every lane busy) pays for its per-channel cost.  With
    blocks at 4j - 1 (no pool) or 4j - 2 (fp32 pool) a row has 8 blocks, and fp32 rows go through
    TMA: bands of one block row of 4 images keep every lane busy and compute the 7 block rows of
    an image exactly (rectangles of 4 block rows compute 8), on the balanced schedule."""
    f16 = torch.float16
    for L in WL.vgg16()[7:10]:
        layer = api.pp_pack(WL.weights(L), None, L.keep)
        shape = (32, L.cin, L.h, L.w)
        pl = layer.plan(shape, layer.workspace_bytes(shape, True, f16), pool2x2=True, dtype=f16)
        assert (pl["tile_by"], pl["tile_bx"], pl["tile_nb"], pl["splits"], pl["shift"]) == (4, 7, 1, 1, 0), L.name
        pl = layer.plan(shape, layer.workspace_bytes(shape, True), pool2x2=True)
        assert (pl["tile_by"], pl["tile_bx"], pl["tile_nb"], pl["splits"], pl["shift"]) == (1, 8, 4, 1, 2), L.name
        assert pl["streamk"] == 1, L.name
        pl = layer.plan(shape, layer.workspace_bytes(shape))
        assert (pl["tile_by"], pl["tile_bx"], pl["tile_nb"], pl["splits"], pl["shift"]) == (1, 8, 4, 1, 1), L.name
        assert pl["streamk"] == 1, L.name
    rng = np.random.default_rng(7)
    W = (rng.standard_normal((256, 256, 3, 3)) * np.sqrt(2 / (9 * 256))).astype(np.float32)
    shape = (64, 256, 28, 28)
    dense = api.pp_pack(W, None, 1.0)
    pl = dense.plan(shape, dense.workspace_bytes(shape, True, f16), pool2x2=True, dtype=f16)
    assert (pl["tile_by"], pl["tile_bx"]) == (7, 7) and pl["tile_nb"] > 1     # linear
    sparse = api.pp_pack(W, None, 0.25)
    pl = sparse.plan(shape, sparse.workspace_bytes(shape, True, f16), pool2x2=True, dtype=f16)
    assert (pl["tile_by"], pl["tile_bx"], pl["tile_nb"]) == (4, 7, 1)


@pytest.mark.parametrize("which", ["vgg16", "resnet50"])
def test_pool_plans_keep_block_origins_even(which):
    """The fused pool needs every 2x2 window inside one lane's block: its plans start blocks at
    4j, or at 4j - 2 for fp32, never at 4j - 1, and they obey the same invariants.  Layers without
    the fused pool refuse the query."""
    layers = WL.vgg16() if which == "vgg16" else WL.resnet50_3x3()
    n = 32 if which == "vgg16" else 64
    for L in layers:
        layer = api.pp_pack(WL.weights(L), None, L.keep, 1, L.stride)
        shape = (n, L.cin, L.h, L.w)
        for ws in (0, layer.workspace_bytes(shape, True)):
            pl = layer.plan(shape, ws, pool2x2=True)
            assert pl["path"] == 1 and pl["shift"] in (0, 2)
            assert layer.plan(shape, ws, pool2x2=True, dtype=torch.float16)["shift"] == 0
            assert 0 < pl["smem_bytes"] <= SMEM_MAX and pl["filter_groups"] * pl["spatial_warps"] == 16
    rng = np.random.default_rng(3)
    dw = api.pp_pack(rng.standard_normal((16, 1, 3, 3)).astype(np.float32), None, 1.0, 16, 1)
    with pytest.raises(_lib.PatconvError):
        dw.plan((2, 16, 20, 20), 0, pool2x2=True)


@pytest.mark.parametrize("seed", range(30))
def test_lane_order_random_shapes(seed):
    """The planner's bank-group lane order agrees with an independent model of the window loads'
    wavefronts on random stride-1 shapes (rectangles and linear tiles)."""
    rng = np.random.default_rng(100 + seed)
    c = int(rng.choice([16, 64, 128, 256]))
    n = int(rng.choice([1, 2, 3, 8, 32]))
    h, w = int(rng.integers(5, 120)), int(rng.integers(5, 120))
    keep = float(rng.choice([1.0, 0.5, 0.3]))
    W = rng.standard_normal((c, c, 3, 3)).astype(np.float32)
    layer = api.pp_pack(W, None, keep)
    shape = (n, c, h, w)
    for ws in (0, layer.workspace_bytes(shape)):
        pl = layer.plan(shape, ws)
        linear = _is_linear(pl, shape, 1)
        if linear is None:
            continue
        tiles = 1
        if linear:
            nby, nbx = (h + 3) // 4, _nbx(pl, w)
            tiles = min(64, (n * nby * nbx + 32 * pl["spatial_warps"] - 1) // (32 * pl["spatial_warps"]))
        raster = sum(_window_wavefronts(pl, shape, 1, t, False) for t in range(tiles))
        dealt = sum(_window_wavefronts(pl, shape, 1, t, True) for t in range(tiles))
        assert pl["lane_sort"] == (1 if dealt < raster else 0), (shape, ws, raster, dealt, pl)


def test_one_handle_planned_from_many_threads():
    """pp_conv_plan from 8 host threads on one fresh handle at once: every thread gets the same
    plans (the per-handle plan cache is created once and guarded; ctypes releases the GIL)."""
    import threading
    rng = np.random.default_rng(21)
    W = rng.standard_normal((256, 128, 3, 3)).astype(np.float32)
    layer = api.pp_pack(W, None, 0.3)
    shapes = [(n, 128, h, h) for n in (1, 8, 32) for h in (7, 14, 28, 56)]
    out, errors = [None] * 8, []

    def work(i):
        try:
            got = []
            for rep in range(5):
                for sh in shapes[i % 3:] + shapes[:i % 3]:
                    got.append((sh, tuple(layer.plan(sh, 1 << 30).items())))
            out[i] = sorted(set(got))
        except Exception as e:        # pragma: no cover - reported below
            errors.append(e)
    threads = [threading.Thread(target=work, args=(i,)) for i in range(8)]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    assert not errors
    assert all(o == out[0] for o in out) and len(out[0]) == len(shapes)


# --------------------------------------------------------------------------- streamed depthwise

SMEM_OPTIN = 232448   # shared memory one CTA may opt into on a GB300


def _dw_layer(C, stride=1, seed=5):
    rng = np.random.default_rng(seed)
    return api.pp_pack(rng.standard_normal((C, 1, 3, 3)).astype(np.float32), None, 1.0, C, stride)


@pytest.mark.parametrize("idx,kernel", [(0, 1), (1, 1), (2, 1), (3, 1),      # 112 / 56-wide rows
                                        (4, 6), (7, 6), (11, 6),             # 28 / 14-wide tiles
                                        (13, 7), (14, 5), (6, 7)])           # 14 -> 7, 28 -> 14, 7-wide
def test_streamed_depthwise_mode_per_mobilenet_layer(idx, kernel):
    """MobileNet-V2's fp16 layers at batch 128: 112- and 56-wide maps stream bands of whole rows
    through tensor copies (rows of 224 or 112 bytes); 28-, 14- and 7-wide maps stream runs of whole
    planes, each lane a band of 7 output rows by 7 or 14 columns."""
    L = WL.mobilenet_v2_dw()[idx]
    lay = _dw_layer(L.cout, L.stride)
    pl = lay.plan((128, L.cin, L.h, L.w), 0, dtype=torch.float16)
    assert pl["path"] == 2 and pl["dw_kernel"] == kernel, pl
    assert 2 <= pl["stages"] <= 4 and pl["smem_bytes"] <= SMEM_OPTIN
    es, ho, wo = 2, L.ho, L.wo
    n_planes = 128 * L.cout
    if kernel == 1:   # rows mode: bands of R output rows, every band's input rows in one stage
        R = pl["rows_or_planes"]
        assert 1 <= R <= ho and ((R - 1) * L.stride + 3) * L.w * es <= 4096
        assert pl["chunks"] == n_planes * -(-ho // R)
    else:             # planes and tiles modes: chunk starts 16-byte aligned in x and y
        P = pl["rows_or_planes"]
        assert (P * L.h * L.w * es) % 16 == 0 and (P * ho * wo * es) % 16 == 0
        assert pl["chunks"] == -(-n_planes // P)
        if kernel >= 5:   # tiles: lane items (plane, 7 output rows, 7 or 14 columns), 32 a pass
            items = P * (ho // 7) * (wo // (14 if kernel == 6 else 7))
            assert items % 32 == 0
        else:
            lpp = -(-wo // (1 if kernel == 2 else 2))
            assert lpp <= 32 and P % (32 // lpp) == 0      # whole passes of the warp
    assert 4 <= pl["warps"] <= 16
    assert pl["ctas"] == min(152, -(-pl["chunks"] // pl["warps"]))


@pytest.mark.parametrize("shape,stride,dtype,kernel", [
    ((3, 21, 13, 12), 1, torch.float32, 1),     # 48-byte rows
    ((3, 21, 13, 12), 2, torch.float32, 2),     # 6 output columns: planes
    ((3, 21, 13, 12), 1, torch.float16, 3),     # 24-byte rows: planes, two columns a lane
    ((2, 24, 9, 9), 1, torch.float32, 4),       # odd width
    ((1, 4, 9, 2100), 1, torch.float16, 0),     # rows too wide for either mode
    ((2, 16, 20, 100), 1, torch.float16, 0),    # 200-byte rows, 100 columns: neither mode
])
def test_streamed_depthwise_applicability(shape, stride, dtype, kernel):
    lay = _dw_layer(shape[1], stride)
    assert lay.plan(shape, 0, dtype=dtype)["dw_kernel"] == kernel
