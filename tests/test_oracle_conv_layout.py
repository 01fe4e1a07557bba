"""Pins of the oracle's convolution and layout (CPU only).

The convolution is pinned to hand-computed values and to torch's CPU float64 ``conv2d`` (a
library routine the oracle does not call); the layout to a hand-packed fixture and to a decoder
that must rebuild the projected weights from the sections.
"""
import numpy as np
import pytest
import torch
import torch.nn.functional as Fnn

from conftest import golden_kv, golden_lines
from oracle import conv as C
from oracle import layout as L
from oracle import patterns as P
from oracle import project as PR


def _f(v):
    return np.array([float(a) for a in v], dtype=np.float64)


def _hand_case():
    g = golden_kv("conv_hand.txt")
    W = np.stack([_f(g["w_ci0"]), _f(g["w_ci1"])]).reshape(1, 2, 3, 3).astype(np.float32)
    x = np.stack([_f(g["x_ci0"]), _f(g["x_ci1"])]).reshape(1, 2, 3, 3).astype(np.float32)
    return g, W, x


@pytest.mark.parametrize("fn", [C.conv_loop, C.conv_ref])
def test_hand_convolution(fn):
    g, W, x = _hand_case()
    np.testing.assert_array_equal(fn(x, W, None, 1).reshape(9), _f(g["y_stride1"]))
    b = np.array([float(g["bias"][0])], np.float32)
    np.testing.assert_array_equal(fn(x, W, b, 1, relu=True).reshape(9),
                                  _f(g["y_stride1_bias_relu"]))
    np.testing.assert_array_equal(fn(x, W, None, 2).reshape(4), _f(g["y_stride2"]))


def test_hand_weights_are_patterns():
    """The fixture's two kernels are p0 and p4 exactly; projection leaves them unchanged."""
    _, W, _ = _hand_case()
    r = PR.project(W, P.default8(), 1.0)
    assert r["pid"].tolist() == [[0, 4]]
    np.testing.assert_array_equal(r["W_hat"], W)


def _torch_ref(x, W, b, stride, relu, depthwise):
    xt = torch.from_numpy(np.asarray(x, np.float64))
    wt = torch.from_numpy(np.asarray(W, np.float64))
    bt = None if b is None else torch.from_numpy(np.asarray(b, np.float64))
    y = Fnn.conv2d(xt, wt, bt, stride=stride, padding=1, groups=x.shape[1] if depthwise else 1)
    return (torch.relu(y) if relu else y).numpy()


@pytest.mark.parametrize("N,Cin,Cout,H,W,s,dw,relu", [
    (1, 1, 1, 1, 1, 1, False, False), (2, 3, 5, 7, 6, 1, False, True), (1, 4, 3, 5, 9, 2, False, False),
    (2, 6, 6, 8, 7, 2, True, True), (1, 5, 5, 4, 4, 1, True, False), (1, 2, 9, 2, 3, 2, False, True)])
def test_conv_loop_and_ref_match_torch(N, Cin, Cout, H, W, s, dw, relu):
    rng = np.random.default_rng(N * 100 + Cin * 10 + H)
    x = rng.standard_normal((N, Cin, H, W)).astype(np.float32)
    cin_g = 1 if dw else Cin
    Wt = rng.standard_normal((Cout, cin_g, 3, 3)).astype(np.float32)
    Wh = PR.project(Wt, P.default8(), 0.6)["W_hat"]
    b = rng.standard_normal(Cout).astype(np.float32)
    ref = _torch_ref(x, Wh, b, s, relu, dw)
    np.testing.assert_allclose(C.conv_loop(x, Wh, b, s, relu, dw), ref, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(C.conv_ref(x, Wh, b, s, relu, dw), ref, rtol=1e-12, atol=1e-12)


def test_conv_ref_medium_matches_torch():
    rng = np.random.default_rng(5)
    x = rng.standard_normal((2, 32, 17, 23)).astype(np.float32)
    Wt = rng.standard_normal((24, 32, 3, 3)).astype(np.float32)
    Wh = PR.project(Wt, P.default8(), 0.3)["W_hat"]
    b = rng.standard_normal(24).astype(np.float32)
    for s in (1, 2):
        np.testing.assert_allclose(C.conv_ref(x, Wh, b, s, True), _torch_ref(x, Wh, b, s, True, False),
                                   rtol=1e-11, atol=1e-11)


def test_denominator_bounds_output():
    rng = np.random.default_rng(9)
    x = rng.standard_normal((1, 8, 9, 9)).astype(np.float32)
    Wh = PR.project(rng.standard_normal((8, 8, 3, 3)).astype(np.float32), P.default8(), 0.5)["W_hat"]
    b = rng.standard_normal(8).astype(np.float32)
    y = C.conv_ref(x, Wh, b, 1)
    d = C.denominator(x, Wh, b, 1)
    assert np.all(np.abs(y) <= d)
    assert C.max_norm_err(y, y, d) == 0.0


def test_lossless_when_conforming_and_keep_one():
    """keep = 1 and pattern-shaped weights: packing loses nothing and the pattern-sparse conv is
    the dense conv of the original weights (§3.2)."""
    rng = np.random.default_rng(12)
    lib = P.default8()
    pid = rng.integers(0, 8, size=(6, 5))
    W = np.zeros((6, 5, 9), np.float32)
    for co in range(6):
        for ci in range(5):
            for t in P.taps_of(lib[pid[co, ci]]):
                W[co, ci, t] = rng.uniform(0.5, 1.5) * rng.choice([-1, 1])
    W = W.reshape(6, 5, 3, 3)
    r = PR.project(W, lib, 1.0)
    np.testing.assert_array_equal(r["W_hat"], W)
    assert (r["pid"] == pid).all()
    x = rng.standard_normal((1, 5, 6, 6)).astype(np.float32)
    np.testing.assert_allclose(C.conv_ref(x, r["W_hat"], None), _torch_ref(x, W, None, 1, False, False),
                               rtol=1e-12, atol=1e-12)


def test_maxpool_matches_torch():
    rng = np.random.default_rng(1)
    for shape in [(2, 3, 8, 8), (1, 2, 7, 9)]:
        x = rng.standard_normal(shape).astype(np.float32)
        ref = Fnn.max_pool2d(torch.from_numpy(x), 2, 2).numpy()
        np.testing.assert_array_equal(C.maxpool2x2(x), ref)


# ------------------------------------------------------------------------------------- layout

def _tiny_fixture():
    W = np.zeros((3, 2, 9), np.float32)
    for line in golden_lines("layout_tiny.txt"):
        if line.startswith("k "):
            parts = line.split()
            co, ci = int(parts[1]), int(parts[2])
            for tv in parts[3:]:
                t, v = tv.split(":")
                W[co, ci, int(t)] = float(v)
    return W.reshape(3, 2, 3, 3), golden_kv("layout_tiny.txt")


def test_layout_hand_packed_fixture():
    W, g = _tiny_fixture()
    lib = P.default8()
    r = PR.project(W, lib, 0.5)
    assert r["pid"].reshape(-1).tolist() == [int(v) for v in g["pid"]]
    s = L.build(W, r["pid"], lib, 1, 1, r["beta"])
    assert s["perm"].tolist() == [int(v) for v in g["perm"]]
    assert s["desc"].tolist() == [int(v) for v in g["desc"]]
    assert s["kofs"].tolist() == [int(v) for v in g["kofs"]]
    assert s["vals"].reshape(-1).tolist() == [float(v) for v in g["vals"]]
    assert s["header"][:14].tolist() == [int(v) for v in g["header"]]


def _snake_fixture():
    g = golden_kv("layout_snake.txt")
    pa, pb = [int(v) for v in g["pa"]], [int(v) for v in g["pb"]]
    W = np.zeros((20, 2, 9), np.float32)
    for co in range(20):
        for ci, p in enumerate((pa[co], pb[co])):
            for k, t in enumerate(P.taps_of(P.default8()[p])):
                W[co, ci, t] = co + 0.25 * ci + 0.0625 * k + 1
    return W.reshape(20, 2, 3, 3), g


def _snake_expected(g):
    """desc words assembled by the specification's bit rule from the fixture's codes, and the
    vals rows: the (co, ci) kernels in (g, ci, slot) order, values by the fixture's rule."""
    desc, rows = [], []
    perm = [int(v) for v in g["perm"]]
    for grp in range(3):
        for ci in range(2):
            cnt, *codes = [int(v) for v in g[f"desc_g{grp}c{ci}"]]
            assert len(codes) == cnt
            desc.append(cnt | sum(c << (4 + 6 * j) for j, c in enumerate(codes)))
            for c in codes:
                co = perm[8 * grp + (c >> 3)]
                rows.append([co + 0.25 * ci + 0.0625 * k + 1 for k in range(4)])
    return desc, rows


def test_layout_snake_deal_hand_fixture():
    """Three groups: the sorted filters are dealt in snake order (round r fills slot r of every
    group, direction alternating), which the hand-dealt fixture pins exactly."""
    W, g = _snake_fixture()
    lib = P.default8()
    r = PR.project(W, lib, 1.0)
    assert r["beta"] == 40
    pa, pb = [int(v) for v in g["pa"]], [int(v) for v in g["pb"]]
    assert r["pid"].tolist() == [[a, b] for a, b in zip(pa, pb)]
    assert L.filter_order(r["pid"]) == [int(v) for v in g["order"]]
    s = L.build(W, r["pid"], lib, 1, 1, r["beta"])
    desc, rows = _snake_expected(g)
    assert s["perm"].tolist() == [int(v) for v in g["perm"]]
    assert s["desc"].tolist() == desc
    assert s["kofs"].tolist() == [int(v) for v in g["kofs"]]
    assert s["vals"].tolist() == rows


def test_packer_snake_deal_hand_fixture():
    """The C++ packer (pp_export) on the same hand-dealt fixture."""
    from paper_2003_06513_gb300 import api
    W, g = _snake_fixture()
    layer = api.pp_pack(W, None, 1.0)
    desc, rows = _snake_expected(g)
    assert layer.export("perm").tolist() == [int(v) for v in g["perm"]]
    assert layer.export("desc").tolist() == desc
    assert layer.export("kofs").tolist() == [int(v) for v in g["kofs"]]
    assert layer.export("vals").reshape(-1, 4).tolist() == rows


@pytest.mark.parametrize("cout,cin,keep,dw", [(3, 2, 0.5, False), (8, 8, 1.0, False), (13, 5, 0.3, False),
                                              (17, 1, 0.6, False), (20, 20, 1.0, True), (9, 9, 0.5, True),
                                              (64, 3, 1.0, False)])
def test_layout_decodes_to_projection(cout, cin, keep, dw):
    rng = np.random.default_rng(cout * 31 + cin)
    cin_g = 1 if dw else cin
    W = rng.standard_normal((cout, cin_g, 3, 3)).astype(np.float32)
    lib = P.default8()
    r = PR.project(W, lib, keep)
    s = L.build(W, r["pid"], lib, cout if dw else 1, 1, r["beta"])
    np.testing.assert_array_equal(L.decode(s, lib), r["W_hat"])
    np.testing.assert_array_equal(s["dense"].reshape(r["W_hat"].shape), r["W_hat"])
    # structure of the sections
    G = (cout + 7) // 8
    perm = s["perm"]
    real = perm[perm != L.PAD]
    assert sorted(real.tolist()) == list(range(cout)) and perm.size == 8 * G
    # filter kernel reorder: filters in kept-count order, dealt to groups in snake order, so
    # group totals differ by at most the largest single filter's count
    count = np.count_nonzero(r["pid"] >= 0, axis=1)
    order = L.filter_order(r["pid"])
    assert [count[c] for c in order] == sorted(count, reverse=True)
    totals = [sum(int(count[c]) for c in perm[8 * g:8 * g + 8] if c != L.PAD) for g in range(G)]
    if cout % G == 0 or cout < G:
        assert max(totals) - min(totals) <= int(count.max())
    assert (np.diff(s["kofs"].astype(np.int64)) >= 0).all() and s["kofs"][-1] == r["beta"]
    assert s["vals"].shape == (r["beta"], 4)
    assert s["image"].size % 256 == 0


def test_layout_image_sections_aligned():
    W, _ = _tiny_fixture()
    lib = P.default8()
    r = PR.project(W, lib, 0.5)
    s = L.build(W, r["pid"], lib, 1, 1, r["beta"])
    img = s["image"].tobytes()
    # perm (32 B) | desc (16 B) | kofs (12 B) | vals (48 B), each padded to 256 B
    assert len(img) == 4 * 256
    assert img[0:32] == s["perm"].tobytes() and img[32:256] == bytes(224)
    assert img[256:272] == s["desc"].tobytes()
    assert img[512:524] == s["kofs"].tobytes()
    assert img[768:816] == s["vals"].tobytes()
