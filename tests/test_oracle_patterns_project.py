"""Pins of the oracle's pattern library, projection and connectivity pruning (CPU only).

Each test checks the oracle against something other than itself: hand-drawn / hand-computed
fixtures, brute-force enumeration of the Euclidean projection (§4.3, Eq. 6 with C_n and C'_n of
§4.4), and the paper's counting invariants (4 nonzeros per kernel, at most beta kernels, the
2.25x pattern-only compression of §5.2).
"""
import itertools
import math

import numpy as np
import pytest

from conftest import golden_kv, golden_lines
from oracle import patterns as P
from oracle import project as PR


def _fixture_patterns():
    lines = golden_lines("patterns8.txt")
    out = []
    i = 0
    while i < len(lines):
        head = lines[i].split()
        assert head[0] == f"p{len(out)}"
        mask = int(head[1].split("=")[1])
        rows = lines[i + 1:i + 4]
        drawn = 0
        for r, row in enumerate(rows):
            for c, ch in enumerate(row.strip()):
                if ch == "x":
                    drawn |= 1 << (3 * r + c)
        assert drawn == mask, f"fixture drawing and mask disagree for {head[0]}"
        out.append(mask)
        i += 4
    return out


def test_default_library_matches_hand_drawing():
    assert P.default8() == _fixture_patterns()


def test_default_library_properties():
    lib = P.default8()
    P.validate(lib)
    for m in lib:
        assert bin(m).count("1") == 4
        assert (m >> P.CENTRE) & 1, "centre tap always kept (§4.2)"
    assert len(set(lib)) == 8


@pytest.mark.parametrize("bad", [[], [0x17] * 2, [0x1F], [0x7], list(range(1, 10)), [512 | 7]])
def test_validate_rejects(bad):
    with pytest.raises(ValueError):
        P.validate(bad)


def test_hand_projection():
    g = golden_kv("projection_hand.txt")
    w = np.array([float(v) for v in g["w"]], dtype=np.float32).reshape(1, 1, 3, 3)
    r = PR.project(w, P.default8(), 1.0)
    np.testing.assert_allclose(r["s"][0, 0], [float(v) for v in g["scores"]], rtol=1e-6)
    assert int(r["pid"][0, 0]) == int(g["best"][0])
    np.testing.assert_array_equal(r["W_hat"].reshape(9),
                                  np.array([float(v) for v in g["projected"]], dtype=np.float32))
    resid = float(np.sum((w.astype(np.float64) - r["W_hat"].astype(np.float64)) ** 2))
    assert abs(resid - float(g["residual"][0])) < 1e-5


@pytest.mark.parametrize("p", range(8))
def test_conforming_kernel_is_fixed_point(p):
    rng = np.random.default_rng(p)
    mask = P.default8()[p]
    w = np.zeros(9, dtype=np.float32)
    for t in P.taps_of(mask):
        w[t] = np.float32(rng.uniform(0.5, 2.0) * rng.choice([-1, 1]))
    r = PR.project(w.reshape(1, 1, 3, 3), P.default8(), 1.0)
    # another pattern can only tie if it covers the same energy, impossible with 4 nonzero taps
    assert int(r["pid"][0, 0]) == p
    np.testing.assert_array_equal(r["W_hat"].reshape(9), w)


def test_ties_go_to_lowest_index():
    lib = P.default8()
    zero = np.zeros((1, 1, 3, 3), np.float32)
    assert int(PR.project(zero, lib, 1.0)["pid"][0, 0]) == 0
    centre = zero.copy()
    centre[0, 0, 1, 1] = 5
    assert int(PR.project(centre, lib, 1.0)["pid"][0, 0]) == 0
    edges = zero.copy()
    for (dy, dx) in P.EDGES:
        edges[0, 0, 1 + dy, 1 + dx] = 1
    edges[0, 0, 1, 1] = 1                     # p0..p3 all retain 4: lowest is p0
    assert int(PR.project(edges, lib, 1.0)["pid"][0, 0]) == 0
    # p5 {0,3,4,6} and p6 {2,4,5,8} tie above every other pattern -> p5
    k = np.zeros(9, np.float32)
    k[[0, 3, 6, 2, 5, 8]] = 1                 # both side columns: p5 = p6 = 4, others <= 3
    k[4] = 1
    r = PR.project(k.reshape(1, 1, 3, 3), lib, 1.0)
    s = r["s"][0, 0]
    assert s[5] == s[6] and s[5] > max(s[[0, 1, 2, 3, 4, 7]])
    assert int(r["pid"][0, 0]) == 5


def test_scores_are_fixed_order_float64():
    rng = np.random.default_rng(7)
    W = rng.standard_normal((3, 4, 3, 3)).astype(np.float32)
    s = PR.scores(W, P.default8())
    for co in range(3):
        for ci in range(4):
            for p, m in enumerate(P.default8()):
                acc = 0.0
                for t in P.taps_of(m):
                    v = float(W[co, ci, t // 3, t % 3])
                    acc = acc + v * v
                assert s[co, ci, p] == acc      # bit-identical to the scalar left-to-right sum


def _brute_force(W, masks, beta):
    """min ||W - A||_F^2 over A with each kernel inside one pattern or zero, <= beta nonzero
    kernels; enumerates every assignment and measures the distance directly."""
    cout, cin = W.shape[:2]
    K = cout * cin
    w = W.reshape(K, 9).astype(np.float64)
    options = list(range(len(masks))) + [-1]
    best, arg, count = math.inf, None, 0
    for assign in itertools.product(options, repeat=K):
        if sum(a >= 0 for a in assign) > beta:
            continue
        A = np.zeros_like(w)
        for k, a in enumerate(assign):
            if a >= 0:
                for t in P.taps_of(masks[a]):
                    A[k, t] = w[k, t]
        d = float(np.sum((w - A) ** 2))
        if d < best - 1e-12:
            best, arg, count = d, assign, 1
        elif abs(d - best) <= 1e-12:
            count += 1
    return best, arg, count


@pytest.mark.parametrize("shape,keep,seed", [((1, 1), 1.0, 0), ((1, 2), 0.5, 1), ((2, 1), 0.5, 2),
                                             ((2, 2), 0.5, 3), ((2, 2), 0.25, 4), ((1, 3), 0.7, 5),
                                             ((2, 2), 1.0, 6), ((4, 1), 0.5, 7)])
def test_projection_is_euclidean_by_brute_force(shape, keep, seed):
    lib = P.default8()
    rng = np.random.default_rng(seed)
    W = rng.standard_normal(shape + (3, 3)).astype(np.float32)
    r = PR.project(W, lib, keep)
    d = float(np.sum((W.astype(np.float64) - r["W_hat"].astype(np.float64)) ** 2))
    best, arg, count = _brute_force(W, lib, r["beta"])
    assert abs(d - best) <= 1e-9 * max(1.0, best)
    if count == 1:
        assert tuple(int(p) for p in r["pid"].reshape(-1)) == arg


def test_brute_force_catches_a_wrong_rule():
    """The brute-force pin is strong enough to reject plausible mistakes: keeping the smallest
    retained energy, or pruning by the original (unprojected) kernel norm."""
    lib = P.default8()
    rng = np.random.default_rng(11)
    W = rng.standard_normal((2, 2, 3, 3)).astype(np.float32)
    s = PR.scores(W, lib)
    wrong = np.argmin(s, axis=-1)
    A = np.zeros((4, 9))
    w = W.reshape(4, 9).astype(np.float64)
    for k, p in enumerate(wrong.reshape(-1)):
        for t in P.taps_of(lib[p]):
            A[k, t] = w[k, t]
    best, _, _ = _brute_force(W, lib, 4)
    assert float(np.sum((w - A) ** 2)) > best + 1e-6
    # connectivity ranked by the unprojected kernel norm instead of the retained energy
    for seed in range(100):
        W = np.random.default_rng(seed).standard_normal((2, 2, 3, 3)).astype(np.float32)
        r = PR.project(W, lib, 0.5)
        full = np.sum(W.reshape(4, 9).astype(np.float64) ** 2, axis=1)
        wrong_kept = set(np.argsort(-full, kind="stable")[:r["beta"]].tolist())
        if wrong_kept != set(np.flatnonzero(r["pid"].reshape(-1) >= 0).tolist()):
            break
    w = W.reshape(4, 9).astype(np.float64)
    A = np.zeros((4, 9))
    for k in wrong_kept:
        for t in P.taps_of(lib[int(r["best"].reshape(-1)[k])]):
            A[k, t] = w[k, t]
    best, _, _ = _brute_force(W, lib, r["beta"])
    assert float(np.sum((w - A) ** 2)) > best + 1e-9


def test_invariants_at_scale():
    lib = P.default8()
    rng = np.random.default_rng(3)
    W = rng.standard_normal((64, 48, 3, 3)).astype(np.float32)
    for keep in (1.0, 0.5, 0.3, 0.01):
        r = PR.project(W, lib, keep)
        pid, Wh, beta = r["pid"], r["W_hat"], r["beta"]
        assert beta == PR.n_keep(keep, 64 * 48)
        assert int(np.count_nonzero(pid >= 0)) == beta
        nz = np.count_nonzero(Wh.reshape(64, 48, 9), axis=-1)
        assert np.all(nz[pid >= 0] == 4) and np.all(nz[pid < 0] == 0)
        assert int(np.count_nonzero(Wh)) == 4 * beta
        for co, ci in zip(*np.nonzero(pid >= 0)):
            support = sum(1 << t for t in range(9) if Wh[co, ci].reshape(9)[t] != 0)
            assert support == lib[pid[co, ci]]
        # every pruned kernel retains no more energy than any kept one (connectivity, §4.4)
        ret = np.take_along_axis(r["s"], r["best"][..., None], -1)[..., 0]
        if beta < 64 * 48:
            assert ret[pid < 0].max() <= ret[pid >= 0].min()
    r = PR.project(W, lib, 1.0)
    assert 9 * W[..., 0, 0].size / np.count_nonzero(r["W_hat"]) == 2.25   # §5.2


def test_compression_rates_fixture():
    for line in golden_lines("compression_rates.txt"):
        rate, keep, beta = line.split()
        b = PR.n_keep(float(keep), 4096)
        assert b == int(beta)
        assert 9 * 4096 / (4 * b) == float(rate)


def test_n_keep_rounding_and_clamp():
    assert PR.n_keep(0.3, 4096) == 1229          # 1228.8 rounds half up
    assert PR.n_keep(0.5, 3) == 2                # 1.5 -> 2
    assert PR.n_keep(1e-9, 10) == 1              # at least one kernel
    for bad in (0.0, -0.1, 1.5, float("nan")):
        with pytest.raises(ValueError):
            PR.n_keep(bad, 10)


def test_rejects_non_finite():
    W = np.zeros((2, 2, 3, 3), np.float32)
    W[1, 0, 2, 2] = np.nan
    with pytest.raises(ValueError):
        PR.project(W, P.default8(), 1.0)
    W[1, 0, 2, 2] = np.inf
    with pytest.raises(ValueError):
        PR.project(W, P.default8(), 1.0)


# --------------------------------------------------------------------------- library design (§4.2)

def _design_fixture():
    rows = [[float(v) for v in line.split()[1:]] for line in golden_lines("pattern_design_hand.txt")
            if line.startswith("k ")]
    return np.array(rows, dtype=np.float32), golden_kv("pattern_design_hand.txt")


def test_design_library_hand_fixture():
    K, g = _design_fixture()
    assert P.design_library(K, 2) == [int(v) for v in g["lib_m2"]]
    assert P.design_library(K, 8) == [int(v) for v in g["lib_m8"]]


def test_design_library_recovers_planted_patterns():
    """Kernels built with three dominant non-central taps propose exactly those taps + centre;
    the library lists the planted masks by how often they were planted."""
    rng = np.random.default_rng(4)
    planted = {}
    rows = []
    for i in range(300):
        taps3 = sorted(rng.choice([0, 1, 2, 3, 5, 6, 7, 8], size=3, replace=False).tolist())
        w = rng.uniform(-0.1, 0.1, size=9)
        w[4] = rng.uniform(-20, 20)                    # the centre may be the largest or not
        for t in taps3:
            w[t] = rng.choice([-1, 1]) * rng.uniform(1.0, 2.0)
        mk = P.mask_of(taps3 + [4])
        planted[mk] = planted.get(mk, 0) + 1
        rows.append(w)
    lib = P.design_library(np.array(rows, np.float32), 8)
    expected = sorted(planted, key=lambda mk: (-planted[mk], mk))[:8]
    assert lib == expected
    assert all(bin(mk).count("1") == 4 and (mk >> 4) & 1 for mk in lib)
