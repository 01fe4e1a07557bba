"""The float64 ADMM oracle (oracle/admm.py: §4.3-4.5, Eq. 4-7, Algorithm 1) and the library's
training-side module (paper_2003_06513_gb300/admm.py) against it.

The oracle is pinned first: its hand-written gradient against central finite differences, and a
model that already satisfies the constraints and reproduces the targets staying exactly where it
is.  Then the module's first iterations are compared with the oracle's, and mistakes planted in
copies of the oracle's iteration (the dual update's sign, the rho/2 factor, projecting W instead
of W + D) are shown to move the result further than the comparison's tolerance."""
import numpy as np
import pytest
import torch

from oracle import admm as OA
from oracle import patterns as OP
from oracle import project as OPR
from paper_2003_06513_gb300 import admm as AD


def _net(seed=0):
    rng = np.random.default_rng(seed)
    return [AD.ConvSpec((rng.standard_normal((8, 3, 3, 3)) * 0.3).astype(np.float32),
                        (rng.standard_normal(8) * 0.1).astype(np.float32), keep=1.0),
            AD.ConvSpec((rng.standard_normal((8, 8, 3, 3)) * 0.2).astype(np.float32),
                        (rng.standard_normal(8) * 0.1).astype(np.float32), keep=0.5, pool_after=True)]


def _specs(layers):
    return [(l.stride, l.pool_after, l.keep) for l in layers]


@pytest.mark.parametrize("stride,pool", [(1, False), (1, True), (2, False)])
def test_oracle_gradient_matches_finite_differences(stride, pool):
    rng = np.random.default_rng(11 + stride + 2 * pool)
    x = rng.standard_normal((2, 3, 6, 7))
    W = rng.standard_normal((4, 3, 3, 3)) * 0.4
    b = rng.standard_normal(4) * 0.1
    Ho, Wo = (6 - 1) // stride + 1, (7 - 1) // stride + 1
    shape = (2, 4, Ho // 2, Wo // 2) if pool else (2, 4, Ho, Wo)
    target = rng.standard_normal(shape) * 0.5
    f, gW, gb = OA.grad(x, W, b, target, stride, pool)
    h = 1e-6
    for idx in [(0, 0, 0, 0), (1, 2, 1, 1), (3, 1, 2, 0), (2, 0, 1, 2)]:
        Wp, Wm = W.copy(), W.copy()
        Wp[idx] += h
        Wm[idx] -= h
        num = (OA.grad(x, Wp, b, target, stride, pool)[0] - OA.grad(x, Wm, b, target, stride, pool)[0]) / (2 * h)
        assert gW[idx] == pytest.approx(num, rel=1e-5, abs=1e-9)
    for co in range(4):
        bp, bm = b.copy(), b.copy()
        bp[co] += h
        bm[co] -= h
        num = (OA.grad(x, W, bp, target, stride, pool)[0] - OA.grad(x, W, bm, target, stride, pool)[0]) / (2 * h)
        assert gb[co] == pytest.approx(num, rel=1e-5, abs=1e-9)


def test_oracle_keeps_a_conforming_model():
    """Weights already inside the constraint sets and targets equal to the model's own outputs:
    zero gradient, so W, b stay, A = W and D stays 0 over several iterations."""
    layers = _net(4)
    masks = OP.default8()
    W0 = [OPR.project(l.weight, masks, l.keep)["W_hat"] for l in layers]
    b0 = [l.bias for l in layers]
    rng = np.random.default_rng(0)
    images = [rng.integers(0, 256, (3, 3, 8, 8)) / 255.0 for _ in range(3)]
    final, bs, hist, As, Ds = OA.run(W0, b0, images, _specs(layers), [1e-2] * 3, 0.05, masks)
    for n in range(2):
        np.testing.assert_array_equal(final[n], W0[n])
        np.testing.assert_array_equal(As[n], W0[n])
        np.testing.assert_array_equal(Ds[n], 0)
        np.testing.assert_array_equal(bs[n], b0[n])
    assert all(v == 0 for row in hist for v in row)


def _module_run(layers, K, rho, lr, seed=3):
    cfg = AD.AdmmConfig(iterations=K, batch=3, image=(3, 10, 10), lr=lr, rho0=rho, rho_growth=1.0, rho_max=rho,
                        seed=seed)
    res = AD.admm_prune(layers, cfg)
    gen = torch.Generator().manual_seed(seed)                # the same synthetic batches
    images = [AD.synthetic_batch(gen, cfg, "cpu").numpy().astype(np.float64) for _ in range(K)]
    return res, images


def _close(res, final, bs, hist):
    for n in range(len(final)):
        np.testing.assert_allclose(res.weights[n], final[n], rtol=2e-4, atol=1e-6)
        np.testing.assert_allclose(res.biases[n], bs[n], rtol=2e-4, atol=1e-6)
    np.testing.assert_allclose(np.array(res.history), np.array(hist), rtol=2e-4, atol=1e-9)


K, RHO, LR = 3, 0.3, 0.05


def test_module_iterations_match_oracle():
    layers = _net(0)
    res, images = _module_run(layers, K, RHO, LR)
    final, bs, hist, _, _ = OA.run([l.weight for l in layers], [l.bias for l in layers], images,
                                   _specs(layers), [RHO] * K, LR, OP.default8())
    _close(res, final, bs, hist)


def _planted_iteration(mistake):
    """A copy of the oracle's iteration with one mistake planted."""
    def it(Ws, bs, As, Ds, W0, b0, x0, specs, rho, lr, masks):
        targets, t = [], np.asarray(x0, np.float64)
        for Wp, bp, (s, pool, _) in zip(W0, b0, specs):
            t = OA.layer_forward(t, Wp, bp, s, pool)
            targets.append(t)
        xin = np.asarray(x0, np.float64)
        losses = []
        for n, (s, pool, keep) in enumerate(specs):
            f, gW, gb = OA.grad(xin, Ws[n], bs[n], targets[n], s, pool)
            scale = 2 * rho if mistake == "rho_not_halved" else rho
            gW = gW + scale * (Ws[n] - As[n] + Ds[n])
            Ws[n] = Ws[n] - lr * gW
            bs[n] = bs[n] - lr * gb
            V = Ws[n] if mistake == "project_w" else Ws[n] + Ds[n]
            As[n] = OPR.project(V.astype(np.float32), masks, keep)["W_hat"].astype(np.float64)
            Ds[n] = Ds[n] - (Ws[n] - As[n]) if mistake == "dual_sign" else Ds[n] + Ws[n] - As[n]
            xin = OA.layer_forward(xin, Ws[n], bs[n], s, pool)
            losses.append(f)
        return losses
    return it


@pytest.mark.parametrize("mistake", ["dual_sign", "rho_not_halved", "project_w"])
def test_planted_mistakes_fail_the_comparison(monkeypatch, mistake):
    layers = _net(0)
    res, images = _module_run(layers, K, RHO, LR)
    monkeypatch.setattr(OA, "iteration", _planted_iteration(mistake))
    final, bs, hist, _, _ = OA.run([l.weight for l in layers], [l.bias for l in layers], images,
                                   _specs(layers), [RHO] * K, LR, OP.default8())
    with pytest.raises(AssertionError):
        _close(res, final, bs, hist)
