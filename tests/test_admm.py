"""Layer-wise ADMM pattern pruning (§4.3-4.5, Algorithm 1) and the masked retraining hook.

Only the mechanism can be checked without the paper's trained models and datasets: the schedule,
that the released weights satisfy the pattern and connectivity constraints exactly, that a model
already inside the constraint set is left untouched, that ADMM reconstructs the pre-trained
layer outputs better than projecting the weights once, and that masked retraining keeps the
pruned structure.  CPU unless marked gpu.
"""
import numpy as np
import pytest
import torch

from oracle import patterns as OP
from oracle import project as OPR
from paper_2003_06513_gb300 import admm as AD


def _net(seed=0):
    rng = np.random.default_rng(seed)
    return [AD.ConvSpec((rng.standard_normal((8, 3, 3, 3)) * 0.3).astype(np.float32),
                        (rng.standard_normal(8) * 0.1).astype(np.float32), keep=1.0),
            AD.ConvSpec((rng.standard_normal((8, 8, 3, 3)) * 0.2).astype(np.float32),
                        (rng.standard_normal(8) * 0.1).astype(np.float32), keep=0.5, pool_after=True)]


def _fast_cfg(**kw):
    base = dict(iterations=150, batch=8, image=(3, 12, 12), lr=0.05, rho0=1e-2, rho_growth=3.0,
                epochs_per_growth=3, rho_max=1.0)
    base.update(kw)
    return AD.AdmmConfig(**base)


def _recon(layers, ws, bs, x):
    tw = [torch.from_numpy(np.asarray(l.weight, np.float32)) for l in layers]
    tb = [torch.from_numpy(np.asarray(l.bias, np.float32)) for l in layers]
    ref = AD.forward(layers, tw, tb, x)[-1]
    out = AD.forward(layers, [torch.from_numpy(w) for w in ws], [torch.from_numpy(b) for b in bs], x)[-1]
    return float(torch.mean((out - ref) ** 2))


def test_rho_schedule_follows_section_5_1():
    cfg = AD.AdmmConfig()
    assert AD.rho_at(cfg, 0) == pytest.approx(1e-4)
    assert AD.rho_at(cfg, 109) == pytest.approx(1e-4)      # epoch 10
    assert AD.rho_at(cfg, 110) == pytest.approx(1e-3)      # epoch 11: x10
    assert AD.rho_at(cfg, 220) == pytest.approx(1e-2)
    assert AD.rho_at(cfg, 330) == pytest.approx(1e-1)
    assert AD.rho_at(cfg, 10_000) == pytest.approx(1e-1)   # capped


def test_projection_is_the_oracles():
    w = _net(3)[1].weight
    np.testing.assert_array_equal(AD.project(w, None, 0.5), OPR.project(w, OP.default8(), 0.5)["W_hat"])


def test_synthetic_images_are_uniform_pixels():
    cfg = AD.AdmmConfig(batch=64, image=(3, 16, 16))
    x = AD.synthetic_batch(torch.Generator().manual_seed(1), cfg, "cpu")
    v = torch.round(x * 255)
    assert torch.equal(v, x * 255) or torch.allclose(v, x * 255, atol=1e-4)
    assert int(v.min()) == 0 and int(v.max()) == 255
    assert abs(float(v.mean()) - 127.5) < 2.0


def test_released_weights_satisfy_the_constraints():
    layers = _net(1)
    res = AD.admm_prune(layers, _fast_cfg(iterations=30))
    masks = OP.default8()
    for spec, w in zip(layers, res.weights):
        k = w.reshape(-1, 9)
        nz = k != 0
        kept = nz.any(axis=1)
        beta = OPR.n_keep(spec.keep, k.shape[0])
        assert kept.sum() <= beta
        for row in nz[kept]:
            m = sum(1 << t for t in np.flatnonzero(row))
            assert any(m & ~mask == 0 for mask in masks), "a kept kernel outside every pattern"


def test_model_inside_the_constraints_is_left_alone():
    """W^0 in C: the outputs already match, A^0 = W^0 and D = 0, so no step moves W."""
    layers = _net(2)
    for spec in layers:
        spec.weight = AD.project(spec.weight, None, spec.keep)
    res = AD.admm_prune(layers, _fast_cfg(iterations=12))
    for spec, w, b in zip(layers, res.weights, res.biases):
        np.testing.assert_array_equal(w, spec.weight)
        np.testing.assert_array_equal(b, spec.bias)


def test_admm_reconstructs_better_than_one_shot_projection():
    layers = _net(0)
    res = AD.admm_prune(layers, _fast_cfg())
    x = AD.synthetic_batch(torch.Generator().manual_seed(999), _fast_cfg(), "cpu")
    one_shot = [AD.project(l.weight, None, l.keep) for l in layers]
    e_one = _recon(layers, one_shot, [l.bias for l in layers], x)
    e_admm = _recon(layers, res.weights, res.biases, x)
    assert e_admm < 0.7 * e_one, (e_admm, e_one)


def test_masked_retraining_keeps_the_pruned_structure():
    w = torch.from_numpy(AD.project(_net(4)[1].weight, None, 0.5)).requires_grad_(True)
    zeros = (w.detach() == 0)
    handles = AD.masked_retraining_hook([w])
    opt = torch.optim.SGD([w], lr=0.1)
    x = torch.randn(2, 8, 6, 6)
    for _ in range(5):
        opt.zero_grad()
        torch.nn.functional.conv2d(x, w, padding=1).pow(2).mean().backward()
        opt.step()
    assert torch.all(w.detach()[zeros] == 0)
    assert not torch.equal(w.detach()[~zeros], torch.from_numpy(AD.project(_net(4)[1].weight, None, 0.5))[~zeros])
    for h in handles:
        h.remove()


@pytest.mark.gpu
def test_admm_runs_on_the_gpu():
    layers = _net(5)
    res = AD.admm_prune(layers, _fast_cfg(iterations=20), device="cuda")
    assert all(np.isfinite(w).all() for w in res.weights) and len(res.history) == 20
