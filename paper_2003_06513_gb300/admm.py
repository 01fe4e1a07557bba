"""Layer-wise ADMM pattern pruning on synthetic images (§4.3-4.5, Algorithm 1) and the masked
retraining hook released with the pruned model.

This is the training-side procedure that produces the pattern-pruned weights the inference
library runs; it is not on the inference path.  Per iteration k a batch of T synthetic images
(every pixel drawn uniformly from 0..255, independent of any user data) goes through the
pre-trained model and the current one; then, layer by layer:

* primal step (Eq. 4): one SGD step on W_n, b_n for
  mean (sigma(W_n X_{n-1} + b_n) - X'_n)^2 + rho/2 ||W_n - A_n + D_n||_F^2,
  X_{n-1} the current model's input to layer n, X'_n the pre-trained model's output of layer n;
* proximal step (Eq. 5-6): A_n = projection of W_n + D_n onto the constraint set -- computed by
  the library's own packer (pattern per kernel by largest retained norm, then connectivity);
* dual step: D_n += W_n - A_n.

rho starts at 1e-4 and grows 10x every 11 epochs of 10 iterations up to 1e-1; SGD with learning
rate 1e-3; T = 32 (§5.1).  Readings of this implementation: images are scaled to [0, 1] before
the first layer; the reconstruction term is the mean over its elements (the Frobenius norm
squared divided by the element count, so that the learning rate does not depend on the layer
size); the bias is trained with the weights; the model handed back is the projection of the
final weights, Pi(W^K), so that it satisfies the constraints exactly.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import List, Optional, Sequence

import numpy as np
import torch
import torch.nn.functional as F

from . import api


@dataclass
class ConvSpec:
    """One 3x3 convolution of a plain conv net: weights [Cout, Cin, 3, 3], bias [Cout], stride,
    ReLU after it, optional 2x2 max-pool after the ReLU, connectivity keep ratio."""
    weight: np.ndarray
    bias: np.ndarray
    stride: int = 1
    pool_after: bool = False
    keep: float = 1.0


@dataclass
class AdmmConfig:
    iterations: int = 220                 # K
    batch: int = 32                       # T
    image: Sequence[int] = (3, 32, 32)    # C, H, W of the synthetic images
    lr: float = 1e-3
    rho0: float = 1e-4
    rho_growth: float = 10.0
    epochs_per_growth: int = 11
    rho_max: float = 1e-1
    iters_per_epoch: int = 10
    patterns: Optional[Sequence[int]] = None   # None: the library's default 8-pattern set
    seed: int = 0


def rho_at(cfg: AdmmConfig, k: int) -> float:
    """Penalty of iteration k (0-based): rho0 x growth^(epoch // epochs_per_growth), capped."""
    epoch = k // cfg.iters_per_epoch
    return min(cfg.rho_max, cfg.rho0 * cfg.rho_growth ** (epoch // cfg.epochs_per_growth))


def project(weight: np.ndarray, patterns: Optional[Sequence[int]], keep: float, stride: int = 1) -> np.ndarray:
    """Euclidean projection onto the pattern and connectivity constraints, by the library's packer."""
    w = np.ascontiguousarray(weight, dtype=np.float32)
    return api.pp_pack(w, patterns, keep, 1, stride).export("dense").reshape(w.shape)


def synthetic_batch(gen: torch.Generator, cfg: AdmmConfig, device) -> torch.Tensor:
    """T images with every pixel uniform on 0..255 (no user data), scaled to [0, 1]."""
    c, h, w = cfg.image
    x = torch.randint(0, 256, (cfg.batch, c, h, w), generator=gen, dtype=torch.int64)
    return (x.to(torch.float32) / 255.0).to(device)


def _layer(x: torch.Tensor, w: torch.Tensor, b: torch.Tensor, spec: ConvSpec) -> torch.Tensor:
    y = F.relu(F.conv2d(x, w, b, stride=spec.stride, padding=1))
    return F.max_pool2d(y, 2) if spec.pool_after else y


def forward(layers: Sequence[ConvSpec], weights: Sequence[torch.Tensor], biases: Sequence[torch.Tensor],
            x: torch.Tensor) -> List[torch.Tensor]:
    """Outputs of every layer of the conv net (dense convolutions)."""
    outs = []
    for spec, w, b in zip(layers, weights, biases):
        x = _layer(x, w, b, spec)
        outs.append(x)
    return outs


@dataclass
class AdmmResult:
    weights: List[np.ndarray]             # Pi(W^K) per layer: satisfies the constraints exactly
    biases: List[np.ndarray]
    history: List[List[float]] = field(default_factory=list)   # per iteration: primal loss per layer


def admm_prune(layers: Sequence[ConvSpec], cfg: AdmmConfig = AdmmConfig(), device="cpu") -> AdmmResult:
    """Algorithm 1: layer-wise ADMM pattern + connectivity pruning on synthetic images."""
    device = torch.device(device)
    gen = torch.Generator().manual_seed(cfg.seed)
    w0 = [torch.from_numpy(np.asarray(s.weight, np.float32)).to(device) for s in layers]
    b0 = [torch.from_numpy(np.asarray(s.bias, np.float32)).to(device) for s in layers]
    W = [w.clone().requires_grad_(True) for w in w0]
    B = [b.clone().requires_grad_(True) for b in b0]
    A = [w.detach().clone() for w in w0]                       # A^0 = W^0
    D = [torch.zeros_like(w) for w in w0]                      # D^0 = 0
    history = []
    for k in range(cfg.iterations):
        rho = rho_at(cfg, k)
        x = synthetic_batch(gen, cfg, device)
        with torch.no_grad():
            targets = forward(layers, w0, b0, x)               # the pre-trained model's outputs
        losses = []
        xin = x
        for n, spec in enumerate(layers):
            # primal problem (Eq. 4): one SGD step on W_n, b_n
            y = _layer(xin, W[n], B[n], spec)
            rec = torch.mean((y - targets[n]) ** 2)
            pen = 0.5 * rho * torch.sum((W[n] - A[n] + D[n]) ** 2)
            loss = rec + pen
            gw, gb = torch.autograd.grad(loss, [W[n], B[n]])
            with torch.no_grad():
                W[n] -= cfg.lr * gw
                B[n] -= cfg.lr * gb
                # proximal problem (Eq. 5-6): projection of W + D onto the constraint set
                A[n] = torch.from_numpy(project((W[n] + D[n]).cpu().numpy(), cfg.patterns, spec.keep,
                                                spec.stride)).to(device)
                D[n] += W[n] - A[n]                            # dual update
                xin = _layer(xin, W[n], B[n], spec)            # the current model's next input
            losses.append(float(rec.detach()))
        history.append(losses)
    final_w = [project(w.detach().cpu().numpy(), cfg.patterns, s.keep, s.stride) for w, s in zip(W, layers)]
    final_b = [b.detach().cpu().numpy().copy() for b in B]
    return AdmmResult(final_w, final_b, history)


def masked_retraining_hook(weights: Sequence[torch.Tensor]) -> list:
    """The retraining function sent back with the pruned model: gradient hooks that zero the
    gradient wherever a weight is zero now (pruned taps and pruned kernels), so that retraining
    on the user's own data updates only the kept weights and the model keeps its patterns and
    connectivity.  Returns the hook handles (``handle.remove()`` ends masked training)."""
    handles = []
    for w in weights:
        mask = (w.detach() != 0).to(w.dtype)
        handles.append(w.register_hook(lambda g, m=mask: g * m))
    return handles
