"""Layer-wise ADMM pruning (§4.3-4.5, Eq. 3-7, Algorithm 1) in plain float64 numpy.

TEST INFRASTRUCTURE ONLY (see the package docstring).  It pins the training-side module of the
library, which runs the same algorithm in float32 torch with autograd.

Algorithm 1 for a plain conv net x -> sigma(W_1 x + b_1) -> ... with sigma = ReLU, optionally a
2x2 max-pool after it, and constraint sets C_n (one pattern per kernel) and C'_n (at most beta_n
kernels):

    A_n^0 = W_n^0,  D_n^0 = 0
    for k = 1 .. K:
        a batch of T synthetic images X_0 (passed in: the images are the method's random draw)
        for n = 1 .. N:
            X'_n   = output of layer n of the pre-trained model
            X_{n-1} = input of layer n in the current model (layers 1 .. n-1 already updated)
            W_n^k, b_n^k: problem (Eq. 4), min f(W, b) + rho/2 ||W - A_n^{k-1} + D_n^{k-1}||_F^2
            A_n^k = projection of W_n^k + D_n^k-1 onto C_n and C'_n          (Eq. 5-6)
            D_n^k = D_n^{k-1} + W_n^k - A_n^k                                 (dual update)

Readings (the paper leaves them open; the library makes the same ones):
* "standard solvers" for Eq. 4: one gradient step of size lr per iteration and layer, on W and b;
* f(W, b) is the mean of (sigma(W X + b) - X')^2 over its elements (the squared Frobenius norm
  divided by the element count), so the step size does not depend on the layer size;
* the projection (oracle.project) takes float32 weights like the library's packer: W + D is
  rounded to float32 before it is projected, everything else stays float64;
* the max-pool passes its gradient to the first position (row-major) of each window that holds
  the maximum.

The gradient is written out by hand (no autodiff): with z = W * X + b (the 3x3 convolution,
pad 1, oracle.conv), r = max(z, 0), y = pool(r) or r, g_y = 2 (y - X') / |y|,
g_z = (g_y routed back through the pool) * [z > 0], and
    dF/dW[co, ci, ky, kx] = sum_{n, oy, ox} g_z[n, co, oy, ox] X_pad[n, ci, s oy + ky, s ox + kx]
                            + rho (W - A + D)[co, ci, ky, kx]
    dF/db[co] = sum_{n, oy, ox} g_z[n, co, oy, ox].
"""
from __future__ import annotations

from typing import List, Sequence, Tuple

import numpy as np

from . import conv as C
from . import project as PR


def layer_forward(x, W, b, stride: int, pool: bool):
    """sigma(W x + b), then the 2x2 max-pool where the layer has one (float64)."""
    y = C.conv_ref(x, W, b, stride, relu=True)
    return C.maxpool2x2(y) if pool else y


def _pool_backward(g, r):
    """Gradient of the 2x2/2 max-pool (floor mode) w.r.t. its input r: each window's gradient
    goes to the first position in row-major order that holds the window's maximum."""
    N, Cc, H, W = r.shape
    out = np.zeros_like(r)
    for i in range(H // 2):
        for j in range(W // 2):
            win = r[:, :, 2 * i:2 * i + 2, 2 * j:2 * j + 2].reshape(N, Cc, 4)
            first = np.argmax(win, axis=2)           # argmax returns the first maximum
            for q in range(4):
                a, c = divmod(q, 2)
                out[:, :, 2 * i + a, 2 * j + c] += np.where(first == q, g[:, :, i, j], 0.0)
    return out


def grad(x, W, b, target, stride: int, pool: bool):
    """(f, dF/dW, dF/db) of the reconstruction term f = mean((sigma(W x + b) - target)^2)."""
    x = np.asarray(x, np.float64)
    W = np.asarray(W, np.float64)
    z = C.conv_ref(x, W, b, stride, relu=False)
    r = np.maximum(z, 0.0)
    y = C.maxpool2x2(r) if pool else r
    f = float(np.mean((y - target) ** 2))
    gy = 2.0 * (y - target) / y.size
    gr = _pool_backward(gy, r) if pool else gy
    gz = gr * (z > 0)
    N, Cin, H, Wd = x.shape
    Ho, Wo = z.shape[2:]
    xp = np.zeros((N, Cin, H + 2, Wd + 2))
    xp[:, :, 1:H + 1, 1:Wd + 1] = x
    gW = np.zeros_like(W)
    for ky in range(3):
        for kx in range(3):
            xs = xp[:, :, ky:ky + stride * (Ho - 1) + 1:stride, kx:kx + stride * (Wo - 1) + 1:stride]
            gW[:, :, ky, kx] = np.einsum("nkij,ncij->kc", gz, xs)
    gb = gz.sum(axis=(0, 2, 3))
    return f, gW, gb


def iteration(Ws: List[np.ndarray], bs: List[np.ndarray], As: List[np.ndarray], Ds: List[np.ndarray],
              W0: Sequence[np.ndarray], b0: Sequence[np.ndarray], x0, specs, rho: float, lr: float,
              masks: Sequence[int]) -> List[float]:
    """One iteration k of Algorithm 1 over all layers, in place.  specs: (stride, pool, keep) per
    layer.  Returns the reconstruction term f of every layer (before its step)."""
    targets, t = [], np.asarray(x0, np.float64)
    for Wp, bp, (s, pool, _) in zip(W0, b0, specs):       # the pre-trained model's outputs
        t = layer_forward(t, Wp, bp, s, pool)
        targets.append(t)
    xin = np.asarray(x0, np.float64)
    losses = []
    for n, (s, pool, keep) in enumerate(specs):
        f, gW, gb = grad(xin, Ws[n], bs[n], targets[n], s, pool)
        gW = gW + rho * (Ws[n] - As[n] + Ds[n])           # gradient of rho/2 ||W - A + D||_F^2
        Ws[n] = Ws[n] - lr * gW
        bs[n] = bs[n] - lr * gb
        V = (Ws[n] + Ds[n]).astype(np.float32)            # projected as float32 (the packer's input)
        As[n] = PR.project(V, masks, keep)["W_hat"].astype(np.float64)
        Ds[n] = Ds[n] + Ws[n] - As[n]
        xin = layer_forward(xin, Ws[n], bs[n], s, pool)   # the current model's next input
        losses.append(f)
    return losses


def run(W0, b0, images: Sequence[np.ndarray], specs, rhos: Sequence[float], lr: float,
        masks: Sequence[int]) -> Tuple[List[np.ndarray], List[np.ndarray], List[List[float]],
                                        List[np.ndarray], List[np.ndarray]]:
    """Algorithm 1 for len(images) iterations; returns (Pi(W^K) per layer, b^K, losses, A^K, D^K).
    Pi(W^K) is the projection of the final weights (rounded to float32 like the packer's input)."""
    Ws = [np.asarray(w, np.float64).copy() for w in W0]
    bs = [np.asarray(b, np.float64).copy() for b in b0]
    As = [w.copy() for w in Ws]
    Ds = [np.zeros_like(w) for w in Ws]
    hist = []
    for x, rho in zip(images, rhos):
        hist.append(iteration(Ws, bs, As, Ds, W0, b0, x, specs, rho, lr, masks))
    final = [PR.project(w.astype(np.float32), masks, keep)["W_hat"] for w, (_, _, keep) in zip(Ws, specs)]
    return final, bs, hist, As, Ds
