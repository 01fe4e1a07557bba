"""Layer forward X_n = sigma(W_n X_{n-1} + b_n) (§4.1, Eq. 1) for a 3x3 convolution, pad 1.

With pattern and connectivity pruning the layer computes exactly the dense convolution over the
projected weights with the pruned taps and kernels set to zero, so the oracle is that definition:

    y[n, co, oy, ox] = sum_{ci, t} W_hat[co, ci, t] * x[n, ci, s*oy + dy(t), s*ox + dx(t)] + b[co]

(x read as zero outside the image), then max(y, 0) when sigma is ReLU.  For a depthwise layer
(groups = channels) the sum runs over ci = co only.  All arithmetic is IEEE float64 on inputs
widened exactly from fp32/fp16.

Two forms of the same sum:
* ``conv_loop``: scalar Python loops, for tiny cases;
* ``conv_ref``: nine shifted matrix products y = sum_t W_hat[:, :, t] @ shift_t(x) (a library
  matmul per tap), for workload sizes.

Error metric (reading of the tolerance "max relative error normalised by sum|w||x| per output"):
err = |y_gpu - y_ref| / (sum_{ci,t} |W_hat| |x| + |b| + 2^-1000); the |b| term covers outputs
whose receptive field is all zero, the tiny constant avoids 0/0.
"""
from __future__ import annotations

import numpy as np


def out_size(h: int, stride: int) -> int:
    return (h + 2 - 3) // stride + 1


def conv_loop(x, W_hat, b, stride: int = 1, relu: bool = False, depthwise: bool = False):
    """Scalar-loop definition (float64). x [N, C, H, W], W_hat [Cout, Cin_g, 3, 3], b [Cout]|None."""
    x = np.asarray(x, dtype=np.float64)
    W = np.asarray(W_hat, dtype=np.float64)
    N, C, H, Wd = x.shape
    cout, cin_g = W.shape[:2]
    Ho, Wo = out_size(H, stride), out_size(Wd, stride)
    y = np.zeros((N, cout, Ho, Wo), dtype=np.float64)
    for n in range(N):
        for co in range(cout):
            cis = [co] if depthwise else list(range(C))
            for oy in range(Ho):
                for ox in range(Wo):
                    acc = 0.0
                    for k, ci in enumerate(cis):
                        for ky in range(3):
                            for kx in range(3):
                                iy = stride * oy + ky - 1
                                ix = stride * ox + kx - 1
                                if 0 <= iy < H and 0 <= ix < Wd:
                                    acc += W[co, 0 if depthwise else k, ky, kx] * x[n, ci, iy, ix]
                    if b is not None:
                        acc += float(b[co])
                    y[n, co, oy, ox] = max(acc, 0.0) if relu else acc
    return y


def _shifted(xp: np.ndarray, ky: int, kx: int, Ho: int, Wo: int, s: int) -> np.ndarray:
    """x[:, :, s*oy + ky - 1, s*ox + kx - 1] for all (oy, ox), from the zero-padded input."""
    return xp[:, :, ky:ky + s * (Ho - 1) + 1:s, kx:kx + s * (Wo - 1) + 1:s]


def conv_ref(x, W_hat, b, stride: int = 1, relu: bool = False, depthwise: bool = False,
             absolute: bool = False):
    """Same sum as ``conv_loop`` as nine shifted float64 matrix products.

    ``absolute=True`` returns sum |W_hat| |x| + |b| instead (the error normaliser)."""
    x = np.asarray(x, dtype=np.float64)
    W = np.asarray(W_hat, dtype=np.float64)
    if absolute:
        x, W = np.abs(x), np.abs(W)
    N, C, H, Wd = x.shape
    cout, cin_g = W.shape[:2]
    Ho, Wo = out_size(H, stride), out_size(Wd, stride)
    xp = np.zeros((N, C, H + 2, Wd + 2), dtype=np.float64)
    xp[:, :, 1:H + 1, 1:Wd + 1] = x
    y = np.zeros((N, cout, Ho * Wo), dtype=np.float64)
    for ky in range(3):
        for kx in range(3):
            xs = _shifted(xp, ky, kx, Ho, Wo, stride).reshape(N, C, Ho * Wo)
            if depthwise:
                y += W[:, 0, ky, kx][None, :, None] * xs
            else:
                y += np.matmul(W[:, :, ky, kx], xs)
    y = y.reshape(N, cout, Ho, Wo)
    if b is not None:
        bb = np.asarray(b, dtype=np.float64)
        y += (np.abs(bb) if absolute else bb)[None, :, None, None]
    if relu and not absolute:
        np.maximum(y, 0.0, out=y)
    return y


def denominator(x, W_hat, b, stride: int = 1, depthwise: bool = False):
    """sum_{ci,t} |W_hat| |x| + |b| + 2^-1000 per output (float64)."""
    return conv_ref(x, W_hat, b, stride, False, depthwise, absolute=True) + 2.0 ** -1000


def max_norm_err(y_test, y_ref, denom) -> float:
    """max over outputs of |y_test - y_ref| / denom (y_test widened exactly to float64)."""
    d = np.abs(np.asarray(y_test, dtype=np.float64) - np.asarray(y_ref, dtype=np.float64))
    return float(np.max(d / denom)) if d.size else 0.0


def maxpool2x2(x):
    """2x2 max-pool, stride 2, floor mode: y[n,c,i,j] = max over x[n,c,2i+a,2j+b], a,b in {0,1}."""
    x = np.asarray(x)
    N, C, H, W = x.shape
    Ho, Wo = H // 2, W // 2
    v = x[:, :, :2 * Ho, :2 * Wo].reshape(N, C, Ho, 2, Wo, 2)
    return v.max(axis=(3, 5))
