"""Projection onto the pattern set (§4.3, Eq. 5-6) and connectivity pruning (§4.4).

Kernel pattern pruning.  The proximal step of the ADMM solution is the Euclidean projection of a
layer's weights onto C_n = {every 3x3 kernel has its support inside one pattern of P} (Eq. 6).
C_n is a union of coordinate subspaces, so the projection acts kernel by kernel: restricting a
kernel w to a mask M keeps the energy s_M = sum_{t in M} w_t^2 and leaves ||w||^2 - s_M behind,
hence the closest point keeps the pattern whose pruned kernel has the largest Frobenius norm
(the closed form stated in §4.3).

Readings where the paper is silent (each one is a convention of this implementation):

* scores are computed in IEEE float64 from the fp32 weights, each square exact, summed strictly
  left to right over the pattern's taps in ascending raster order: ((a^2 + b^2) + c^2) + d^2;
* ties in the argmax go to the lowest pattern index (so an all-zero or centre-only kernel gets
  pattern 0);
* a non-finite weight is an error.

Connectivity pruning.  C'_n = {at most beta_n nonzero kernels} (§4.4).  Applied after the pattern
projection, keeping the beta kernels with the largest retained energy s_{p*} makes the result the
Euclidean projection onto C_n intersected with C'_n: dropping a projected kernel costs exactly its
retained energy.  Readings: beta = floor(keep * K + 0.5) in float64 (K = number of kernels),
clamped to [1, K]; ranking by (retained energy descending, flat index co*Cin_g + ci ascending).
"""
from __future__ import annotations

import math
from typing import Dict, Sequence

import numpy as np

from . import patterns as P


def check_weights(W: np.ndarray) -> np.ndarray:
    W = np.asarray(W)
    if W.dtype != np.float32 or W.ndim != 4 or W.shape[2:] != (3, 3):
        raise ValueError("weights must be float32 [Cout, Cin_g, 3, 3]")
    if W.shape[0] < 1 or W.shape[1] < 1:
        raise ValueError("empty weight tensor")
    if not np.all(np.isfinite(W)):
        raise ValueError("non-finite weight")
    return W


def scores(W: np.ndarray, masks: Sequence[int]) -> np.ndarray:
    """Retained energy s[co, ci, p] of every kernel under every pattern, float64.

    Elementwise float64 operations in a fixed order, so the result is the same bit pattern as a
    scalar loop ((a*a + b*b) + c*c) + d*d over the pattern's ascending taps."""
    W = check_weights(W)
    P.validate(masks)
    w = W.reshape(W.shape[0], W.shape[1], 9).astype(np.float64)
    out = np.empty(W.shape[:2] + (len(masks),), dtype=np.float64)
    for p, m in enumerate(masks):
        t = P.taps_of(int(m))
        s = w[:, :, t[0]] * w[:, :, t[0]]
        for k in t[1:]:
            s = s + w[:, :, k] * w[:, :, k]
        out[:, :, p] = s
    return out


def choose(s: np.ndarray) -> np.ndarray:
    """p* = the first index of the maximum score over the pattern axis (ties -> lowest index)."""
    return np.argmax(s, axis=-1).astype(np.int64)


def n_keep(keep: float, n_kernels: int) -> int:
    """beta = floor(keep * K + 0.5) in float64, clamped to [1, K]."""
    keep = float(keep)
    if not (keep > 0.0 and keep <= 1.0):
        raise ValueError("keep must lie in (0, 1]")
    b = math.floor(keep * float(n_kernels) + 0.5)
    return int(min(max(b, 1), n_kernels))


def connectivity(retained: np.ndarray, beta: int) -> np.ndarray:
    """Boolean keep-mask over kernels [Cout, Cin_g]: the beta largest retained energies, ties
    broken by the lower flat index."""
    flat = retained.reshape(-1)
    order = np.lexsort((np.arange(flat.size), -flat))   # primary: -score; secondary: index
    kept = np.zeros(flat.size, dtype=bool)
    kept[order[:beta]] = True
    return kept.reshape(retained.shape)


def project(W: np.ndarray, masks: Sequence[int], keep: float) -> Dict[str, object]:
    """Pattern projection followed by connectivity pruning.

    Returns ``pid`` (int64 [Cout, Cin_g], pattern index or -1 for a pruned kernel), ``W_hat``
    (float32 [Cout, Cin_g, 3, 3], the projected weights: bit copies of W on the kept taps, zeros
    elsewhere), ``beta``, the score table ``s`` and the chosen pattern ``best`` before pruning."""
    W = check_weights(W)
    s = scores(W, masks)
    best = choose(s)
    retained = np.take_along_axis(s, best[..., None], axis=-1)[..., 0]
    beta = n_keep(keep, W.shape[0] * W.shape[1])
    kept = connectivity(retained, beta)
    pid = np.where(kept, best, -1)
    mask_arr = np.array([[(int(m) >> t) & 1 for t in range(9)] for m in masks], dtype=bool)
    keep_taps = mask_arr[best] & kept[..., None]                    # [Cout, Cin_g, 9]
    w9 = W.reshape(W.shape[0], W.shape[1], 9)
    W_hat = np.where(keep_taps, w9, np.float32(0)).astype(np.float32).reshape(W.shape)
    return {"pid": pid, "W_hat": W_hat, "beta": beta, "s": s, "best": best}
