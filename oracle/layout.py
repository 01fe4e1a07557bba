"""Filter grouping and compact weight storage (§3.4), as specified by this library.

The paper names two pattern-enabled passes that act on the weights: *filter kernel reorder*
(group filters of similar length and pattern together, against control-flow overhead, thread
divergence and load imbalance) and *compressed weight storage* (a compact format built on the
fact that every kept kernel follows a known pattern).  It gives their intent, not their bytes;
the byte layout below is this library's specification, written here independently of the packer
so that the two can be compared bit for bit.

Specification (F = 8 filters per group, G = ceil(Cout / F), K = Cin_g kernels per filter):

* filter order: filters sorted by (kept-kernel count descending, pattern-id sequence over ci
  ascending with a pruned kernel counted as 15, original index ascending); the j-th filter of
  that order goes to group g = j mod G in round r = j div G (g = G-1 - (j mod G) when r is odd:
  snake order, so every group gets a similar number of kept kernels) and slot r, i.e.
  perm[8g + r]; group g owns perm[8g .. 8g+7]; missing slots are padding (perm = 0xFFFFFFFF);
* header  u32[16]: magic 'PPK1' (0x314B5050), version 1, Cout, Cin_g, groups, stride,
  n_patterns, beta, F, G, the masks two per word (low half first) in 4 words, 0, 0;
* pid     i8 [Cout][Cin_g]: pattern index, -1 = pruned, original filter order;
* perm    u32[G*F];
* desc    u64[G][Cin_g]: bits 0-3 = number c of kept kernels of group g at input channel ci;
  entry j < c at bits 4+6j .. 9+6j = (slot f << 3) | pattern index, slots ascending;
* kofs    u32[G*Cin_g + 1]: kept kernels preceding (g, ci) in (g, ci, slot) order; last = beta;
* vals    f32[beta][4]: per kept kernel in (g, ci, slot) order, the weights at the pattern's four
  taps in ascending raster order (bit copies);
* dense   f32[Cout][Cin_g][9]: the projected weights with zeros in place;
* image   the device image: perm | desc | kofs | vals, each section starting at a multiple of
  256 bytes, gaps zero.
"""
from __future__ import annotations

from typing import Dict, Sequence

import numpy as np

from . import patterns as P

F = 8
MAGIC = 0x314B5050
VERSION = 1
PAD = 0xFFFFFFFF


def _align(n: int, a: int = 256) -> int:
    return (n + a - 1) // a * a


def filter_order(pid: np.ndarray) -> list:
    """Original filter indices in slot order (the filter kernel reorder)."""
    cout = pid.shape[0]
    keys = []
    for co in range(cout):
        row = pid[co]
        count = int(np.count_nonzero(row >= 0))
        seq = tuple(int(p) if p >= 0 else 15 for p in row)
        keys.append((-count, seq, co))
    keys.sort()
    return [k[2] for k in keys]


def build(W: np.ndarray, pid: np.ndarray, masks: Sequence[int], groups: int, stride: int,
          beta: int) -> Dict[str, np.ndarray]:
    """All sections of the packed layer, as numpy arrays (``image`` as uint8 bytes)."""
    cout, cin_g = pid.shape
    G = (cout + F - 1) // F
    order = filter_order(pid)
    perm = np.full(G * F, PAD, dtype=np.uint32)
    for j, co in enumerate(order):
        r, pos = divmod(j, G)
        g = pos if r % 2 == 0 else G - 1 - pos
        perm[g * F + r] = co

    desc = np.zeros(G * cin_g, dtype=np.uint64)
    kofs = np.zeros(G * cin_g + 1, dtype=np.uint32)
    vals = []
    n = 0
    for g in range(G):
        for ci in range(cin_g):
            kofs[g * cin_g + ci] = n
            word = 0
            c = 0
            for f in range(F):
                if perm[g * F + f] == PAD:
                    continue
                co = int(perm[g * F + f])
                p = int(pid[co, ci])
                if p < 0:
                    continue
                word |= ((f << 3) | p) << (4 + 6 * c)
                c += 1
                taps = P.taps_of(int(masks[p]))
                vals.append([W[co, ci, t // 3, t % 3] for t in taps])
                n += 1
            desc[g * cin_g + ci] = word | c
    kofs[G * cin_g] = n
    assert n == beta
    vals_arr = np.array(vals, dtype=np.float32).reshape(-1, 4)

    header = np.zeros(16, dtype=np.uint32)
    header[:10] = [MAGIC, VERSION, cout, cin_g, groups, stride, len(masks), beta, F, G]
    mk = list(int(m) for m in masks) + [0] * (8 - len(masks))
    for i in range(4):
        header[10 + i] = mk[2 * i] | (mk[2 * i + 1] << 16)

    dense = np.zeros((cout, cin_g, 9), dtype=np.float32)
    for co in range(cout):
        for ci in range(cin_g):
            p = int(pid[co, ci])
            if p >= 0:
                for t in P.taps_of(int(masks[p])):
                    dense[co, ci, t] = W[co, ci, t // 3, t % 3]

    parts = [perm.tobytes(), desc.tobytes(), kofs.tobytes(), vals_arr.tobytes()]
    image = bytearray()
    for b in parts:
        image += b + bytes(_align(len(b)) - len(b))
    return {"header": header, "pid": pid.astype(np.int8), "perm": perm, "desc": desc,
            "kofs": kofs, "vals": vals_arr, "dense": dense,
            "image": np.frombuffer(bytes(image), dtype=np.uint8)}


def decode(sections: Dict[str, np.ndarray], masks: Sequence[int]) -> np.ndarray:
    """Rebuild the dense projected weights [Cout, Cin_g, 3, 3] from header/perm/desc/kofs/vals."""
    h = sections["header"]
    cout, cin_g, G = int(h[2]), int(h[3]), int(h[9])
    out = np.zeros((cout, cin_g, 9), dtype=np.float32)
    perm, desc, kofs, vals = (sections[k] for k in ("perm", "desc", "kofs", "vals"))
    for g in range(G):
        for ci in range(cin_g):
            word = int(desc[g * cin_g + ci])
            c = word & 15
            base = int(kofs[g * cin_g + ci])
            assert int(kofs[g * cin_g + ci + 1]) - base == c
            for j in range(c):
                code = (word >> (4 + 6 * j)) & 63
                f, p = code >> 3, code & 7
                co = int(perm[g * F + f])
                for k, t in enumerate(P.taps_of(int(masks[p]))):
                    out[co, ci, t] = vals[base + j, k]
    return out.reshape(cout, cin_g, 3, 3)
