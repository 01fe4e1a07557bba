"""Pattern library P = {M_1, ..., M_m} (§3.2 "kernel pattern pruning", §4.2).

A pattern is a binary 3x3 mask with exactly four ones: the kernel keeps four weights so that one
kernel maps onto a 4-wide SIMD operation (§3.2).  Masks are written here as 9-bit integers, bit t
for tap t, taps in raster order t = 3*(dy+1) + (dx+1) for dy, dx in {-1, 0, 1}:

    0 1 2
    3 4 5
    6 7 8

The library used by the workloads has m = 8 patterns (§4.2 finds m = 6-8 the sweet spot), all
containing the centre tap (§4.2 insight 1):

* family A (indices 0-3): centre + three of the four edge neighbours; index i drops the i-th edge
  in raster order (up, left, right, down);
* family B (indices 4-7): centre + one edge neighbour + the two corners flanking that edge; index
  4+i uses the i-th edge in raster order.

The paper draws its own 8-pattern library in a figure that is not available; this ordering is the
convention of this implementation and matters because ties go to the lowest index.
"""
from __future__ import annotations

from typing import List, Sequence, Tuple

CENTRE = 4


def tap(dy: int, dx: int) -> int:
    """Raster tap index of offset (dy, dx)."""
    return 3 * (dy + 1) + (dx + 1)


def offset(t: int) -> Tuple[int, int]:
    """(dy, dx) of raster tap t."""
    return t // 3 - 1, t % 3 - 1


# edge neighbours in raster order: up, left, right, down
EDGES = [(-1, 0), (0, -1), (0, 1), (1, 0)]


def _flanking_corners(edge: Tuple[int, int]) -> List[Tuple[int, int]]:
    """The two corners that share the edge's nonzero coordinate (e.g. up -> up-left, up-right)."""
    ey, ex = edge
    corners = [(-1, -1), (-1, 1), (1, -1), (1, 1)]
    if ey != 0:
        return [c for c in corners if c[0] == ey]
    return [c for c in corners if c[1] == ex]


def mask_of(taps: Sequence[int]) -> int:
    m = 0
    for t in taps:
        m |= 1 << t
    return m


def taps_of(mask: int) -> List[int]:
    """Taps of a mask in ascending raster order."""
    return [t for t in range(9) if (mask >> t) & 1]


def default8() -> List[int]:
    """The 8-pattern library described in the module docstring, as 9-bit masks."""
    fam_a = []
    for missing in EDGES:
        taps = [CENTRE] + [tap(*e) for e in EDGES if e != missing]
        fam_a.append(mask_of(taps))
    fam_b = []
    for e in EDGES:
        taps = [CENTRE, tap(*e)] + [tap(*c) for c in _flanking_corners(e)]
        fam_b.append(mask_of(taps))
    return fam_a + fam_b


def validate(masks: Sequence[int]) -> None:
    """A pattern library: 1 <= m <= 8 distinct 9-bit masks with exactly four taps each."""
    if not 1 <= len(masks) <= 8:
        raise ValueError("pattern library size must be in [1, 8]")
    for m in masks:
        if not 0 < int(m) < 512 or bin(int(m)).count("1") != 4:
            raise ValueError(f"pattern mask {m:#x} does not have exactly 4 taps")
    if len(set(int(m) for m in masks)) != len(masks):
        raise ValueError("duplicate pattern masks")


def grid(mask: int) -> str:
    """ASCII 3x3 drawing of a mask, 'x' = kept tap, '.' = pruned tap (rows top to bottom)."""
    rows = []
    for r in range(3):
        rows.append("".join("x" if (mask >> (3 * r + c)) & 1 else "." for c in range(3)))
    return "\n".join(rows)


def design_library(kernels, m: int) -> List[int]:
    """Pattern library by the heuristic of §4.2 (plain loops over the kernels).

    The central weight is never pruned; each kernel proposes the pattern formed by the centre and
    the locations of its three largest weights (largest magnitude, among the eight non-central
    taps -- readings of this library: magnitude, and equal magnitudes take the lower raster tap
    first).  The m most commonly proposed patterns over all kernels form the library, ordered by
    count descending, equal counts by mask value ascending.  ``kernels``: rows of 9 raster taps.
    """
    counts = {}
    for row in kernels:
        w = [float(v) for v in row]
        chosen = [CENTRE]
        for _ in range(3):
            best = None
            for t in range(9):
                if t in chosen:
                    continue
                if best is None or abs(w[t]) > abs(w[best]):
                    best = t
            chosen.append(best)
        mk = mask_of(chosen)
        counts[mk] = counts.get(mk, 0) + 1
    ranked = sorted(counts, key=lambda mk: (-counts[mk], mk))
    return ranked[:m]
