"""CPU oracle for pattern-pruned 3x3 convolution inference (arXiv 2003.06513).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg
of ``bench.py`` import this package.  The product path (``paper_2003_06513_gb300`` and its CUDA
library) never imports, calls or links anything here, and this package imports nothing from it
except the seeded input generators, which hold no arithmetic of the method.

Plain, slow, obviously-correct numpy in IEEE float64:

* ``patterns``  -- the 4-tap pattern library (§3.2, §4.2).
* ``project``   -- Euclidean projection of each kernel onto the pattern set (§4.3, Eq. 5-6) and
                   connectivity pruning to at most beta kernels (§4.4, set C'_n).
* ``layout``    -- filter grouping and the compact weight layout (§3.4: filter kernel reorder,
                   compressed weight storage), written from this library's layout specification.
* ``conv``      -- the layer forward sigma(W X + b) (§4.1, Eq. 1) as a dense 3x3 convolution over
                   the projected weights with the zeros in place, and the normalised error metric.
* ``admm``      -- the layer-wise ADMM pruning of Algorithm 1 (§4.3-4.5, Eq. 4-7) with a hand-written
                   gradient, for the training-side module of the library.

Every function is pinned by ``tests/test_oracle_*.py`` against something other than itself:
brute-force enumeration, torch's CPU convolution, hand-computed fixtures under
``tests/golden/`` and the paper's invariants (4 nonzeros per kernel, beta kept kernels, the 2.25x
pattern-only compression rate).  The layout is pinned by a decoder that rebuilds the projected
weights from the sections; its byte-level encoding itself is a specification of this library,
not a result the paper prints ("parity unpinned" against the paper for the byte encoding).
"""

from . import admm, conv, layout, patterns, project  # noqa: F401
