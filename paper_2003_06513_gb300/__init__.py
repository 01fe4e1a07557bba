"""Pattern-pruned 3x3 convolution inference on one GB300 (arXiv 2003.06513).

The C library (``include/patconv.h``, built in-tree by ``build.py``) holds the whole path: the
host packer (pattern projection §4.3, connectivity pruning §4.4, filter grouping and compact
storage §3.4) and the sm_103a CUDA kernels (pattern-sparse convolution with fused bias + ReLU,
depthwise variant, max-pool).  This package is a thin ctypes binding over it; ``workloads``
holds the seeded synthetic inputs.  Importing the package does not load the library; the first
call that needs it does, and fails loudly if it cannot be built or loaded.
"""

__all__ = ["Layer", "pp_pack", "pp_conv", "pp_maxpool2x2", "default_patterns", "PatconvError"]


def __getattr__(name):
    if name in ("Layer", "pp_pack", "pp_conv", "pp_maxpool2x2", "default_patterns"):
        from . import api
        return getattr(api, name)
    if name == "PatconvError":
        from ._lib import PatconvError
        return PatconvError
    raise AttributeError(name)
