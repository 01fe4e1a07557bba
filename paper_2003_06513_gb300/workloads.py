"""Seeded synthetic workloads shaped like the CNN layers of the paper's experiments (§5.1).

The paper evaluates VGG-16, ResNet-18/50 on CIFAR-10/ImageNet with pre-trained weights; none of
those are available here, so every tensor below is drawn from numpy's ``default_rng(seed)`` with
the layer shapes of those networks and He-normal weights.  This module holds shapes and random
draws only -- no projection, packing or convolution arithmetic -- and is the one module that both
the GPU path (tests, benchmark) and the CPU oracle take their inputs from.
"""
from __future__ import annotations

import dataclasses
from typing import List, Tuple

import numpy as np


@dataclasses.dataclass(frozen=True)
class ConvLayer:
    """One 3x3 convolution, pad 1: ``x[N, cin, h, w] -> y[N, cout, ho, wo]``."""

    name: str
    cin: int
    cout: int
    h: int
    w: int
    stride: int = 1
    depthwise: bool = False
    keep: float = 1.0
    w_seed: int = 0
    b_seed: int = 0
    x_seed: int = 0
    w_std: float = 0.0          # 0 -> He-normal sqrt(2 / (9 * cin_per_group))
    relu: bool = True
    pool_after: bool = False    # 2x2/2 max-pool applied to this layer's output (VGG block ends)

    @property
    def cin_g(self) -> int:
        return 1 if self.depthwise else self.cin

    @property
    def ho(self) -> int:
        return (self.h - 1) // self.stride + 1

    @property
    def wo(self) -> int:
        return (self.w - 1) // self.stride + 1


def he_std(cin_g: int) -> float:
    return float(np.sqrt(2.0 / (9.0 * cin_g)))


def weights(layer: ConvLayer) -> np.ndarray:
    """fp32 [cout, cin_g, 3, 3], N(0, std^2) from ``layer.w_seed``."""
    std = layer.w_std if layer.w_std > 0 else he_std(layer.cin_g)
    rng = np.random.default_rng(layer.w_seed)
    return (rng.standard_normal((layer.cout, layer.cin_g, 3, 3)) * std).astype(np.float32)


def bias(layer: ConvLayer, std: float = 0.1) -> np.ndarray:
    """fp32 [cout], N(0, std^2) from ``layer.b_seed``."""
    rng = np.random.default_rng(layer.b_seed)
    return (rng.standard_normal(layer.cout) * std).astype(np.float32)


def activations(shape: Tuple[int, ...], seed: int, relu: bool = False,
                dtype=np.float32) -> np.ndarray:
    """N(0,1) (optionally passed through max(.,0)) of ``shape`` from ``seed``, as ``dtype``."""
    rng = np.random.default_rng(seed)
    a = rng.standard_normal(shape, dtype=np.float32)
    if relu:
        np.maximum(a, 0, out=a)
    return a.astype(dtype, copy=False)


def layer_input(layer: ConvLayer, n: int, relu: bool = True, dtype=np.float32) -> np.ndarray:
    return activations((n, layer.cin, layer.h, layer.w), layer.x_seed, relu=relu, dtype=dtype)


# --------------------------------------------------------------------------------------------
# Workloads (shapes follow the networks named in the paper's §5.1; seeds are fixed here)
# --------------------------------------------------------------------------------------------

def single_layer() -> ConvLayer:
    """Single 3x3 conv, N=1, Cin=Cout=64, 32x32, stride 1, keep 0.5, bias + ReLU."""
    return ConvLayer("single64", 64, 64, 32, 32, 1, False, 0.5, w_seed=0, b_seed=2, x_seed=1)


VGG16_CHANNELS = [(3, 64), (64, 64), (64, 128), (128, 128), (128, 256), (256, 256), (256, 256),
                  (256, 512), (512, 512), (512, 512), (512, 512), (512, 512), (512, 512)]
VGG16_POOL_AFTER = {2, 4, 7, 10, 13}


def vgg16() -> List[ConvLayer]:
    """The 13 3x3 convs of VGG-16 on a 224x224 image; keep 1.0 on the first layer, 0.3 after."""
    layers = []
    h = 224
    for i, (cin, cout) in enumerate(VGG16_CHANNELS, start=1):
        layers.append(ConvLayer(f"vgg{i}", cin, cout, h, h, 1, False, 1.0 if i == 1 else 0.3,
                                w_seed=100 + i, b_seed=200 + i, x_seed=1 if i == 1 else 150 + i,
                                pool_after=i in VGG16_POOL_AFTER))
        if i in VGG16_POOL_AFTER:
            h //= 2
    return layers


def vgg16_image(n: int) -> np.ndarray:
    return activations((n, 3, 224, 224), seed=1, relu=False)


def resnet50_3x3() -> List[ConvLayer]:
    """The 16 3x3 bottleneck convs of ResNet-50 (widths 64/128/256/512), keep 0.4.

    Stage heads of stages 2-4 carry the stride 2 (torchvision placement)."""
    spec = ([(64, 56, 1)] * 3 + [(128, 56, 2)] + [(128, 28, 1)] * 3 + [(256, 28, 2)]
            + [(256, 14, 1)] * 5 + [(512, 14, 2)] + [(512, 7, 1)] * 2)
    return [ConvLayer(f"r50_{l}", c, c, h, h, s, False, 0.4, w_seed=300 + l, b_seed=450 + l,
                      x_seed=400 + l) for l, (c, h, s) in enumerate(spec)]


def mobilenet_v2_dw() -> List[ConvLayer]:
    """The 17 3x3 depthwise convs of MobileNet-V2 (224 input, standard strides), keep 1."""
    spec = [(32, 112, 1), (96, 112, 2), (144, 56, 1), (144, 56, 2), (192, 28, 1), (192, 28, 1),
            (192, 28, 2), (384, 14, 1), (384, 14, 1), (384, 14, 1), (384, 14, 1), (576, 14, 1),
            (576, 14, 1), (576, 14, 2), (960, 7, 1), (960, 7, 1), (960, 7, 1)]
    return [ConvLayer(f"mbv2_dw{l}", c, c, h, h, s, True, 1.0, w_seed=500 + l, b_seed=550 + l,
                      x_seed=600 + l, w_std=float(np.sqrt(2.0 / 9.0)))
            for l, (c, h, s) in enumerate(spec)]


def sweep() -> List[Tuple[ConvLayer, int, str]]:
    """Single-layer roofline sweep: (layer, batch, io dtype) over 288 points."""
    pts = []
    idx = 0
    for c in (128, 256, 512):
        for hw in (7, 14, 28, 56):
            for n in (1, 16, 64, 256):
                for keep in (1.0, 0.5, 0.25):
                    for dt in ("f32", "f16"):
                        pts.append((ConvLayer(f"sweep{idx}", c, c, hw, hw, 1, False, keep,
                                              w_seed=1000 + idx, b_seed=2000 + idx,
                                              x_seed=3000 + idx), n, dt))
                        idx += 1
    return pts
