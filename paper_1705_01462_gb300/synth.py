"""Seeded synthetic inputs and workload shapes for FGQ.

This module holds no FGQ arithmetic.  It only describes layer shapes and draws the
seeded random tensors (fp32 weights and fp32 pre-quantisation activations) that both
the CUDA path and the CPU oracle consume.

Input recipe (stand-ins for the pre-trained ImageNet models of Section 4, which are not
available here):
  * weights  w ~ N(0, 2 / fan_in), fp32, fan_in = R*S*C/groups, stored [M][R][S][C/groups]
    (the reduction axis Kred in (r, s, c) order, c fastest);
  * activations |N(0, 1)| (half-normal, sigma = 1), fp32 NHWC, as produced by a ReLU;
  * one independent seed per layer: seed = 170501462 + layer index (+ a per-tensor offset).

Layer shapes follow the ResNet-50 / ResNet-101 / AlexNet networks of Section 4 (Table 1).
For ResNet the stride of a stage's first block sits on its first 1x1 convolution and on
the projection, as in the original Caffe models the paper's Caffe setup used.
"""
from __future__ import annotations

from dataclasses import dataclass, asdict
from typing import List

import numpy as np

BASE_SEED = 170501462


@dataclass(frozen=True)
class ConvLayer:
    name: str
    C: int          # input channels
    M: int          # output filters
    R: int
    S: int
    stride: int
    pad: int
    H: int          # input height
    W: int          # input width
    groups: int = 1

    @property
    def Ho(self) -> int:
        return (self.H + 2 * self.pad - self.R) // self.stride + 1

    @property
    def Wo(self) -> int:
        return (self.W + 2 * self.pad - self.S) // self.stride + 1

    @property
    def Kred(self) -> int:
        return self.R * self.S * (self.C // self.groups)

    @property
    def fan_in(self) -> int:
        return self.Kred

    def P(self, B: int) -> int:
        return B * self.Ho * self.Wo

    def ops(self, B: int) -> int:
        """Dense-equivalent operation count 2*M*P*Kred."""
        return 2 * self.M * self.P(B) * self.Kred

    def as_dict(self) -> dict:
        return asdict(self)


def _bottleneck_stack(blocks_per_stage: List[int]) -> List[ConvLayer]:
    layers = [ConvLayer("conv1", 3, 64, 7, 7, 2, 3, 224, 224)]
    H = 56
    cin = 64
    widths = [64, 128, 256, 512]
    for si, (nb, wd) in enumerate(zip(blocks_per_stage, widths)):
        stage = si + 2
        for b in range(nb):
            first = b == 0
            stride = 2 if (first and si > 0) else 1
            Hin = H
            Hmid = Hin // stride
            pfx = f"res{stage}{chr(ord('a') + b) if nb <= 26 else b}"
            layers.append(ConvLayer(f"{pfx}_branch2a", cin, wd, 1, 1, stride, 0, Hin, Hin))
            layers.append(ConvLayer(f"{pfx}_branch2b", wd, wd, 3, 3, 1, 1, Hmid, Hmid))
            layers.append(ConvLayer(f"{pfx}_branch2c", wd, 4 * wd, 1, 1, 1, 0, Hmid, Hmid))
            if first:
                layers.append(ConvLayer(f"{pfx}_branch1", cin, 4 * wd, 1, 1, stride, 0, Hin, Hin))
            cin = 4 * wd
            H = Hmid
    return layers


def resnet50_convs() -> List[ConvLayer]:
    """The 53 convolutions of ResNet-50 at 224x224 input."""
    return _bottleneck_stack([3, 4, 6, 3])


def resnet101_convs() -> List[ConvLayer]:
    """The 104 convolutions of ResNet-101 (23 blocks in conv4_x) at 224x224 input."""
    return _bottleneck_stack([3, 4, 23, 3])


def alexnet_convs() -> List[ConvLayer]:
    """AlexNet convolutions (two-tower convs as groups=2), 227x227 input."""
    return [
        ConvLayer("conv1", 3, 96, 11, 11, 4, 0, 227, 227),
        ConvLayer("conv2", 96, 256, 5, 5, 1, 2, 27, 27, groups=2),
        ConvLayer("conv3", 256, 384, 3, 3, 1, 1, 13, 13),
        ConvLayer("conv4", 384, 384, 3, 3, 1, 1, 13, 13, groups=2),
        ConvLayer("conv5", 384, 256, 3, 3, 1, 1, 13, 13, groups=2),
    ]


def alexnet_fcs() -> List[ConvLayer]:
    """AlexNet fully connected layers, expressed as 1x1 convolutions on a 1x1 map."""
    return [
        ConvLayer("fc6", 9216, 4096, 1, 1, 1, 0, 1, 1),
        ConvLayer("fc7", 4096, 4096, 1, 1, 1, 0, 1, 1),
        ConvLayer("fc8", 4096, 1000, 1, 1, 1, 0, 1, 1),
    ]


def resnet50_fc() -> ConvLayer:
    return ConvLayer("fc1000", 2048, 1000, 1, 1, 1, 0, 1, 1)


def conv2x_3x3() -> ConvLayer:
    """The ResNet-50 conv2_x 3x3 layer: 64 -> 64 filters, K = 3*3*64 = 576, 56x56 map."""
    return ConvLayer("res2a_branch2b", 64, 64, 3, 3, 1, 1, 56, 56)


# --------------------------------------------------------------------------- generators

def rng(seed: int) -> np.random.Generator:
    return np.random.default_rng(seed)


def weights(layer: ConvLayer, seed: int) -> np.ndarray:
    """fp32 [M][Kred] with Kred in (r, s, c) order; w ~ N(0, 2/fan_in)."""
    g = rng(seed)
    std = np.sqrt(2.0 / layer.fan_in)
    return (g.standard_normal((layer.M, layer.Kred), dtype=np.float32) * np.float32(std)).astype(np.float32)


def weights_matrix(M: int, K: int, seed: int, fan_in: int | None = None) -> np.ndarray:
    g = rng(seed)
    std = np.sqrt(2.0 / (fan_in or K))
    return (g.standard_normal((M, K), dtype=np.float32) * np.float32(std)).astype(np.float32)


def pow2_ternary_weights(layer: ConvLayer, seed: int) -> np.ndarray:
    """fp32 [M][Kred] with values in {-c, 0, +c}, c = 2^round(log2(sqrt(2 / fan_in))): each
    weight zero with probability 1/3, else of random sign.  Already ternary with one
    magnitude, so every group's scaling factor is c and every contraction sum is a multiple
    of c below 2^24 c: exact in fp32 in any order."""
    g = rng(seed)
    c = np.float32(2.0 ** round(np.log2(np.sqrt(2.0 / layer.fan_in))))
    u = g.integers(0, 3, size=(layer.M, layer.Kred))
    return ((u == 1).astype(np.float32) - (u == 2).astype(np.float32)) * c


def activations(shape, seed: int) -> np.ndarray:
    """fp32 half-normal (sigma = 1) post-ReLU activations of the given shape."""
    g = rng(seed)
    return np.abs(g.standard_normal(shape, dtype=np.float32)).astype(np.float32)


def torch_weights_matrix(M: int, K: int, seed: int, device, fan_in: int | None = None):
    """Same distribution as `weights_matrix`, drawn on `device` with a seeded torch generator."""
    import torch
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    std = float(np.sqrt(2.0 / (fan_in or K)))
    return torch.randn((M, K), generator=gen, device=device, dtype=torch.float32) * std


def torch_weights(layer: ConvLayer, seed: int, device):
    """Same distribution as `weights`, drawn on `device` with a seeded torch generator."""
    import torch
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    std = float(np.sqrt(2.0 / layer.fan_in))
    return torch.randn((layer.M, layer.Kred), generator=gen, device=device, dtype=torch.float32) * std


def torch_activations(shape, seed: int, device):
    import torch
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    return torch.randn(tuple(shape), generator=gen, device=device, dtype=torch.float32).abs_()


def layer_seed(index: int, offset: int = 0) -> int:
    return BASE_SEED + index + 1000 * offset
