"""Seeded synthetic inputs shaped like the CNN workloads of arXiv 1910.11971.

This module only draws random tensors and lists layer shapes.  It holds none of
the method's arithmetic (no packing, no products), so both the GPU path and the
CPU oracle can take their inputs from it.

The paper trains on ImageNet / CIFAR (Sec. 6); neither the datasets nor trained
weights are used here.  Inputs are random tensors with the layer shapes of the
paper's networks: dense weights drawn from a normal distribution (He-normal for
convolutions), activations drawn as ReLU(N(0, 1)) (post-ReLU feature maps) or
U(-1, 1) / N(0, 1) where stated.  Draws are fp32 from a seeded ``torch.Generator``
and are rounded to bf16 (round-to-nearest-even) for the bf16 workloads.

Workloads:
  * ``tiny_linear``   Cin=Cout=64, N=32, G=4, K=2, fp32 (parity / latency case)
  * ``bottleneck_1x1`` ResNet 1x1 bottleneck as a product: N = 32*56*56 = 100352,
    256 -> 1024, G=8, K=2, fp32, W ~ N(0, 2/256), X = ReLU(N(0,1))
  * ``conv3x3_28``    3x3 NHWC conv, batch 64, 28x28, 128 -> 128, s1 p1, G=16,
    K=4, bf16, He-normal W, ReLU(N(0,1)) X
  * ``resnet50_stack`` the 52 convolutions of ResNet-50 (v1.5: stride on the 3x3)
    after the stem, batch 128 at 224x224 input, bf16, G=8, K in {1, 2, 4}; each
    layer has its own He-normal W and ReLU(N(0,1)) input, seed = layer index
  * ``sweep_4096``    4096 -> 4096 product, N=8192, bf16, W ~ N(0, 1/4096),
    X ~ N(0,1), (G, K) over G in {4,8,16,32} and K/G in {1/8, 1/4, 1/2}
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import List, Optional, Tuple

import torch


@dataclass(frozen=True)
class LinearCase:
    name: str
    N: int
    Cin: int
    Cout: int
    G: int
    K: int
    dtype: str  # "f32" or "bf16"
    w_std: float
    x_dist: str  # "uniform", "relu_normal", "normal"
    seed: int = 0

    @property
    def R(self) -> int:
        return self.Cin

    def nz_flops(self) -> int:
        return 2 * self.N * self.R * self.Cout * self.K // self.G

    def dense_flops(self) -> int:
        return 2 * self.N * self.R * self.Cout


@dataclass(frozen=True)
class ConvCase:
    name: str
    B: int
    H: int
    W: int
    Cin: int
    Cout: int
    KH: int
    KW: int
    stride: int
    pad: int
    G: int
    K: int
    dtype: str
    seed: int = 0

    @property
    def R(self) -> int:
        return self.Cin * self.KH * self.KW

    @property
    def P(self) -> int:
        return (self.H + 2 * self.pad - self.KH) // self.stride + 1

    @property
    def Q(self) -> int:
        return (self.W + 2 * self.pad - self.KW) // self.stride + 1

    @property
    def N(self) -> int:
        return self.B * self.P * self.Q

    @property
    def w_std(self) -> float:
        return math.sqrt(2.0 / self.R)  # He-normal, fan_in = Cin*KH*KW

    def nz_flops(self) -> int:
        return 2 * self.N * self.R * self.Cout * self.K // self.G

    def dense_flops(self) -> int:
        return 2 * self.N * self.R * self.Cout


TINY_LINEAR = LinearCase("tiny_linear", N=32, Cin=64, Cout=64, G=4, K=2, dtype="f32",
                         w_std=1.0, x_dist="uniform")
BOTTLENECK_1X1 = LinearCase("bottleneck_1x1", N=32 * 56 * 56, Cin=256, Cout=1024, G=8, K=2,
                            dtype="f32", w_std=math.sqrt(2.0 / 256), x_dist="relu_normal")
CONV3X3_28 = ConvCase("conv3x3_28", B=64, H=28, W=28, Cin=128, Cout=128, KH=3, KW=3, stride=1,
                      pad=1, G=16, K=4, dtype="bf16")

SWEEP_POINTS: Tuple[Tuple[int, int], ...] = (
    (4, 1), (4, 2),
    (8, 1), (8, 2), (8, 4),
    (16, 2), (16, 4), (16, 8),
    (32, 4), (32, 8), (32, 16),
)


def sweep_case(G: int, K: int) -> LinearCase:
    return LinearCase(f"sweep_4096_G{G}_K{K}", N=8192, Cin=4096, Cout=4096, G=G, K=K,
                      dtype="bf16", w_std=math.sqrt(1.0 / 4096), x_dist="normal")


def resnet50_layers(batch: int = 128, G: int = 8, K: int = 2) -> List[ConvCase]:
    """The 52 convolutions of ResNet-50 v1.5 after the stem (input 224x224 ->
    56x56x64 after the stem), in network order."""
    layers: List[ConvCase] = []

    def add(h, cin, cout, k, s):
        i = len(layers)
        layers.append(ConvCase(f"resnet50_l{i:02d}_{k}x{k}_{cin}to{cout}_s{s}_h{h}", B=batch, H=h,
                               W=h, Cin=cin, Cout=cout, KH=k, KW=k, stride=s, pad=k // 2,
                               G=G, K=K, dtype="bf16", seed=i))

    h, cin = 56, 64
    for width, blocks, stride in ((64, 3, 1), (128, 4, 2), (256, 6, 2), (512, 3, 2)):
        out = 4 * width
        for b in range(blocks):
            s = stride if b == 0 else 1
            add(h, cin, width, 1, 1)
            add(h, width, width, 3, s)
            h2 = (h + 2 - 3) // s + 1
            add(h2, width, out, 1, 1)
            if b == 0:
                add(h, cin, out, 1, s)
            h, cin = h2, out
    assert len(layers) == 52
    return layers


def mobilenetv2_pointwise_layers(batch: int = 128, G: int = 8, K: int = 2) -> List[ConvCase]:
    """The 34 pointwise (1x1) convolutions of MobileNetV2 (width 1.0, 224x224
    input, torchvision layout): per inverted-residual block the expansion (when
    the expansion factor is 6) at the block's input resolution and the projection
    at its output resolution, then the final 1x1 320 -> 1280; the paper makes
    these layers CCI-sparse (Sec. 4, Sec. 5; G = 8, K = 2 is its 75 % case)."""
    layers: List[ConvCase] = []

    def add(h, cin, cout):
        i = len(layers)
        layers.append(ConvCase(f"mobilenetv2_pw{i:02d}_{cin}to{cout}_h{h}", B=batch, H=h, W=h, Cin=cin,
                               Cout=cout, KH=1, KW=1, stride=1, pad=0, G=G, K=K, dtype="bf16", seed=100 + i))

    h, cin = 112, 32
    for t, c, n, s in ((1, 16, 1, 1), (6, 24, 2, 2), (6, 32, 3, 2), (6, 64, 4, 2), (6, 96, 3, 1),
                       (6, 160, 3, 2), (6, 320, 1, 1)):
        for b in range(n):
            stride = s if b == 0 else 1
            hidden = cin * t
            if t != 1:
                add(h, cin, hidden)
            h = (h + 2 - 3) // stride + 1  # the 3x3 depthwise convolution (not CCI)
            add(h, hidden, c)
            cin = c
    add(h, cin, 1280)
    assert len(layers) == 34
    return layers


def resnet50_roles() -> List[str]:
    """Role of each of the 52 layers of resnet50_layers() in its bottleneck block:
    'a' (1x1 reduce, reads the block input), 'b' (3x3, reads a's output), 'c' (1x1
    expand, reads b's output; its output is the next block's input when the
    residual add is left out) and 'proj' (strided 1x1 shortcut, reads the block
    input)."""
    roles: List[str] = []
    for blocks in (3, 4, 6, 3):
        for b in range(blocks):
            roles += ["a", "b", "c"] + (["proj"] if b == 0 else [])
    assert len(roles) == 52
    return roles


# ---------------------------------------------------------------------------
# seeded draws
# ---------------------------------------------------------------------------

def _gen(seed: int, device: str) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def _to_dtype(t: torch.Tensor, dtype: str) -> torch.Tensor:
    if dtype == "f32":
        return t.contiguous()
    if dtype == "bf16":
        return t.to(torch.bfloat16).contiguous()  # round to nearest even
    raise ValueError(dtype)


def draw_x(shape, dist: str, dtype: str, seed: int, device: str = "cpu") -> torch.Tensor:
    g = _gen(seed, device)
    if dist == "uniform":
        t = torch.rand(shape, generator=g, device=device, dtype=torch.float32) * 2.0 - 1.0
    elif dist == "normal":
        t = torch.randn(shape, generator=g, device=device, dtype=torch.float32)
    elif dist == "relu_normal":
        t = torch.randn(shape, generator=g, device=device, dtype=torch.float32).clamp_min_(0.0)
    else:
        raise ValueError(dist)
    return _to_dtype(t, dtype)


def draw_w(Cout: int, R: int, std: float, dtype: str, seed: int, device: str = "cpu") -> torch.Tensor:
    """Dense weights W[Cout][R] ~ N(0, std^2); a separate stream from X's."""
    g = _gen(seed + 7919, device)
    t = torch.randn((Cout, R), generator=g, device=device, dtype=torch.float32) * std
    return _to_dtype(t, dtype)


def linear_inputs(case: LinearCase, device: str = "cpu", N: Optional[int] = None):
    """(X[N][Cin], W[Cout][Cin]) for a product workload."""
    n = case.N if N is None else N
    X = draw_x((n, case.Cin), case.x_dist, case.dtype, case.seed, device)
    W = draw_w(case.Cout, case.R, case.w_std, case.dtype, case.seed, device)
    return X, W


def conv_inputs(case: ConvCase, device: str = "cpu"):
    """(X NHWC [B][H][W][Cin], W OHWI flattened [Cout][KH*KW*Cin])."""
    X = draw_x((case.B, case.H, case.W, case.Cin), "relu_normal", case.dtype, case.seed, device)
    W = draw_w(case.Cout, case.R, case.w_std, case.dtype, case.seed, device)
    return X, W


def random_small(seed: int, dtype: str, N: int, Cin: int, Cout: int, dist: str = "normal",
                 device: str = "cpu"):
    """Small random product inputs for edge-case tests."""
    X = draw_x((N, Cin), dist, dtype, seed, device)
    W = draw_w(Cout, Cin, 1.0, dtype, seed, device)
    return X, W


def integer_valued(shape, lo: int, hi: int, seed: int) -> torch.Tensor:
    """Small integers as float32 (exact in fp32, bf16 when |v| <= 256, and fp64):
    products and sums of them are exact, so two correct routines agree bit for bit."""
    g = _gen(seed, "cpu")
    return torch.randint(lo, hi + 1, shape, generator=g, dtype=torch.int64).to(torch.float32)
