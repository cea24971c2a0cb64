"""Seeded synthetic workloads: layer shapes and input generators.

This module draws random numbers and describes layer shapes; it holds none
of the method's arithmetic (no scoring, pruning, packing or convolution).
Both the CUDA path and the CPU oracle are fed from the arrays it returns.

The paper evaluates 1xN pruning on pre-trained MobileNet-V1/V2/V3 and
ResNet-50 on ILSVRC-2012 (Sec. 4.1).  Neither the dataset nor the trained
weights are available, so every workload here is synthetic: layer shapes
follow the standard MobileNet-V2 (width 1.0, 224x224 input) and ResNet-50
bottleneck schedules, weights are Kaiming-normal (std sqrt(2 / fan_in)) or
N(0, 0.05), and activations are ReLU(N(0, 1)), all from
``torch.Generator(seed)`` on the CPU in float32.
"""
from __future__ import annotations

import dataclasses
from typing import List, Optional

import numpy as np
import torch


@dataclasses.dataclass
class ConvLayer:
    """One 1xN-pruned convolution: geometry, block width N, rate, dtype, seeds."""
    name: str
    B: int
    H: int
    W: int
    C_in: int
    C_out: int
    KH: int = 1
    KW: int = 1
    stride: int = 1
    pad: int = 0
    dil: int = 1
    N: int = 4
    rate: float = 0.5
    dtype: str = "f32"          # "f32" or "bf16" (bf16 inputs, fp32 accumulate)
    seed: int = 0
    init: str = "kaiming"       # "kaiming" or "normal005"

    @property
    def Ho(self) -> int:
        return (self.H + 2 * self.pad - self.dil * (self.KH - 1) - 1) // self.stride + 1

    @property
    def Wo(self) -> int:
        return (self.W + 2 * self.pad - self.dil * (self.KW - 1) - 1) // self.stride + 1

    @property
    def pixels(self) -> int:
        return self.B * self.Ho * self.Wo

    @property
    def K(self) -> int:
        return self.KH * self.KW * self.C_in

    def with_(self, **kw) -> "ConvLayer":
        return dataclasses.replace(self, **kw)


def _gen(seed: int) -> torch.Generator:
    g = torch.Generator(device="cpu")
    g.manual_seed(int(seed))
    return g


def weights(layer: ConvLayer, salt: int = 0) -> torch.Tensor:
    """OIHW float32 weights: Kaiming-normal or N(0, 0.05)."""
    shape = (layer.C_out, layer.C_in, layer.KH, layer.KW)
    w = torch.randn(shape, generator=_gen(1_000_003 * layer.seed + 2 * salt + 17),
                    dtype=torch.float32)
    if layer.init == "normal005":
        std = 0.05
    else:
        std = (2.0 / (layer.C_in * layer.KH * layer.KW)) ** 0.5
    return w * std


def activations(layer: ConvLayer, salt: int = 0) -> torch.Tensor:
    """NHWC float32 activations, ReLU(N(0, 1))."""
    shape = (layer.B, layer.H, layer.W, layer.C_in)
    x = torch.randn(shape, generator=_gen(1_000_003 * layer.seed + 2 * salt + 18),
                    dtype=torch.float32)
    return x.clamp_min_(0.0)


def bias(layer: ConvLayer, salt: int = 0, scale: float = 0.1) -> torch.Tensor:
    """Per-output-channel float32 bias, N(0, scale)."""
    b = torch.randn((layer.C_out,), generator=_gen(1_000_003 * layer.seed + 2 * salt + 19),
                    dtype=torch.float32)
    return b * scale


def next_layer_weights(C_in: int, C_out: int, seed: int, std: float = 0.05,
                       KH: int = 1, KW: int = 1) -> torch.Tensor:
    """Random weights of the following layer, for the rearrangement check."""
    w = torch.randn((C_out, C_in, KH, KW), generator=_gen(7_000_001 + seed),
                    dtype=torch.float32)
    return w * std


def sample_pixels(total: int, count: int, seed: int,
                  must: Optional[List[int]] = None) -> np.ndarray:
    """Sorted distinct flattened output-pixel indices for sampled parity."""
    rng = np.random.default_rng(seed)
    count = min(count, total)
    pick = rng.choice(total, size=count, replace=False)
    if must:
        pick = np.concatenate([pick, np.asarray(must, np.int64)])
    return np.unique(pick.astype(np.int64))


# --------------------------------------------------------------------------
# The five synthetic workloads.
# --------------------------------------------------------------------------

def config1() -> List[ConvLayer]:
    """Single 1x1 conv, fp32, 1x28x28x64 -> 64, N=4, 50%, N(0, 0.05) weights."""
    return [ConvLayer("cfg1_1x1_64_64", 1, 28, 28, 64, 64, N=4, rate=0.5,
                      dtype="f32", init="normal005")]


def config2(dtype: str = "f32") -> List[ConvLayer]:
    """ResNet-50 stage-2 3x3: 64x28x28x128 -> 128, s1 p1, N=8, 50%."""
    return [ConvLayer(f"cfg2_3x3_128_128_{dtype}", 64, 28, 28, 128, 128, 3, 3, 1, 1, 1,
                      N=8, rate=0.5, dtype=dtype)]


def mobilenet_v2_1x1(B: int = 128, res: int = 224, N: int = 4, rate: float = 0.5,
                     dtype: str = "f32") -> List[ConvLayer]:
    """All expand/project 1x1 convs of MobileNet-V2 (width 1.0) plus conv_last.

    The first 3x3 conv and the depthwise 3x3 convs are not 1x1 layers and are
    not part of this stack; their stride sets the next 1x1 layer's size."""
    settings = [(1, 16, 1, 1), (6, 24, 2, 2), (6, 32, 3, 2), (6, 64, 4, 2),
                (6, 96, 3, 1), (6, 160, 3, 2), (6, 320, 1, 1)]
    layers: List[ConvLayer] = []
    c_in, hw = 32, res // 2
    li = 0
    for bi, (t, c, n, s) in enumerate(settings):
        for r in range(n):
            stride = s if r == 0 else 1
            hidden = c_in * t
            if t != 1:
                layers.append(ConvLayer(f"mbv2_b{bi + 1}.{r + 1}_expand", B, hw, hw, c_in,
                                        hidden, N=N, rate=rate, dtype=dtype, seed=li))
                li += 1
            hw_out = (hw + 2 - 3) // stride + 1          # depthwise 3x3, pad 1
            layers.append(ConvLayer(f"mbv2_b{bi + 1}.{r + 1}_project", B, hw_out, hw_out,
                                    hidden, c, N=N, rate=rate, dtype=dtype, seed=li))
            li += 1
            c_in, hw = c, hw_out
    layers.append(ConvLayer("mbv2_conv_last", B, hw, hw, c_in, 1280, N=N, rate=rate,
                            dtype=dtype, seed=li))
    return layers


@dataclasses.dataclass(frozen=True)
class MBv2Block:
    """One inverted-residual block of MobileNet-V2 (width 1.0): expand 1x1 to
    `hidden` channels (absent when hidden == c_in, expansion 1), depthwise
    3x3 with `stride`, project 1x1 to c_out; residual when stride 1 and
    c_in == c_out.  Input [B, hw, hw, c_in]."""
    name: str
    B: int
    hw: int
    c_in: int
    hidden: int
    c_out: int
    stride: int
    N: int = 4
    rate: float = 0.5
    dtype: str = "f32"
    seed: int = 0

    @property
    def hw_out(self) -> int:
        return (self.hw + 2 - 3) // self.stride + 1

    @property
    def kept_flops(self) -> float:
        """2 x kept multiply-adds of the two pruned 1x1 convs + the dense depthwise."""
        keep = 1.0 - self.rate
        e = 0 if self.hidden == self.c_in else self.B * self.hw * self.hw * self.c_in * self.hidden * keep
        d = self.B * self.hw_out * self.hw_out * self.hidden * 9
        pr = self.B * self.hw_out * self.hw_out * self.hidden * self.c_out * keep
        return 2.0 * (e + d + pr)


def mobilenet_v2_blocks(B: int = 1, res: int = 224, N: int = 4, rate: float = 0.5,
                        dtype: str = "f32") -> List[MBv2Block]:
    """The 17 inverted-residual blocks of MobileNet-V2 (after the 3x3 stem,
    which leaves res/2 x res/2 x 32)."""
    settings = [(1, 16, 1, 1), (6, 24, 2, 2), (6, 32, 3, 2), (6, 64, 4, 2),
                (6, 96, 3, 1), (6, 160, 3, 2), (6, 320, 1, 1)]
    blocks: List[MBv2Block] = []
    c_in, hw = 32, res // 2
    for bi, (t, c, n, s) in enumerate(settings):
        for r in range(n):
            stride = s if r == 0 else 1
            blk = MBv2Block(f"mbv2_block{bi + 1}.{r + 1}", B, hw, c_in, c_in * t, c, stride, N, rate, dtype,
                            seed=len(blocks))
            blocks.append(blk)
            c_in, hw = c, blk.hw_out
    return blocks


def block_weights(blk: MBv2Block):
    """Seeded Kaiming-normal weights and N(0, 0.1) biases of a block:
    (w_expand or None, b_expand or None, w_dw [hidden, 3, 3], b_dw,
    w_project [c_out, hidden, 1, 1], b_project), float32 numpy."""
    g = _gen(5_000_011 * (blk.seed + 1))
    def kaiming(shape, fan_in):
        return (torch.randn(shape, generator=g, dtype=torch.float32) * (2.0 / fan_in) ** 0.5).numpy()
    def small(n):
        return (torch.randn((n,), generator=g, dtype=torch.float32) * 0.1).numpy()
    we = be = None
    if blk.hidden != blk.c_in:
        we, be = kaiming((blk.hidden, blk.c_in, 1, 1), blk.c_in), small(blk.hidden)
    wd, bd = kaiming((blk.hidden, 3, 3), 9), small(blk.hidden)
    wp, bp = kaiming((blk.c_out, blk.hidden, 1, 1), blk.hidden), small(blk.c_out)
    return we, be, wd, bd, wp, bp


def block_input(blk: MBv2Block) -> torch.Tensor:
    """NHWC float32 block input, N(0, 1) (a project conv's linear output)."""
    return torch.randn((blk.B, blk.hw, blk.hw, blk.c_in), generator=_gen(9_000_013 * (blk.seed + 1)),
                       dtype=torch.float32)


def config7(B: int = 1) -> List[MBv2Block]:
    """MobileNet-V2's 17 inverted-residual blocks at batch 1 (224x224 input),
    N=4, 50%, fp32: the latency analogue of the paper's Sec. 4.3."""
    return mobilenet_v2_blocks(B=B, res=224, N=4, rate=0.5, dtype="f32")


def config3() -> List[ConvLayer]:
    return mobilenet_v2_1x1(B=128, res=224, N=4, rate=0.5, dtype="f32")


def resnet50_bottlenecks(B: int = 256, N: int = 16, rate: float = 0.7,
                         dtype: str = "bf16") -> List[ConvLayer]:
    """All bottleneck 1x1/3x3 convs and the 4 downsample 1x1 convs of ResNet-50
    (stem excluded), torchvision layout: the stride sits on the 3x3."""
    stages = [(64, 3, 1), (128, 4, 2), (256, 6, 2), (512, 3, 2)]
    layers: List[ConvLayer] = []
    c_in, hw, li = 64, 56, 0
    for si, (width, blocks, stride) in enumerate(stages):
        out = width * 4
        for bj in range(blocks):
            s = stride if bj == 0 else 1
            tag = f"r50_s{si + 1}.b{bj + 1}"
            hw_out = (hw + 2 - 3) // s + 1
            layers.append(ConvLayer(f"{tag}_1x1a", B, hw, hw, c_in, width, N=N, rate=rate,
                                    dtype=dtype, seed=li)); li += 1
            layers.append(ConvLayer(f"{tag}_3x3", B, hw, hw, width, width, 3, 3, s, 1, 1,
                                    N=N, rate=rate, dtype=dtype, seed=li)); li += 1
            layers.append(ConvLayer(f"{tag}_1x1b", B, hw_out, hw_out, width, out, N=N,
                                    rate=rate, dtype=dtype, seed=li)); li += 1
            if bj == 0:
                layers.append(ConvLayer(f"{tag}_down", B, hw, hw, c_in, out, 1, 1, s, 0, 1,
                                        N=N, rate=rate, dtype=dtype, seed=li)); li += 1
            c_in, hw = out, hw_out
    return layers


def config4() -> List[ConvLayer]:
    return resnet50_bottlenecks(B=256, N=16, rate=0.7, dtype="bf16")


def config6(B: int = 256) -> List[ConvLayer]:
    """MobileNet-V2's 1280 -> 1000 classifier as a 1x1 convolution on a 1x1
    image (the fully connected layer of Sec. 3.1's Omega when h = w = 1),
    N=4, 50%, an fp32 and a bf16 leg."""
    return [ConvLayer(f"fc_1280_1000_b{B}_{dt}", B, 1, 1, 1280, 1000, 1, 1, 1, 0, 1, N=4, rate=0.5,
                      dtype=dt, seed=0) for dt in ("f32", "bf16")]


SWEEP_N = (1, 2, 4, 8, 16, 32)
SWEEP_RATE = (0.0, 0.3, 0.5, 0.7, 0.9)


def config5(N: int = 8, rate: float = 0.5, dtype: str = "f32", seed: int = 0) -> List[ConvLayer]:
    """Sweep point on 128x14x14x512 -> 512, 3x3 s1 p1."""
    return [ConvLayer(f"cfg5_3x3_512_N{N}_r{int(round(rate * 100))}_{dtype}_s{seed}",
                      128, 14, 14, 512, 512, 3, 3, 1, 1, 1, N=N, rate=rate, dtype=dtype,
                      seed=seed)]


def dense_counterpart(layer: ConvLayer) -> ConvLayer:
    """The library's own dense path at the same shape: rate 0, N = C_out."""
    return layer.with_(N=layer.C_out, rate=0.0, name=layer.name + "_dense")
