"""Layer shapes of the benchmarked PalQuant workloads and their operation counts.

Shapes follow the networks the paper evaluates (ResNet-18/34 on 224x224 ImageNet
inputs, Sec. 5) and a MobileNetV2-shaped pointwise layer.  Operation counts follow
the paper's BitOps definition (Appendix B): for a convolution with t kernels of size
c*k*k and an h*w output, #BitOps = b_w * b_a * t * c * k * k * h * w.  Integer
operations are counted as 2 per multiply-accumulate.
"""
from __future__ import annotations

from dataclasses import dataclass, field


@dataclass(frozen=True)
class LayerShape:
    """One PalQuant layer: NHWC input [N,H,W,G*Cin_g], weights [G,Cout_g,k,k,Cin_g]."""

    N: int
    H: int
    W: int
    G: int
    Cin_g: int
    Cout_g: int
    k: int
    stride: int = 1
    pad: int = 0
    bits_a: int = 2
    bits_w: int = 2
    bits_out: int = 2
    relu: bool = True
    shuffle_kind: int = 1  # 0 none, 1 cyclic pi(g) = (g + shift) mod G, 3 explicit
    shuffle_shift: int = 1
    name: str = ""

    @property
    def Ho(self) -> int:
        return (self.H + 2 * self.pad - self.k) // self.stride + 1

    @property
    def Wo(self) -> int:
        return (self.W + 2 * self.pad - self.k) // self.stride + 1

    @property
    def macs(self) -> int:
        """Multiply-accumulates of the group convolution (all G groups)."""
        return self.N * self.Ho * self.Wo * self.G * self.Cout_g * self.k * self.k * self.Cin_g

    @property
    def int_ops(self) -> int:
        return 2 * self.macs

    @property
    def in_elems(self) -> int:
        return self.N * self.H * self.W * self.G * self.Cin_g

    @property
    def out_elems(self) -> int:
        return self.N * self.Ho * self.Wo * self.G * self.Cout_g

    @property
    def weight_elems(self) -> int:
        return self.G * self.Cout_g * self.k * self.k * self.Cin_g


# The single-layer workloads.  Activations half-normal, weights N(0, 2/fan_in),
# per-group LSQ step initialisation, cyclic shuffle across the groups, seed 0.
CONFIG0 = LayerShape(N=1, H=28, W=28, G=2, Cin_g=32, Cout_g=32, k=3, stride=1, pad=1,
                     name="3x3 layer, 1x28x28, 2 groups of 32, b=2")
CONFIG1 = LayerShape(N=64, H=56, W=56, G=4, Cin_g=64, Cout_g=64, k=3, stride=1, pad=1,
                     name="ResNet-18 stage-1 3x3 layer, 64x56x56, 4 groups of 64, b=2")
CONFIG3 = [
    LayerShape(N=128, H=28, W=28, G=G, Cin_g=512 // G, Cout_g=512 // G, k=3, stride=1, pad=1,
               bits_a=b, bits_w=b, bits_out=b, name=f"3x3 sweep b={b} G={G}, 128x28x28x512")
    for (b, G) in [(2, 2), (2, 4), (2, 8), (4, 2), (4, 4)]
]
CONFIG4 = LayerShape(N=256, H=14, W=14, G=4, Cin_g=96, Cout_g=96, k=1, stride=1, pad=0,
                     name="MobileNetV2 pointwise 1x1 layer, 256x14x14, 4 groups of 96, b=2")


def resnet18_layers(N: int = 128, G: int = 2, bits: int = 2):
    """The PalQuant layers of a ResNet-18-shaped network (per-group widths 64/128/256/512).

    Returns a list of (block_id, role, LayerShape) with role in {conv1, conv2, down}."""
    layers = []
    H = 56
    cin = 64
    for stage, width in enumerate([64, 128, 256, 512]):
        for blk in range(2):
            s = 2 if (stage > 0 and blk == 0) else 1
            Ho = H // s
            bid = f"s{stage + 1}b{blk + 1}"
            layers.append((bid, "conv1", LayerShape(N, H, H, G, cin, width, 3, s, 1, bits, bits, bits, True, 0, 0)))
            layers.append((bid, "conv2", LayerShape(N, Ho, Ho, G, width, width, 3, 1, 1, bits, bits, bits, True, 1, 1)))
            if s != 1 or cin != width:
                layers.append((bid, "down", LayerShape(N, H, H, G, cin, width, 1, s, 0, bits, bits, bits, False, 0, 0)))
            H, cin = Ho, width
    return layers


# ---------------------------------------------------------------------------
# Appendix B BitOps accounting of whole networks (used to pin the operation
# counts against Table 1).
# ---------------------------------------------------------------------------
@dataclass
class ConvCount:
    t: int
    c: int
    k: int
    h: int
    w: int

    def macs(self) -> int:
        return self.t * self.c * self.k * self.k * self.h * self.w


def resnet_convs(blocks=(2, 2, 2, 2), width_mult: int = 1, groups: int = 1, classes: int = 1000,
                 shuffle_module_stages=()):
    """Per-layer (t, c, k, h, w) of a 224x224 ResNet basic-block network.

    width_mult expands every channel count (PalQuant expands by G, Sec. 4.3); groups
    splits each body convolution into that many groups, so c counts the input channels
    one kernel sees.  The stem is a 7x7/2 conv from 3 channels and the head an FC layer.
    shuffle_module_stages lists stages (0-based) that start with a cyclic shuffle module,
    whose 1x1 group convolution is counted as well."""
    convs = [ConvCount(64 * width_mult, 3, 7, 112, 112)]
    H = 56
    cin = 64
    for stage, width in enumerate([64, 128, 256, 512]):
        for b in range(blocks[stage]):
            s = 2 if (stage > 0 and b == 0) else 1
            Ho = H // s
            convs.append(ConvCount(width * width_mult, cin * width_mult // groups, 3, Ho, Ho))
            convs.append(ConvCount(width * width_mult, width * width_mult // groups, 3, Ho, Ho))
            if s != 1:
                convs.append(ConvCount(width * width_mult, cin * width_mult // groups, 1, Ho, Ho))
            if b == 0 and stage in shuffle_module_stages:
                convs.append(ConvCount(width * width_mult, width * width_mult // groups, 1, Ho, Ho))
            H, cin = Ho, width
    convs.append(ConvCount(classes, 512 * width_mult, 1, 1, 1))
    return convs


def bitops(convs, b_w: int, b_a: int) -> int:
    """#BitOps = b_w * b_a * t * c * k * k * h * w summed over the layers (Appendix B)."""
    return sum(b_w * b_a * cv.macs() for cv in convs)


BENCH_CONFIGS = {"config0": CONFIG0, "config1": CONFIG1, "config4": CONFIG4}
for _i, _c in enumerate(CONFIG3):
    BENCH_CONFIGS[f"config3_{_i}"] = _c
