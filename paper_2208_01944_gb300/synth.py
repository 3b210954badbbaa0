"""Seeded synthetic inputs for PalQuant layers (no quantisation arithmetic here).

The paper evaluates on ImageNet-trained ResNet-18/34 (Sec. 5); no dataset or trained
weights are used here.  Inputs take the shapes of those networks and the value
distributions of a freshly initialised network:

* activations entering a quantised layer follow a ReLU, so they are drawn as
  half-normal |N(0, 1)|;
* network inputs (images) are N(0, 1);
* weights are N(0, 2 / fan_in) with fan_in = Cin_g * kh * kw (He initialisation of a
  grouped convolution).

Every tensor is drawn as fp32 from one ``torch.Generator`` seeded with ``seed`` on
the CPU, in a fixed order (activations first, then weights), and returned as numpy
arrays in the library's layouts: activations NHWC, weights [G, Cout_g, kh, kw, Cin_g].
Both the GPU path and the CPU oracle receive these same arrays.
"""
from __future__ import annotations

import math

import numpy as np
import torch


def generator(seed: int = 0) -> torch.Generator:
    return torch.Generator().manual_seed(int(seed))


def half_normal(shape, gen: torch.Generator) -> np.ndarray:
    return torch.randn(tuple(shape), generator=gen, dtype=torch.float32).abs_().numpy()


def normal(shape, gen: torch.Generator, std: float = 1.0) -> np.ndarray:
    t = torch.randn(tuple(shape), generator=gen, dtype=torch.float32)
    if std != 1.0:
        t.mul_(std)
    return t.numpy()


def he_weights(G: int, Cout_g: int, kh: int, kw: int, Cin_g: int, gen: torch.Generator) -> np.ndarray:
    return normal((G, Cout_g, kh, kw, Cin_g), gen, math.sqrt(2.0 / (Cin_g * kh * kw)))


def layer_inputs(N: int, H: int, W: int, G: int, Cin_g: int, Cout_g: int, k: int, seed: int = 0):
    """(x, w): half-normal NHWC activations and He-initialised grouped weights."""
    gen = generator(seed)
    x = half_normal((N, H, W, G * Cin_g), gen)
    w = he_weights(G, Cout_g, k, k, Cin_g, gen)
    return x, w


def random_codes(shape, bits: int, gen: torch.Generator, signed: bool = False) -> np.ndarray:
    """Uniform random integer codes (unsigned [0, 2^b-1] or signed [-2^(b-1), 2^(b-1)-1])."""
    if signed:
        lo, hi = -(1 << (bits - 1)), (1 << (bits - 1))
        return torch.randint(lo, hi, tuple(shape), generator=gen, dtype=torch.int16).numpy().astype(np.int8)
    return torch.randint(0, 1 << bits, tuple(shape), generator=gen, dtype=torch.int16).numpy().astype(np.uint8)


def resnet18_inputs(N: int, H: int = 224, W: int = 224, G: int = 2, widths=(64, 128, 256, 512), classes: int = 1000,
                    seed: int = 0, cyclic_modules: bool = False):
    """(x, params) for the ResNet-18-shaped PalQuant network.

    x: images N(0, 1), NHWC [N, H, W, 3].  params: name -> fp32 weights, drawn after x
    in this order: "stem" [G*widths[0], 7, 7, 3] N(0, 2/147); then for stage s = 1..4
    and block b = 1, 2: "s{s}b{b}.conv1" [G, w, 3, 3, cin], "s{s}b{b}.conv2"
    [G, w, 3, 3, w] and, in the first block of stages 2-4 (stride 2, channels change),
    "s{s}b{b}.down" [G, w, 1, 1, cin], all He-initialised per group (w = widths[s-1],
    cin = the block's per-group input width); last "fc" [classes, G*widths[-1]]
    N(0, 1/fan_in).  With cyclic_modules, then per stage k = 1..4 "s{k}.csm"
    [G, c, 1, 1, c] (the weights of the cyclic shuffle module at the stage's
    beginning, c = the stage's per-group input width), He-initialised."""
    gen = generator(seed)
    x = normal((N, H, W, 3), gen)
    params = {"stem": normal((G * widths[0], 7, 7, 3), gen, math.sqrt(2.0 / 147.0))}
    cin = widths[0]
    for s, w in enumerate(widths):
        for b in range(2):
            name = f"s{s + 1}b{b + 1}"
            params[name + ".conv1"] = he_weights(G, w, 3, 3, cin, gen)
            params[name + ".conv2"] = he_weights(G, w, 3, 3, w, gen)
            if s > 0 and b == 0:
                params[name + ".down"] = he_weights(G, w, 1, 1, cin, gen)
            cin = w
    params["fc"] = normal((classes, G * widths[-1]), gen, math.sqrt(1.0 / (G * widths[-1])))
    if cyclic_modules:
        cin = widths[0]
        for s, w in enumerate(widths):
            params[f"s{s + 1}.csm"] = he_weights(G, cin, 1, 1, cin, gen)
            cin = w
    return x, params
