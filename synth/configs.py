"""Workload descriptions: the five layer/stack configurations, their Hadamard
blocks and the static per-layer DH/WH profile mask.

A *chain* is a sequence of convolutions applied one after another; a *config*
is a list of chains that share nothing but the GPU. Shapes are NHWC, weights
OHWI. Nothing here computes any part of the quantization method; the only
structural rule is which input-side transform each layer's transition applies
(`plan_chain`, read off Table integer_transitions for the CUDA path; the
oracle derives the same from the layers on its own).
"""
from __future__ import annotations

from dataclasses import dataclass, field, replace

import numpy as np

DH = "DH"
WH = "WH"


def hadamard_block(c: int) -> int:
    """Block size of the block-diagonal Sylvester transform used along a channel
    axis of width c: the largest power of two dividing c, capped at 128
    (128 -> 128, 192 -> 64, 320 -> 64, 640 -> 128, 224 -> 32, 32 -> 32)."""
    b = c & (-c)
    return int(min(128, b))


@dataclass(frozen=True)
class LayerSpec:
    name: str
    c_in: int
    c_out: int
    k: int
    stride: int
    pad: int
    form: str            # DH or WH
    act: str             # "relu" or "none"
    hb_in: int = 0       # DH: block along c_in
    hb_out: int = 0      # WH: block along c_out

    def out_hw(self, h: int, w: int):
        ho = (h + 2 * self.pad - self.k) // self.stride + 1
        wo = (w + 2 * self.pad - self.k) // self.stride + 1
        return ho, wo

    def macs(self, n: int, h: int, w: int) -> int:
        ho, wo = self.out_hw(h, w)
        return n * ho * wo * self.c_out * self.c_in * self.k * self.k


def layer(name, c_in, c_out, k, stride, pad, form, act, hb_in=None, hb_out=None):
    if form == DH:
        hb_in = hadamard_block(c_in) if hb_in is None else hb_in
        hb_out = 0
    else:
        hb_out = hadamard_block(c_out) if hb_out is None else hb_out
        hb_in = 0
    return LayerSpec(name, c_in, c_out, k, stride, pad, form, act, hb_in, hb_out)


@dataclass(frozen=True)
class ChainSpec:
    name: str
    layers: tuple
    n: int
    h: int
    w: int
    input_kind: str      # "f16" (real values in fp16) or "i8" (INT8 codes at s_in)
    s_in: float          # scale of the INT8 input codes (ignored for f16)
    input_seed: int
    weight_seed: int     # layer l uses weight_seed + l for W, +50 + l for the bias
    input_gen: str = "activations"   # activations | image | latents
    out_f32: bool = False            # last layer emits dequantized float32

    def with_batch(self, n, h, w, input_seed):
        return replace(self, n=n, h=h, w=w, input_seed=input_seed)

    def shapes(self):
        """Per layer: (n, h, w) of its input."""
        out = []
        h, w = self.h, self.w
        for L in self.layers:
            out.append((self.n, h, w))
            h, w = L.out_hw(h, w)
        return out

    def macs(self):
        return sum(L.macs(*s) for L, s in zip(self.layers, self.shapes()))


@dataclass(frozen=True)
class ConfigSpec:
    name: str
    description: str
    chains: tuple
    images: int          # images per pass (for images/s)
    calib_from: str = ""  # scales are taken from this config's calibration


def plan_chain(chain: ChainSpec):
    """Per layer l, the block of the next layer's DH input transform that layer
    l's epilogue applies after phi (0 = none: the next layer is WH, or l is
    the last layer). Table integer_transitions: DH-to-DH and WH-to-DH apply
    H_in,l+1; DH-to-WH and WH-to-WH do not. The transition is always fused
    into the producer, so every layer boundary inside a chain is one
    requantization."""
    L = chain.layers
    return [L[i + 1].hb_in if i + 1 < len(L) and L[i + 1].form == DH else 0 for i in range(len(L))]


def _cfg0():
    ch = ChainSpec(
        name="dh1x1_128", n=1, h=16, w=16, input_kind="f16", s_in=1.0,
        input_seed=0, weight_seed=0, input_gen="activations", out_f32=True,
        layers=(layer("conv", 128, 128, 1, 1, 0, DH, "none", hb_in=128),))
    return ConfigSpec("cfg0", "single DH 1x1 conv 128->128 on 1x16x16 fp16", (ch,), images=1)


def _cfg1():
    ch = ChainSpec(
        name="dh5x5s2_192", n=1, h=256, w=256, input_kind="i8", s_in=0.05,
        input_seed=1, weight_seed=1000, input_gen="activations",
        layers=(layer("conv", 192, 192, 5, 2, 2, DH, "none", hb_in=64),))
    return ConfigSpec("cfg1", "one 5x5 s2 DH conv 192->192 on 1x256x256 int8", (ch,), images=1)


def analysis_chain(n, h, w, input_seed):
    return ChainSpec(
        name="analysis", n=n, h=h, w=w, input_kind="i8", s_in=1.0 / 127.0,
        input_seed=input_seed, weight_seed=2000, input_gen="image",
        layers=(
            layer("ga1", 3, 192, 5, 2, 2, WH, "relu"),
            layer("ga2", 192, 192, 5, 2, 2, DH, "relu"),
            layer("ga3", 192, 192, 5, 2, 2, DH, "relu"),
            layer("ga4", 192, 320, 5, 2, 2, DH, "none"),
        ))


def _cfg2():
    return ConfigSpec("cfg2", "analysis stack 3->192->192->192->320 (5x5 s2) on 1x768x512 image",
                      (analysis_chain(1, 768, 512, 2),), images=1)


CFG3_WH_FRACTION = 0.3
CFG3_MASK_SEED = 3


def cfg3_mask(n_layers: int = 27):
    """Seeded 30% weight-only mask over the 27 hyperprior/context layers."""
    rng = np.random.Generator(np.random.PCG64(CFG3_MASK_SEED))
    u = rng.random(n_layers)
    return [WH if x < CFG3_WH_FRACTION else DH for x in u]


def entropy_chains(n, h, w, input_seed):
    mask = cfg3_mask()
    forms = iter(mask)
    hyper = ChainSpec(
        name="hyper", n=n, h=h, w=w, input_kind="i8", s_in=0.1,
        input_seed=input_seed, weight_seed=3000, input_gen="latents",
        layers=(
            layer("h1", 320, 640, 3, 1, 1, next(forms), "relu"),
            layer("h2", 640, 640, 3, 1, 1, next(forms), "relu"),
            layer("h3", 640, 640, 1, 1, 0, next(forms), "none"),
        ))
    chains = [hyper]
    for k in range(8):
        chains.append(ChainSpec(
            name=f"slice{k}", n=n, h=h, w=w, input_kind="i8", s_in=0.1,
            input_seed=input_seed * 10 + k + 1, weight_seed=3100 + 100 * k, input_gen="latents",
            layers=(
                layer(f"s{k}a", 32, 224, 3, 1, 1, next(forms), "relu"),
                layer(f"s{k}b", 224, 128, 3, 1, 1, next(forms), "relu"),
                layer(f"s{k}c", 128, 32, 3, 1, 1, next(forms), "none"),
            )))
    return tuple(chains)


def _cfg3():
    return ConfigSpec("cfg3", "hyperprior 320->640->640->640 + 8 context slices 32->224->128->32 on 1x48x32 latent",
                      entropy_chains(1, 48, 32, 3), images=1)


def _cfg4():
    chains = (analysis_chain(8, 2160, 3840, 4),) + entropy_chains(8, 135, 240, 4)
    return ConfigSpec("cfg4", "cfg2 and cfg3 chains at batch 8 on 3840x2160 (latent 240x135)",
                      chains, images=8, calib_from="cfg2+cfg3")


CONFIGS = {c.name: c for c in (_cfg0(), _cfg1(), _cfg2(), _cfg3(), _cfg4())}


def chain_input(chain: ChainSpec) -> np.ndarray:
    """The seeded input of a chain in its stored format (fp16 values or INT8 codes)."""
    from . import inputs
    shape = (chain.n, chain.h, chain.w, chain.layers[0].c_in)
    if chain.input_kind == "f16":
        return inputs.activations_f16(shape, chain.input_seed)
    if chain.input_gen == "image":
        return inputs.image_i8(shape, chain.input_seed)
    if chain.input_gen == "latents":
        return inputs.latents_i8(shape, chain.input_seed, chain.s_in)
    return inputs.activations_i8(shape, chain.input_seed, chain.s_in)


def chain_params(chain: ChainSpec):
    """Per layer: (OHWI float32 weights, float32 bias)."""
    from . import inputs
    out = []
    for i, L in enumerate(chain.layers):
        w = inputs.weights(L.c_out, L.k, L.k, L.c_in, chain.weight_seed + i)
        b = inputs.bias(L.c_out, chain.weight_seed + 50 + i)
        out.append((w, b))
    return out
