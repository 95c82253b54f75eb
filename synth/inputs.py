"""Seeded synthetic tensors with the shapes and value distributions of the
learned-image-coding (LIC) workloads the Hadamard-domain INT8 operator targets.

Every generator takes an explicit integer seed and uses numpy's PCG64, so the
CUDA path and the CPU oracle see identical inputs. Nothing here implements the
quantization method: the only rounding is the one that turns a drawn real
tensor into the INT8 *input* format a workload is specified in (an image in
[0, 1] stored as rint(127 x); an activation stored with a stated incoming
scale).

Distributions (stand-ins for GMM/ELIC activations and weights, which are not
available here):
  activations  x[p, c] = 0.5 + sigma_c * o_c * t,  t ~ Student-t(nu=3),
               sigma_c ~ LogNormal(0, 1), o_c = 20 on 4 channels (the first 4
               of a seeded permutation) and 1 elsewhere.
  weights      W[c, ...] = lambda_c * Laplace(0, 0.02), lambda_c ~ LogNormal(0, 0.5)
  bias         Laplace(0, 0.01)
  image        uniform [0, 1]
  latents      Laplace(0, 1) * LogNormal(0, 1) per channel
"""
from __future__ import annotations

import numpy as np


def _rng(seed: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(int(seed)))


def activations(shape, seed: int, n_outlier: int = 4, outlier_gain: float = 20.0,
                mean: float = 0.5) -> np.ndarray:
    """NHWC float32 activations: heavy-tailed, per-channel log-normal scales,
    a few outlier channels and a nonzero channel mean."""
    n, h, w, c = shape
    rng = _rng(seed)
    sigma = rng.lognormal(0.0, 1.0, size=c)
    gain = np.ones(c)
    gain[rng.permutation(c)[: min(n_outlier, c)]] = outlier_gain
    t = rng.standard_t(3.0, size=(n, h, w, c))
    x = mean + (sigma * gain) * t
    return x.astype(np.float32)


def activations_f16(shape, seed: int) -> np.ndarray:
    """The activation distribution above, stored as IEEE fp16 (the FP16 entry
    format). Values beyond the fp16 range are clipped to +-60000."""
    x = activations(shape, seed)
    return np.clip(x, -60000.0, 60000.0).astype(np.float16)


def to_int8_codes(x: np.ndarray, s_in: float) -> np.ndarray:
    """Store a real tensor as symmetric INT8 codes at a stated scale s_in
    (the INT8 input format of a workload)."""
    q = np.rint(np.asarray(x, dtype=np.float64) / float(s_in))
    return np.clip(q, -127, 127).astype(np.int8)


def activations_i8(shape, seed: int, s_in: float) -> np.ndarray:
    return to_int8_codes(activations(shape, seed), s_in)


def weights(c_out: int, kh: int, kw: int, c_in: int, seed: int) -> np.ndarray:
    """OHWI float32 conv weights with per-output-channel log-normal gain."""
    rng = _rng(seed)
    lam = rng.lognormal(0.0, 0.5, size=c_out)
    w = rng.laplace(0.0, 0.02, size=(c_out, kh, kw, c_in))
    return (w * lam[:, None, None, None]).astype(np.float32)


def bias(c_out: int, seed: int) -> np.ndarray:
    rng = _rng(seed)
    return rng.laplace(0.0, 0.01, size=c_out).astype(np.float32)


def image_i8(shape, seed: int) -> np.ndarray:
    """NHWC image uniform in [0, 1], stored as INT8 codes rint(127 x) (scale 1/127)."""
    rng = _rng(seed)
    x = rng.random(size=shape, dtype=np.float32)
    return np.rint(127.0 * x).astype(np.int8)


def latents(shape, seed: int) -> np.ndarray:
    """NHWC float32 latents: Laplace(0, 1) times a per-channel log-normal scale."""
    n, h, w, c = shape
    rng = _rng(seed)
    scale = rng.lognormal(0.0, 1.0, size=c)
    y = rng.laplace(0.0, 1.0, size=(n, h, w, c)) * scale
    return y.astype(np.float32)


def latents_i8(shape, seed: int, s_in: float) -> np.ndarray:
    return to_int8_codes(latents(shape, seed), s_in)


def uniform_codes(shape, seed: int, lo: int = -127, hi: int = 127) -> np.ndarray:
    """Uniform INT8 codes in [lo, hi] (edge-case and stress inputs)."""
    rng = _rng(seed)
    return rng.integers(lo, hi + 1, size=shape, dtype=np.int64).astype(np.int8)
