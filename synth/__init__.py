"""Seeded synthetic inputs and workload descriptions shared by the CUDA path's
tests/bench and by the CPU oracle.

This package holds no arithmetic of the quantization method itself: it draws
random tensors (activations, weights, biases, images, latents) with the shapes
and distributions of learned-image-coding workloads and describes the layer
stacks (shapes, Hadamard blocks, the static DH/WH profile mask).
"""
from . import configs, inputs  # noqa: F401
