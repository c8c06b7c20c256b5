"""Seeded synthetic inputs for the grouped ternary linear layer.

This module only draws random numbers and reshapes them. It holds none of the
method's arithmetic (no scale, no rounding to codes, no packing, no products),
so both the CUDA path and the oracle can take their inputs from here.

Distributions follow the workloads of the paper's Mamba-2 1.3B projections
(§3.1 for the layer, Table 13 and §8 for the shapes):

* latent weights ``W`` fp32 ``[N, K]`` drawn from N(0, 0.02^2), or from a
  Student-t with 3 degrees of freedom rescaled to the same standard deviation
  (heavier tails, so more groups with a large absmean outlier);
* activations ``X`` and upstream gradients ``dY`` as bf16, from N(0, std^2).

Every array is a pure function of ``(seed, stream)``: ``stream`` names what the
array is ("w", "x", "dy"), so changing one input never shifts another.
"""
from __future__ import annotations

import zlib

import numpy as np
import torch

__all__ = [
    "rng",
    "latent_weights",
    "activations_bf16",
    "activations_f16",
    "MAMBA2_1P3B",
]

# Mamba-2 1.3B projection shapes (out_features N, in_features K); 48 blocks.
MAMBA2_1P3B = {
    "in_proj": (8512, 2048),
    "out_proj": (2048, 4096),
    "n_layers": 48,
}


def rng(seed: int, stream: str) -> np.random.Generator:
    """PCG64 generator for ``(seed, stream)``; independent across streams."""
    tag = zlib.crc32(stream.encode("utf-8"))
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([int(seed), tag])))


def latent_weights(n: int, k: int, seed: int, dist: str = "gauss", std: float = 0.02,
                   stream: str = "w") -> np.ndarray:
    """fp32 ``[n, k]`` latent weights.

    ``dist="gauss"``: N(0, std^2). ``dist="t3"``: Student-t(3) scaled by
    ``std / sqrt(3)`` so that its standard deviation is ``std``.
    """
    g = rng(seed, stream)
    if dist == "gauss":
        w = g.standard_normal((n, k), dtype=np.float32) * np.float32(std)
    elif dist == "t3":
        w = (g.standard_t(3.0, size=(n, k)) * (std / np.sqrt(3.0))).astype(np.float32)
    else:
        raise ValueError(f"unknown weight distribution {dist!r}")
    return np.ascontiguousarray(w)


def activations_f16(m: int, k: int, seed: int, std: float = 1.0, stream: str = "x") -> torch.Tensor:
    """fp16 CPU tensor ``[m, k]``: the draw of :func:`activations_bf16`, rounded to fp16."""
    g = rng(seed, stream)
    a = g.standard_normal((m, k), dtype=np.float32)
    if std != 1.0:
        a *= np.float32(std)
    return torch.from_numpy(a).to(torch.float16).contiguous()


def activations_bf16(m: int, k: int, seed: int, std: float = 1.0, stream: str = "x") -> torch.Tensor:
    """bf16 CPU tensor ``[m, k]`` from N(0, std^2) (fp32 draw, rounded to bf16)."""
    g = rng(seed, stream)
    a = g.standard_normal((m, k), dtype=np.float32)
    if std != 1.0:
        a *= np.float32(std)
    return torch.from_numpy(a).to(torch.bfloat16).contiguous()
