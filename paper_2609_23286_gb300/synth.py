"""Seeded synthetic VGGT-shaped Q/K/V streams.

This module only draws inputs; it holds none of the method's arithmetic and is
shared by the tests, the oracle comparisons and the benchmark.

Recipe (stands in for the real activations of a StreamVGGT-style aggregator,
whose weights and datasets are not available):

* Q, K, V elements are i.i.d. N(0, 1), drawn per (layer, frame).
* Every K row is multiplied by a per-token-position factor
  sigma_{l,p} ~ LogNormal(0, 0.5), drawn once per (layer, token position) and
  shared by all heads and all frames.  Keys at the same position therefore
  stay salient over time, the synthetic analogue of the temporally consistent
  token saliency the paper observes.
* Everything is rounded to bfloat16 (round to nearest even, torch's cast).
* Seeds: layer seed = splitmix64(seed ^ layer); frame seed = splitmix64(layer
  seed + frame).  Generation uses torch.Generator on the requested device, so a
  CPU stream and a CUDA stream with the same seed differ; every comparison
  feeds the oracle the exact bf16 tensors the GPU saw.
"""
from __future__ import annotations

import torch

_MASK = (1 << 64) - 1


def splitmix64(x: int) -> int:
    """SplitMix64 finaliser (Steele, Lea, Flood 2014), used to derive seeds."""
    x = (x + 0x9E3779B97F4A7C15) & _MASK
    x = ((x ^ (x >> 30)) * 0xBF58476D1CE4E5B9) & _MASK
    x = ((x ^ (x >> 27)) * 0x94D049BB133111EB) & _MASK
    return x ^ (x >> 31)


def layer_seed(seed: int, layer: int) -> int:
    return splitmix64((seed ^ layer) & _MASK)


def frame_seed(seed: int, layer: int, frame: int) -> int:
    return splitmix64((layer_seed(seed, layer) + frame) & _MASK)


def _gen(device, s: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(s & ((1 << 63) - 1))
    return g


def key_scale(seed: int, layer: int, n_tokens: int, sigma: float = 0.5,
              device="cpu") -> torch.Tensor:
    """Per-token-position key-norm factor for one layer, [n_tokens] float32."""
    g = _gen(device, splitmix64(layer_seed(seed, layer) ^ 0x5CA1E))
    z = torch.randn(n_tokens, generator=g, device=device, dtype=torch.float32)
    return torch.exp(sigma * z)


def frame_qkv(seed: int, layer: int, frame: int, n_tokens: int, heads: int,
              head_dim: int, device="cpu", sigma: float = 0.5, scale_cache=None):
    """Q, K, V of one (layer, frame): three [n_tokens, heads, head_dim] bf16
    tensors on ``device``."""
    g = _gen(device, frame_seed(seed, layer, frame))
    shape = (3, n_tokens, heads, head_dim)
    x = torch.randn(shape, generator=g, device=device, dtype=torch.float32)
    ks = scale_cache if scale_cache is not None else key_scale(seed, layer, n_tokens, sigma, device)
    x[1] *= ks.view(n_tokens, 1, 1)
    x = x.to(torch.bfloat16)
    return x[0].contiguous(), x[1].contiguous(), x[2].contiguous()
