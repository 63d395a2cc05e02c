"""Seeded synthetic inputs shaped like the LLM layers H-Scale quantizes.

This module only draws random numbers; it holds none of the method's arithmetic,
so both the CUDA path and the CPU oracle can be fed from it.  The paper calibrates
on real model weights and FineWeb activations (Sec. 3.4, Sec. 4.1), which are not
available here; these distributions stand in for them:

* weights  W: Student-t(nu=4) * sigma_w, then round(0.1% * m * n) distinct entries
  scaled by 20 (heavy-tailed LLM weights with rare large outliers);
* activations X: N(0, 1) * a_c with a per-channel magnitude a_c ~ LogNormal(0, sigma_a),
  and a few outlier channels whose a_c is scaled by 50 or 100 (the channel-energy
  spread that makes h = diag(X^T X) non-uniform); tokens are i.i.d.

Everything is generated in fp32 and rounded to bfloat16 (round-to-nearest-even).
Importing this module does not load the CUDA library.
"""
from __future__ import annotations

import dataclasses

import numpy as np
import torch

__all__ = [
    "LayerShape", "Workload", "WORKLOADS", "weight", "channel_magnitudes",
    "activation_chunk", "bf16_bits", "chunk_seed",
]


@dataclasses.dataclass(frozen=True)
class LayerShape:
    name: str
    out_features: int  # m
    in_features: int   # n (groups of 16 run along this axis)
    input_space: str   # matrices with the same input space share one h


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    layers: tuple          # LayerShape per matrix
    tokens: int            # calibration tokens per input space
    chunk_tokens: dict     # input-space width -> tokens per streamed chunk
    sigma_w: float
    sigma_a: float
    outlier_channels: int
    outlier_channel_mult: float
    window: tuple          # symmetric half-widths k (down = up = k) to run
    seed: int
    n_layers: int = 1      # decoder layers (the full-model workload repeats the block)

    def input_spaces(self):
        """Distinct (space name, width) pairs, in first-use order."""
        seen = {}
        for L in self.layers:
            seen.setdefault(L.input_space, L.in_features)
        return list(seen.items())

    def layer_seed(self, layer_index: int) -> int:
        return self.seed if self.n_layers == 1 else self.seed * 1000 + layer_index


_ATTN = "attn_in"
WORKLOADS = {
    # single linear layer, small enough for the oracle to finish in seconds
    "layer-512x1024": Workload(
        "layer-512x1024", (LayerShape("linear", 512, 1024, "x"),), tokens=2048,
        chunk_tokens={1024: 2048}, sigma_w=0.02, sigma_a=1.0, outlier_channels=8,
        outlier_channel_mult=50.0, window=(4,), seed=0),
    # Llama-style 8B attention q_proj, 262144 calibration tokens in 8192-token chunks
    "llama8b-q_proj": Workload(
        "llama8b-q_proj", (LayerShape("q_proj", 4096, 4096, _ATTN),), tokens=262144,
        chunk_tokens={4096: 8192}, sigma_w=0.02, sigma_a=1.0, outlier_channels=8,
        outlier_channel_mult=50.0, window=(4,), seed=1),
    # MLP down_proj, 262144 tokens of width 14336 (7.5 GB) in 4096-token chunks
    "mlp-down_proj": Workload(
        "mlp-down_proj", (LayerShape("down_proj", 4096, 14336, "down_in"),), tokens=262144,
        chunk_tokens={14336: 4096}, sigma_w=0.015, sigma_a=1.5, outlier_channels=32,
        outlier_channel_mult=100.0, window=(8,), seed=2),
    # full 8B-class decoder: 32 layers; q/k/v share one h, gate/up share one h
    "llama8b-decoder": Workload(
        "llama8b-decoder",
        (LayerShape("q_proj", 4096, 4096, _ATTN), LayerShape("k_proj", 1024, 4096, _ATTN),
         LayerShape("v_proj", 1024, 4096, _ATTN), LayerShape("o_proj", 4096, 4096, "o_in"),
         LayerShape("gate_proj", 14336, 4096, "mlp_in"), LayerShape("up_proj", 14336, 4096, "mlp_in"),
         LayerShape("down_proj", 4096, 14336, "down_in")),
        tokens=131072, chunk_tokens={4096: 8192, 14336: 4096}, sigma_w=0.02, sigma_a=1.5,
        outlier_channels=32, outlier_channel_mult=100.0, window=(4,), seed=3, n_layers=32),
    # 70B-class MLP block at wide shapes; k = 4 first, then the sweep k in {1, 2, 8, 16}
    "llama70b-mlp": Workload(
        "llama70b-mlp",
        (LayerShape("gate_proj", 28672, 8192, "mlp_in"), LayerShape("up_proj", 28672, 8192, "mlp_in"),
         LayerShape("down_proj", 8192, 28672, "down_in")),
        tokens=65536, chunk_tokens={8192: 4096, 28672: 2048}, sigma_w=0.015, sigma_a=1.5,
        outlier_channels=32, outlier_channel_mult=100.0, window=(4, 1, 2, 8, 16), seed=4),
}


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed) & 0x7FFFFFFFFFFFFFFF)
    return g


def chunk_seed(seed: int, stream: str, index: int) -> int:
    """A distinct, reproducible seed per (workload seed, named stream, index)."""
    h = 1469598103934665603
    for ch in f"{seed}/{stream}/{index}".encode():
        h = ((h ^ ch) * 1099511628211) & 0xFFFFFFFFFFFFFFFF
    return h & 0x7FFFFFFFFFFFFFFF


def weight(m: int, n: int, sigma: float, seed: int, device="cpu",
           outlier_frac: float = 1e-3, outlier_mult: float = 20.0) -> torch.Tensor:
    """bf16 [m, n]: Student-t(4) * sigma with round(outlier_frac*m*n) entries scaled."""
    g = _gen(chunk_seed(seed, "w", 0), device)
    z = torch.randn(m, n, generator=g, device=device)
    chi = torch.zeros(m, n, device=device)
    for _ in range(4):
        e = torch.randn(m, n, generator=g, device=device)
        chi.addcmul_(e, e)
    w = z * torch.rsqrt(chi / 4.0) * sigma
    del z, chi
    k = int(round(outlier_frac * m * n))
    if k:
        idx = torch.randperm(m * n, generator=g, device=device)[:k]
        w.view(-1)[idx] *= outlier_mult
    return w.to(torch.bfloat16)


def channel_magnitudes(n: int, sigma_a: float, outliers: int, mult: float, seed: int,
                       device="cpu") -> torch.Tensor:
    """fp32 [n]: per-channel activation magnitude a_c ~ LogNormal(0, sigma_a), with
    ``outliers`` random channels scaled by ``mult``."""
    g = _gen(chunk_seed(seed, "a", n), device)
    a = torch.exp(torch.randn(n, generator=g, device=device) * sigma_a)
    if outliers:
        idx = torch.randperm(n, generator=g, device=device)[:outliers]
        a[idx] *= mult
    return a


def activation_chunk(tokens: int, magnitudes: torch.Tensor, seed: int, index: int,
                     out: torch.Tensor | None = None) -> torch.Tensor:
    """bf16 [tokens, n] = N(0,1) * a_c for chunk ``index`` of a stream (i.i.d. tokens)."""
    device = magnitudes.device
    n = magnitudes.numel()
    g = _gen(chunk_seed(seed, "x", index), device)
    x = torch.randn(tokens, n, generator=g, device=device)
    x.mul_(magnitudes)
    if out is None:
        return x.to(torch.bfloat16)
    out.copy_(x)
    return out


def bf16_bits(t: torch.Tensor) -> np.ndarray:
    """Host numpy uint16 view of a bf16 tensor's bit patterns (copies to host)."""
    if t.dtype != torch.bfloat16:
        raise TypeError("expected a bfloat16 tensor")
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
