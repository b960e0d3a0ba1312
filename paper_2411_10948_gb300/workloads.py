"""Seeded synthetic inputs shaped like the paper's training workloads.

The paper trains ResNets on CIFAR10/ImageNet and Transformers (ViT, WMT14) (Sec. 5.1);
none of those datasets or weights exist here, so every tensor is synthetic, with the
shapes of those layers and the channel structure the paper describes for gradients
(Sec. 3.1: a few channels with far wider range than the rest).  This module holds no
quantizer arithmetic: only random numbers.

Two backends draw from the same recipe: numpy (bit-reproducible on any host; the parity
tests feed it to both the oracle and the GPU) and torch on the device (fast; the
benchmark, which compares nothing).
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

# ----------------------------------------------------------------------- recipes
# act:  ("halfnormal",)                         |N(0,1)|  (post-ReLU)
#       ("normal_outlier", frac, factor)        N(0,1), a fraction of channels x factor
# grad: ("grad", base, sigma, frac, factor)     base(0,1) x per-channel lognormal(0, sigma),
#                                               a fraction of channels x factor
#                                               (base "normal" or "laplace")
# weight: ("weight", std)                       N(0, std)


@dataclass(frozen=True)
class LayerSpec:
    name: str
    M: int            # tokens (or im2col rows)
    K: int            # in-channels
    N: int            # out-channels
    bits: int
    n_groups: int
    act: tuple
    grad: tuple
    weight: tuple = ("weight", 0.02)


@dataclass
class Workload:
    name: str
    description: str
    layers: list = field(default_factory=list)

    @property
    def gemm_ops(self) -> int:
        return sum(3 * 2 * l.M * l.N * l.K for l in self.layers)


C3_ACT = ("normal_outlier", 0.02, 50.0)
C3_GRAD = ("grad", "laplace", 2.0, 0.0, 1.0)


def workload(name: str) -> Workload:
    """The workloads: wgrad_small, conv3x3, vit_mlp, large_linear(_8bit), vit_block, and
    large_linear_t4096 (large_linear's layers on 4096 tokens: a profiling-size case of the
    same kernels)."""
    if name == "wgrad_small":
        g = ("grad", "normal", 1.5, 0.01, 100.0)
        return Workload(name, "4-bit wgrad/dgrad, dY and X [256, 512], W [512, 512]",
                        [LayerSpec("l0", 256, 512, 512, 4, 4, ("grad", "normal", 1.5, 0.01, 100.0),
                                   g)])
    if name == "conv3x3":
        return Workload(name, "ResNet 3x3 conv 256->256 as im2col GEMMs, batch 64, 14x14, 4-bit",
                        [LayerSpec("conv", 64 * 14 * 14, 256 * 9, 256, 4, 4, ("halfnormal",),
                                   ("grad", "normal", 2.0, 0.005, 1000.0))])
    if name == "vit_mlp":
        M = 64 * 197
        return Workload(name, "ViT-B MLP fc1 768->3072 and fc2 3072->768, 12608 tokens, 6-bit",
                        [LayerSpec("fc1", M, 768, 3072, 6, 4, C3_ACT, C3_GRAD),
                         LayerSpec("fc2", M, 3072, 768, 6, 4, C3_ACT, C3_GRAD)])
    if name in ("large_linear", "large_linear_8bit", "large_linear_t4096"):
        bits = 8 if name.endswith("8bit") else 6
        T = 4096 if name.endswith("t4096") else 16384
        g = ("grad", "laplace", 2.5, 0.001, 1.0e4)
        return Workload(name, f"{T} tokens, 4096->11008 and 11008->4096, {bits}-bit",
                        [LayerSpec("up", T, 4096, 11008, bits, 4, C3_ACT, g),
                         LayerSpec("down", T, 11008, 4096, bits, 4, C3_ACT, g)])
    if name == "vit_block":
        M = 64 * 197
        return Workload(name, "ViT-B/16 block (QKV, proj, fc1, fc2), batch 64 x 197 tokens, 6-bit",
                        [LayerSpec("qkv", M, 768, 2304, 6, 4, C3_ACT, C3_GRAD),
                         LayerSpec("proj", M, 768, 768, 6, 4, C3_ACT, C3_GRAD),
                         LayerSpec("fc1", M, 768, 3072, 6, 4, C3_ACT, C3_GRAD),
                         LayerSpec("fc2", M, 3072, 768, 6, 4, C3_ACT, C3_GRAD)])
    raise KeyError(name)


WORKLOADS = ("wgrad_small", "conv3x3", "vit_mlp", "large_linear", "large_linear_8bit",
             "vit_block", "large_linear_t4096")


def tensor_seed(seed: int, layer_idx: int, which: str) -> int:
    return (seed * 1_000_003 + layer_idx * 97 + {"x": 1, "w": 2, "dy": 3}[which]) & 0x7FFFFFFF


# ------------------------------------------------------------------ numpy backend
def _np_channel_factor(rng, C, sigma, frac, factor):
    f = np.exp(rng.normal(0.0, sigma, C)).astype(np.float32)
    if frac > 0:
        n = max(1, int(round(frac * C)))
        idx = rng.choice(C, n, replace=False)
        f[idx] *= np.float32(factor)
    return f


def np_tensor(recipe: tuple, rows: int, cols: int, seed: int) -> np.ndarray:
    rng = np.random.default_rng(seed)
    kind = recipe[0]
    if kind == "halfnormal":
        return np.abs(rng.standard_normal((rows, cols), dtype=np.float32))
    if kind == "normal_outlier":
        _, frac, factor = recipe
        x = rng.standard_normal((rows, cols), dtype=np.float32)
        n = max(1, int(round(frac * cols)))
        x[:, rng.choice(cols, n, replace=False)] *= np.float32(factor)
        return x
    if kind == "grad":
        _, base, sigma, frac, factor = recipe
        if base == "normal":
            x = rng.standard_normal((rows, cols), dtype=np.float32)
        else:  # Laplace(0, 1) as a random sign times Exp(1)
            x = rng.standard_exponential((rows, cols), dtype=np.float32)
            x *= np.where(rng.integers(0, 2, (rows, cols), dtype=np.int8) == 0, -1, 1).astype(
                np.float32)
        x *= _np_channel_factor(rng, cols, sigma, frac, factor)[None, :]
        return x
    if kind == "weight":
        return rng.standard_normal((rows, cols), dtype=np.float32) * np.float32(recipe[1])
    raise KeyError(kind)


def np_layer_inputs(spec: LayerSpec, seed: int = 0, layer_idx: int = 0, rows: int | None = None):
    """x [M, K], w [K, N], dy [M, N] as float32 numpy arrays (rows overrides M)."""
    M = spec.M if rows is None else rows
    x = np_tensor(spec.act, M, spec.K, tensor_seed(seed, layer_idx, "x"))
    w = np_tensor(spec.weight, spec.K, spec.N, tensor_seed(seed, layer_idx, "w"))
    dy = np_tensor(spec.grad, M, spec.N, tensor_seed(seed, layer_idx, "dy"))
    return x, w, dy


# ------------------------------------------------------------------ torch backend
def torch_tensor(recipe: tuple, rows: int, cols: int, seed: int, device="cuda"):
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    kind = recipe[0]
    if kind == "halfnormal":
        return torch.randn((rows, cols), generator=g, device=device).abs_()
    if kind == "normal_outlier":
        _, frac, factor = recipe
        x = torch.randn((rows, cols), generator=g, device=device)
        n = max(1, int(round(frac * cols)))
        idx = torch.randperm(cols, generator=g, device=device)[:n]
        x[:, idx] *= factor
        return x
    if kind == "grad":
        _, base, sigma, frac, factor = recipe
        if base == "normal":
            x = torch.randn((rows, cols), generator=g, device=device)
        else:
            x = torch.empty((rows, cols), device=device).exponential_(1.0, generator=g)
            sign = torch.randint(0, 2, (rows, cols), generator=g, device=device, dtype=torch.int8)
            x *= sign.to(torch.float32).mul_(2).sub_(1)
        f = torch.randn(cols, generator=g, device=device).mul_(sigma).exp_()
        if frac > 0:
            n = max(1, int(round(frac * cols)))
            f[torch.randperm(cols, generator=g, device=device)[:n]] *= factor
        x *= f[None, :]
        return x
    if kind == "weight":
        return torch.randn((rows, cols), generator=g, device=device).mul_(recipe[1])
    raise KeyError(kind)


def torch_layer_inputs(spec: LayerSpec, seed: int = 0, layer_idx: int = 0, device="cuda"):
    x = torch_tensor(spec.act, spec.M, spec.K, tensor_seed(seed, layer_idx, "x"), device)
    w = torch_tensor(spec.weight, spec.K, spec.N, tensor_seed(seed, layer_idx, "w"), device)
    dy = torch_tensor(spec.grad, spec.M, spec.N, tensor_seed(seed, layer_idx, "dy"), device)
    return x, w, dy
