"""Seeded synthetic inputs shared by the tests, the smoke check and the benchmark.

This module holds no Log_bQuant arithmetic: it draws weights, activations
and per-layer bases, and lists the layer shapes of the workloads.

Weights stand in for the bell-shaped, heavy-tailed weight histograms the
paper shows (Fig. 1): i.i.d. Student-t with 4 degrees of freedom scaled by
0.02, optionally with 0.1 % of the entries (distinct positions drawn
uniformly) multiplied by 20 as outliers.  A Student-t(4) draw is made from
five standard normals, Z / sqrt((Z1^2 + Z2^2 + Z3^2 + Z4^2) / 4), so the same
recipe runs with numpy on the host and with torch on a CUDA device.
Activations are standard normal in bf16 or fp16.  Seeds follow
seed = cfg_seed * 1000 + layer * 10 + projection index.
"""
from __future__ import annotations

import numpy as np

# Projection order of one transformer layer: q, k, v, o, gate, up, down.
PROJ_NAMES = ("q", "k", "v", "o", "gate", "up", "down")

# (out, in) = (N, K) of each projection, PyTorch nn.Linear layout.
LLAMA_1B_SHAPES = {
    "q": (2048, 2048), "k": (512, 2048), "v": (512, 2048), "o": (2048, 2048),
    "gate": (8192, 2048), "up": (8192, 2048), "down": (2048, 8192),
}
LLAMA_8B_SHAPES = {
    "q": (4096, 4096), "k": (1024, 4096), "v": (1024, 4096), "o": (4096, 4096),
    "gate": (14336, 4096), "up": (14336, 4096), "down": (4096, 14336),
}
LLAMA_1B_LAYERS = 16
LLAMA_8B_LAYERS = 32

SINGLE_LAYER_SHAPE = (512, 2048)       # the single-layer quantize + GEMV case
STUDENT_DF = 4
WEIGHT_SCALE = 0.02
OUTLIER_FRACTION = 1e-3
OUTLIER_FACTOR = 20.0


def layer_seed(cfg_seed: int, layer: int, proj: int) -> int:
    return cfg_seed * 1000 + layer * 10 + proj


# ---------------------------------------------------------------- numpy ---

def weights_np(N: int, K: int, seed: int, outliers: bool = False) -> np.ndarray:
    """Student-t(4) * 0.02 fp32 weights [N, K] drawn with numpy PCG64."""
    rng = np.random.Generator(np.random.PCG64(seed))
    z = rng.standard_normal((N, K))
    chi = np.zeros((N, K))
    for _ in range(STUDENT_DF):
        chi += rng.standard_normal((N, K)) ** 2
    w = z / np.sqrt(chi / STUDENT_DF) * WEIGHT_SCALE
    if outliers:
        count = int(OUTLIER_FRACTION * N * K)
        idx = rng.choice(N * K, size=count, replace=False)
        w.reshape(-1)[idx] *= OUTLIER_FACTOR
    return w.astype(np.float32)


def activations_np(B: int, K: int, seed: int) -> np.ndarray:
    """N(0, 1) activations [B, K] in fp64 (callers round them to bf16/fp16)."""
    rng = np.random.Generator(np.random.PCG64(seed + 7_000_000))
    return rng.standard_normal((B, K))


def layer_bases(n_layers: int, seed: int, lo: float = 1.2, hi: float = 2.0) -> np.ndarray:
    """Per-layer Log_b bases drawn from U[lo, hi]."""
    rng = np.random.Generator(np.random.PCG64(seed + 9_000_000))
    return rng.uniform(lo, hi, size=n_layers)


# ---------------------------------------------------------------- torch ---

def weights_torch(N: int, K: int, seed: int, outliers: bool = False, device="cpu"):
    """The same recipe as weights_np, drawn with a seeded torch generator on
    ``device`` (fast for the large layers; not bit-identical to numpy)."""
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    z = torch.randn((N, K), generator=g, device=device, dtype=torch.float32)
    chi = torch.zeros((N, K), device=device, dtype=torch.float32)
    for _ in range(STUDENT_DF):
        e = torch.randn((N, K), generator=g, device=device, dtype=torch.float32)
        chi.addcmul_(e, e)
        del e
    w = z.div_(chi.div_(STUDENT_DF).sqrt_()).mul_(WEIGHT_SCALE)
    del chi
    if outliers:
        count = int(OUTLIER_FRACTION * N * K)
        idx = torch.randperm(N * K, generator=g, device=device)[:count]
        w.view(-1)[idx] *= OUTLIER_FACTOR
    return w


def activations_torch(B: int, K: int, seed: int, dtype=None, device="cpu"):
    import torch
    dtype = dtype or torch.bfloat16
    g = torch.Generator(device=device)
    g.manual_seed(seed + 7_000_000)
    return torch.randn((B, K), generator=g, device=device, dtype=torch.float32).to(dtype)
