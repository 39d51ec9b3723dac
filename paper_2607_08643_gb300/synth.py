"""Seeded synthetic inputs shaped like the paper's workloads.

This module only draws random numbers and rounds them to bf16 bit patterns;
it holds none of the coding method's arithmetic, so both the CUDA path's
tests/benchmark and the CPU oracle's tests can take their inputs from it.

Workload recipe (Qwen3-8B linear shapes; the paper evaluates real Qwen3-8B
and LLaMA checkpoints, which these synthetic layers stand in for):

* weights: N(0, 0.02) (or unit-variance Student-t(4) scaled to std 0.02),
  drawn in float64 from ``numpy.random.default_rng(seed)``, plus 8 outlier
  input columns (chosen by the same generator, without replacement) scaled
  by 20, then rounded to float32 and to bf16 (round to nearest even);
* activations: N(0, 1) rounded the same way;
* protected count p = ceil(rho * K) computed exactly from rho in percent.
"""
from __future__ import annotations

import numpy as np

HIDDEN, FFN, N_LAYERS = 4096, 12288, 36

# name -> (N = out features, K = in features)
QWEN3_8B_SHAPES = {
    "q_proj": (4096, 4096),
    "k_proj": (1024, 4096),
    "v_proj": (1024, 4096),
    "o_proj": (4096, 4096),
    "gate_proj": (12288, 4096),
    "up_proj": (12288, 4096),
    "down_proj": (4096, 12288),
}
ATTN = ("q_proj", "k_proj", "v_proj", "o_proj")
MLP = ("gate_proj", "up_proj", "down_proj")


def protected_count(K: int, rho_percent: float) -> int:
    """ceil(rho * K) with rho given in percent, in exact integer arithmetic."""
    num = int(round(rho_percent * 1000))          # rho in units of 1e-5
    return (num * K + 100000 - 1) // 100000


def f32_to_bf16_bits(a) -> np.ndarray:
    """Round float32 values to bf16 (nearest even); returns uint16 bits."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32).astype(np.uint64)
    nan = np.isnan(np.asarray(a, dtype=np.float32))
    r = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    r = r.astype(np.uint16)
    r[nan] = 0x7FC0
    return r


def bf16_bits_to_f32(b) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def layer_weights(N: int, K: int, seed: int, dist: str = "normal", sigma: float = 0.02,
                  n_outliers: int = 8, outlier_scale: float = 20.0) -> np.ndarray:
    """bf16 bits uint16[N][K] of one synthetic linear layer (row = out feature)."""
    rng = np.random.default_rng(seed)
    if dist == "normal":
        w = rng.standard_normal((N, K)) * sigma
    elif dist == "t4":
        w = rng.standard_t(4.0, size=(N, K)) / np.sqrt(2.0) * sigma
    else:
        raise ValueError(dist)
    if n_outliers:
        cols = rng.choice(K, size=min(n_outliers, K), replace=False)
        w[:, cols] *= outlier_scale
    return f32_to_bf16_bits(w.astype(np.float32))


def outlier_columns(K: int, seed: int, dist: str = "normal", N: int = 1,
                    n_outliers: int = 8) -> np.ndarray:
    """The outlier columns :func:`layer_weights` picks for the same arguments."""
    rng = np.random.default_rng(seed)
    if dist == "normal":
        rng.standard_normal((N, K))
    else:
        rng.standard_t(4.0, size=(N, K))
    return np.sort(rng.choice(K, size=min(n_outliers, K), replace=False))


def activations(B: int, K: int, seed: int, scale: float = 1.0) -> np.ndarray:
    """bf16 bits uint16[B][K], N(0, scale^2)."""
    rng = np.random.default_rng(seed)
    return f32_to_bf16_bits((rng.standard_normal((B, K)) * scale).astype(np.float32))


def lora_adapter(N: int, K: int, rank: int, seed: int, sigma_a: float = None,
                 sigma_b: float = 0.02):
    """bf16 bits of one synthetic low-rank adapter: A uint16[rank][K] with
    N(0, 1/K) entries (unless sigma_a is given) and Bm uint16[N][rank] with
    N(0, sigma_b^2) entries (a trained adapter, not the all-zero Bm of LoRA's
    initialisation)."""
    rng = np.random.default_rng(seed)
    sa = (1.0 / np.sqrt(K)) if sigma_a is None else sigma_a
    A = f32_to_bf16_bits((rng.standard_normal((rank, K)) * sa).astype(np.float32))
    Bm = f32_to_bf16_bits((rng.standard_normal((N, rank)) * sigma_b).astype(np.float32))
    return A, Bm


# --------------------------------------------------- device-side generation

def layer_weights_torch(N: int, K: int, seed: int, device, dist: str = "normal",
                        sigma: float = 0.02, n_outliers: int = 8,
                        outlier_scale: float = 20.0):
    """Same recipe drawn on the device with a seeded torch generator (used for
    the large multi-layer benchmark stacks; a different random stream from
    :func:`layer_weights`).  Returns an int16 tensor of bf16 bits [N][K]."""
    import torch
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    if dist == "normal":
        w = torch.randn((N, K), generator=gen, device=device, dtype=torch.float32) * sigma
    elif dist == "t4":
        z = torch.randn((N, K), generator=gen, device=device, dtype=torch.float32)
        chi = torch.randn((4, N, K), generator=gen, device=device, dtype=torch.float32)
        w = z / torch.sqrt((chi * chi).sum(0) / 4.0) / (2.0 ** 0.5) * sigma
    else:
        raise ValueError(dist)
    if n_outliers:
        cols = torch.randperm(K, generator=gen, device=device)[:n_outliers]
        w[:, cols] *= outlier_scale
    return w.to(torch.bfloat16).view(torch.int16)


def activations_torch(B: int, K: int, seed: int, device):
    import torch
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    x = torch.randn((B, K), generator=gen, device=device, dtype=torch.float32)
    return x.to(torch.bfloat16).view(torch.int16)
