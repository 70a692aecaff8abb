"""Seeded synthetic inputs shared by the tests, the oracle checks and bench.py.

This module holds no arithmetic of the method: it draws random numbers, rounds
them to bf16 (the input dtype of the layer) and builds width maps.  Both the
CUDA path and the CPU oracle consume what it returns.

Recipe (the paper's workloads are LLaMA-family linear layers; their weights and
calibration data are not available, so these draws stand in for them):
  * every tensor has its own stream: PCG64(SeedSequence([seed, *keys]));
  * values are drawn in fp32 and rounded once to bf16 (ties to even);
  * weights ~ N(0, sigma_w); activations ~ N(0, 1) with a few outlier columns,
    either scaled by a constant or redrawn from a Student-t(3);
  * a width map draws n8 = round(p8*nb), n6 = round(p6*nb) blocks, the rest
    4-bit; 8-bit blocks are placed first (randomly, or as one contiguous run),
    6-bit blocks are a random subset of the remaining blocks; outlier columns
    fall inside 8-bit blocks (the paper gives its top-32 sensitive columns
    8 bits, Sec. 4.1 / Alg. 3).
"""
from __future__ import annotations

import numpy as np


def rng(seed: int, *keys: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([int(seed)] + [int(k) for k in keys])))


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """fp32 -> bf16 bit patterns (uint16), round to nearest even; inputs finite."""
    u = np.array(x, dtype=np.float32, copy=True).view(np.uint32)
    lsb = (u >> 16) & 1          # finite inputs: u + 0x8000 stays below 2^32
    u += 0x7FFF
    u += lsb
    u >>= 16
    return u.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def width_map(nb: int, p4: float, p6: float, p8: float, g: np.random.Generator,
              clustered: bool = False, n8: int | None = None, n6: int | None = None) -> np.ndarray:
    """uint8 [nb] of widths {4, 6, 8}."""
    assert abs(p4 + p6 + p8 - 1.0) < 1e-9
    if n8 is None:
        n8 = int(np.floor(p8 * nb + 0.5))
    if n6 is None:
        n6 = int(np.floor(p6 * nb + 0.5))
    n8 = min(n8, nb)
    n6 = min(n6, nb - n8)
    bits = np.full(nb, 4, np.uint8)
    if clustered and n8 > 0:
        start = int(g.integers(0, nb - n8 + 1))
        idx8 = np.arange(start, start + n8)
    else:
        idx8 = g.choice(nb, size=n8, replace=False)
    bits[idx8] = 8
    rest = np.flatnonzero(bits == 4)
    idx6 = g.choice(rest, size=n6, replace=False) if n6 > 0 else np.zeros(0, np.int64)
    bits[idx6] = 6
    return bits


def outlier_columns(bits: np.ndarray, count: int, g: np.random.Generator) -> np.ndarray:
    """count column indices, inside 8-bit blocks when there is room, else anywhere."""
    cols8 = np.concatenate([np.arange(32 * kb, 32 * kb + 32) for kb in np.flatnonzero(bits == 8)]) \
        if np.any(bits == 8) else np.zeros(0, np.int64)
    K = 32 * bits.size
    pool = cols8 if cols8.size >= count else np.arange(K)
    return np.sort(g.choice(pool, size=count, replace=False))


def normal_bf16(shape, sigma: float, g: np.random.Generator) -> np.ndarray:
    x = g.standard_normal(size=shape, dtype=np.float32) * np.float32(sigma)
    return f32_to_bf16_bits(x)


def activations_bf16(M: int, bits: np.ndarray, g: np.random.Generator, outlier_frac: float,
                     outlier_scale: float | None = None, student_t: bool = False) -> np.ndarray:
    """bf16 bits [M, K]: N(0,1) with round(outlier_frac*K) outlier columns."""
    K = 32 * bits.size
    x = g.standard_normal(size=(M, K), dtype=np.float32)
    n_out = int(np.floor(outlier_frac * K + 0.5))
    if n_out > 0:
        cols = outlier_columns(bits, n_out, g)
        if student_t:
            x[:, cols] = g.standard_t(3.0, size=(M, cols.size)).astype(np.float32)
        else:
            x[:, cols] *= np.float32(outlier_scale)
    return f32_to_bf16_bits(x)


# ------------------------------------------------------------------ workloads
# LLaMA-3-8B: hidden 4096, MLP 14336, GQA k/v 1024; LLaMA-2-70B: 8192 / 28672 / 1024.
# Shapes are (name, K, N) with y[M,N] = x[M,K] @ W[N,K]^T.
LLAMA3_8B = [("q", 4096, 4096), ("k", 4096, 1024), ("v", 4096, 1024), ("o", 4096, 4096),
             ("gate", 4096, 14336), ("up", 4096, 14336), ("down", 14336, 4096)]
LLAMA2_70B = [("q", 8192, 8192), ("k", 8192, 1024), ("v", 8192, 1024), ("o", 8192, 8192),
              ("gate", 8192, 28672), ("up", 8192, 28672), ("down", 28672, 8192)]


def llama70b_layer_map(K: int, layer: int, n_layers: int, g: np.random.Generator) -> np.ndarray:
    """4-bit share linear from 60% (layer 0) to 95% (last layer); 8-bit blocks cover
    the 1% outlier columns (ceil(0.01K/32) blocks); the rest of the share is 6-bit."""
    nb = K // 32
    p4 = 0.60 + 0.35 * layer / max(1, n_layers - 1)
    n_out = int(np.floor(0.01 * K + 0.5))
    n8 = -(-n_out // 32)
    n4 = int(np.floor(p4 * nb + 0.5))
    n6 = max(0, nb - n4 - n8)
    return width_map(nb, 1.0, 0.0, 0.0, g, n8=n8, n6=n6)
