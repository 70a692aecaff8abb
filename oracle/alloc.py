"""CPU oracle for MXSens's offline allocation: column sensitivity (Alg. 1) and
sensitivity-based bit allocation (Alg. 3 with the control parameter of
Theorem 1).  Plain numpy, fp64, written from the paper's definitions.

TEST INFRASTRUCTURE ONLY: imported by tests/, __graft_entry__.smoke() and the
cpu_baseline / reference legs of bench.py.  The CUDA library never imports it
and it never imports the CUDA library.

Readings (the paper is silent on these):
  A1  Alg. 3 assigns 6 bits to "the next N6 columns"; Sec. 4.1 puts mild
      outliers in full MXINT blocks.  The columns are laid out in the order of
      Alg. 3 (most sensitive first) and cut into blocks of 32: block 0 is the
      8-bit block, the next floor(N6 / 32) blocks are 6-bit, the rest 4-bit.
  A2  N6 = floor(R * S_layer * (d_in - 32)) is clamped to [0, d_in - 32].
  A3  argsort(descending) breaks ties by column index (stable order).
  A4  The layer sensitivity S_layer (Alg. 2) is an input: it needs a trained
      model, which is out of scope.
"""
from __future__ import annotations

import math

import numpy as np

BLOCK = 32


def bf16_to_f64(x_bits: np.ndarray) -> np.ndarray:
    """bf16 bit patterns (uint16) -> exact fp64 values."""
    u = np.asarray(x_bits, dtype=np.uint16).astype(np.uint32) << 16
    return u.view(np.float32).astype(np.float64)


def column_sensitivity(x_bits: np.ndarray) -> np.ndarray:
    """Alg. 1 for one calibration batch X [T, d_in]: diag(X^T X), i.e. for each
    column j the sum over the rows of X[k, j]^2 (Sec. 3.1: H_jj = sum_k X_kj^2).
    Each square of a bf16 value is exact in fp64; the sum is numpy's fp64 sum."""
    x = bf16_to_f64(x_bits)
    return np.sum(x * x, axis=0)


def allocation_r(d_in, s_layer, B: float) -> float:
    """Theorem 1: the control parameter R for which the average width of the
    triplet allocation (32 columns at 8 bits per layer, R * S_i * (d_i - 32)
    at 6 bits, the rest at 4 bits) is exactly B before any flooring:
        R = ((B - 4) * sum_i d_i - 4 * 32 * n) / sum_i 2 * S_i * (d_i - 32)."""
    d = np.asarray(d_in, dtype=np.float64)
    s = np.asarray(s_layer, dtype=np.float64)
    n = d.size
    num = (B - 4.0) * d.sum() - 4.0 * BLOCK * n
    den = np.sum(2.0 * s * (d - BLOCK))
    return float(num / den)


def n6_columns(d_in: int, R: float, s_layer: float) -> int:
    """Alg. 3: N6 = floor(R * S_layer * (d_in - 32)), clamped to [0, d_in - 32] (A2)."""
    v = math.floor(R * s_layer * (d_in - BLOCK))
    return int(min(max(v, 0), d_in - BLOCK))


def column_order(s: np.ndarray) -> np.ndarray:
    """Alg. 3: argsort of the column sensitivities, descending, ties by index (A3)."""
    s = np.asarray(s, dtype=np.float64)
    return np.argsort(-s, kind="stable").astype(np.int32)


def allocate_layer(s: np.ndarray, R: float, s_layer: float):
    """Alg. 3 for one layer: the column order (perm[p] = original column at
    position p), the width of each 32-column block of that order (A1), and N6."""
    s = np.asarray(s, dtype=np.float64)
    K = s.size
    assert K % BLOCK == 0 and K >= BLOCK
    perm = column_order(s)
    n6 = n6_columns(K, R, s_layer)
    nb = K // BLOCK
    n6b = n6 // BLOCK
    bits = np.full(nb, 4, dtype=np.uint8)
    bits[0] = 8
    bits[1:1 + n6b] = 6
    return perm, bits, n6


def average_width(bits_per_layer, d_in) -> float:
    """Average mantissa width over all columns of all layers (each block's width
    counted for its 32 columns)."""
    tot = sum(int(np.sum(b.astype(np.int64))) * BLOCK for b in bits_per_layer)
    return tot / float(sum(d_in))
