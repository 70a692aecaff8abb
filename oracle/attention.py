"""CPU oracle for attention over an MXINT-quantized KV cache (the paper
quantizes the KV cache with a 4-8 bit configuration, Appendix A.2, and keeps
Softmax in FP16).  Plain numpy, fp64.

TEST INFRASTRUCTURE ONLY: imported by tests/, __graft_entry__.smoke() and the
cpu_baseline / reference legs of bench.py.  The CUDA library never imports it
and it never imports the CUDA library.

One decode step of one sequence: query q [H, D] (H query heads of D dims),
cache rows t < T of K and V, each row the H_kv * D values of one token,
quantized along that row in blocks of 32 with the row's own width map (the
activation layout of this library).  Query head h reads KV head
h // (H / H_kv) (grouped-query attention).  For each query head:
    s_t = scale * <q_h, k_t[kv head]>,  p = softmax(s),  out_h = sum_t p_t v_t[kv head].
Readings: the scores, the softmax and the weighted sum are taken in real
arithmetic on the dequantized cache (the paper keeps Softmax in FP16 and
does not say how the products are formed); a block with S = 255 gives NaN.

A decode batch (attention_batch) is B independent sequences: sequence b
owns cache rows [b * T_cap, b * T_cap + T_b) and its own query; rows past
its length are not read.  A sequence of length 0 attends to nothing and its
output reads as zero (the paper does not define it).
"""
from __future__ import annotations

import numpy as np

from oracle import mxo


def dequantized_cache(x_bits: np.ndarray, bits) -> np.ndarray:
    """bf16 rows [T, H_kv * D] -> the fp64 values of their MXINT quantization."""
    scales, codes = mxo.quantize_bf16(x_bits, bits)
    return mxo.dequantize(codes, scales, bits)


def attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, n_kv_heads: int, scale: float) -> np.ndarray:
    """q [H, D] fp64, k and v [T, H_kv * D] fp64 -> out [H, D] fp64 (see the module text)."""
    q = np.asarray(q, np.float64)
    H, D = q.shape
    T = k.shape[0]
    G = H // n_kv_heads
    out = np.zeros((H, D))
    for h in range(H):
        c = (h // G) * D
        kh = k[:, c:c + D]
        vh = v[:, c:c + D]
        s = scale * (kh @ q[h])
        m = np.max(s) if T else 0.0
        p = np.exp(s - m)
        out[h] = (p @ vh) / np.sum(p)
    return out


def attention_batch(q: np.ndarray, k: np.ndarray, v: np.ndarray, lengths, T_cap: int, n_kv_heads: int,
                    scale: float) -> np.ndarray:
    """q [B, H, D]; k, v [B * T_cap, H_kv * D] fp64; lengths[b] tokens of
    sequence b -> out [B, H, D] fp64 (see the module text)."""
    q = np.asarray(q, np.float64)
    B, H, D = q.shape
    out = np.zeros((B, H, D))
    for b in range(B):
        T = int(lengths[b])
        if T > 0:
            rows = slice(b * T_cap, b * T_cap + T)
            out[b] = attention(q[b], k[rows], v[rows], n_kv_heads, scale)
    return out
