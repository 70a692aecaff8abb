"""Pins of the attention oracle (oracle/attention.py) to closed forms:
equal scores give the mean of the values, one dominant key gives its value,
a common shift of the scores changes nothing, grouped heads read their own
KV head, and a two-token case against the logistic function."""
import math

import numpy as np

from oracle import attention as AT
from oracle import mxo
from paper_2607_17733_gb300 import inputs as I


def test_equal_scores_average_the_values():
    g = np.random.default_rng(1)
    T, D = 37, 128
    q = np.zeros((1, D))
    v = g.standard_normal((T, D))
    out = AT.attention(q, g.standard_normal((T, D)), v, 1, 0.1)
    assert np.allclose(out[0], v.mean(axis=0), rtol=0, atol=1e-14)


def test_one_dominant_key_returns_its_value():
    g = np.random.default_rng(2)
    T, D = 20, 64
    k = g.standard_normal((T, D)) * 0.01
    q = np.zeros((1, D))
    q[0, 0] = 1.0
    k[7, 0] = 1e4
    v = g.standard_normal((T, D))
    assert np.allclose(AT.attention(q, k, v, 1, 1.0)[0], v[7], rtol=0, atol=1e-12)


def test_two_tokens_follow_the_logistic_function():
    q = np.array([[1.0, 2.0]])
    k = np.array([[0.5, 0.0], [0.0, 1.0]])
    v = np.array([[1.0, 0.0], [0.0, 1.0]])
    s0, s1 = 0.5 * 0.3, 2.0 * 0.3
    p1 = 1.0 / (1.0 + math.exp(s0 - s1))
    assert np.allclose(AT.attention(q, k, v, 1, 0.3)[0], [1 - p1, p1], rtol=0, atol=1e-15)


def test_grouped_heads_read_their_kv_head():
    """H = 4 query heads over H_kv = 2: heads 0, 1 read KV head 0, heads 2, 3 KV head 1."""
    g = np.random.default_rng(3)
    T, D = 9, 32
    q = g.standard_normal((4, D))
    k = g.standard_normal((T, 2 * D))
    v = g.standard_normal((T, 2 * D))
    out = AT.attention(q, k, v, 2, 0.2)
    for h in range(4):
        c = (h // 2) * D
        assert np.allclose(out[h], AT.attention(q[h:h + 1], k[:, c:c + D], v[:, c:c + D], 1, 0.2)[0])


def test_shifting_the_scores_changes_nothing():
    """softmax(s + c) = softmax(s): q + a component orthogonal to every key."""
    g = np.random.default_rng(4)
    T, D = 50, 16
    k = g.standard_normal((T, D))
    k[:, -1] = 1.0
    q = g.standard_normal((1, D))
    v = g.standard_normal((T, D))
    q2 = q.copy()
    q2[0, -1] += 3.0  # every score moves by the same 3 * scale
    assert np.allclose(AT.attention(q, k, v, 1, 0.5), AT.attention(q2, k, v, 1, 0.5), rtol=1e-12, atol=1e-12)


def test_cache_values_are_the_mxint_values():
    """The dequantized cache is codes x 2^(S - 127 - (b - 2)), the MXINT element value."""
    g = I.rng(5)
    bits = I.width_map(8, 0.75, 0, 0.25, g)
    xb = I.activations_bf16(6, bits, g, 0.02, outlier_scale=30.0)
    c = AT.dequantized_cache(xb, bits)
    s, codes = mxo.quantize_bf16(xb, bits)
    for r in range(6):
        for kb in range(8):
            b = int(bits[kb])
            for i in range(32):
                assert c[r, 32 * kb + i] == math.ldexp(int(codes[r, 32 * kb + i]), int(s[r, kb]) - 127 - (b - 2))


def test_batch_reads_each_sequence_up_to_its_length():
    """Sequence b sees rows [b*T_cap, b*T_cap + T_b) only: rows past its
    length (set to NaN here) change nothing, an empty sequence is zero, and
    each output equals the one-sequence call on its own rows."""
    g = np.random.default_rng(6)
    B, T_cap, H, H_kv, D = 4, 11, 4, 2, 16
    lengths = [11, 0, 1, 6]
    q = g.standard_normal((B, H, D))
    k = g.standard_normal((B * T_cap, H_kv * D))
    v = g.standard_normal((B * T_cap, H_kv * D))
    for b, T in enumerate(lengths):
        k[b * T_cap + T:(b + 1) * T_cap] = np.nan
        v[b * T_cap + T:(b + 1) * T_cap] = np.nan
    out = AT.attention_batch(q, k, v, lengths, T_cap, H_kv, 0.25)
    assert np.all(np.isfinite(out))
    assert np.all(out[1] == 0.0)
    # one token: softmax of one score is 1, so the output is that token's value
    for h in range(H):
        c = (h // (H // H_kv)) * D
        assert np.array_equal(out[2, h], v[2 * T_cap, c:c + D])
    for b in (0, 3):
        rows = slice(b * T_cap, b * T_cap + lengths[b])
        assert np.array_equal(out[b], AT.attention(q[b], k[rows], v[rows], H_kv, 0.25))
