"""Decode attention over an MXINT KV cache against the oracle.

The cache rows are quantized by mxs_quantize_act (the paper's 4-8 bit KV
configuration, plus a 4/6/8 map to exercise every code width); the kernel's
element values are exact in fp32, so its error comes from fp32 dot products
(up to 36 roundings per score), expf and the fp32 sums over a 128-token chunk
and over chunks.  Bound used: for every output element,
|out - ref| <= 1e-4 * sum_t p_t |v_t[d]|, the componentwise scale of the
weighted sum (estimated error ~3e-5 of it for scores of a few units)."""
import numpy as np
import pytest

from oracle import attention as AT
from paper_2607_17733_gb300 import inputs as I
from paper_2607_17733_gb300 import mxs
import gpu_util as U

pytestmark = pytest.mark.gpu
TOL = 1e-4


@pytest.fixture(scope="module")
def torch():
    return U.torch_or_skip()


def kv_map(nb, g, six=False):
    """One 8-bit block (the paper's KV setting keeps its most sensitive 32
    columns at 8 bits), the rest 4-bit; optionally a quarter at 6 bits."""
    bits = np.full(nb, 4, np.uint8)
    bits[g.integers(nb)] = 8
    if six:
        bits[g.choice(np.flatnonzero(bits == 4), size=nb // 4, replace=False)] = 6
    return bits


def make_case(T, H, H_kv, D, seed, six=False, key_outliers=True):
    g = I.rng(31, T, H, H_kv, D, seed)
    K = H_kv * D
    kb_map, vb_map = kv_map(K // 32, g, six), kv_map(K // 32, g, six)
    k = g.standard_normal((T, K)).astype(np.float32)
    if key_outliers:
        k[:, g.choice(K, size=max(1, K // 100), replace=False)] *= 20.0
    v = g.standard_normal((T, K)).astype(np.float32)
    q = g.standard_normal((H, D)).astype(np.float32)
    return (I.f32_to_bf16_bits(q), I.f32_to_bf16_bits(k), I.f32_to_bf16_bits(v), kb_map, vb_map)


def run_gpu(torch, qb, kb, vb, k_bits, v_bits, H_kv, scale):
    T = kb.shape[0]
    kc, ks, _ = mxs.quantize_act(U.to_dev_bf16(torch, kb), k_bits)
    vc, vs, _ = mxs.quantize_act(U.to_dev_bf16(torch, vb), v_bits)
    out = mxs.attention_decode(U.to_dev_bf16(torch, qb), H_kv, kc, ks, k_bits, vc, vs, v_bits, T, scale)
    torch.cuda.synchronize()
    return out.cpu().numpy().astype(np.float64)


def oracle(qb, kb, vb, k_bits, v_bits, H_kv, scale):
    qv = (qb.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    kd = AT.dequantized_cache(kb, k_bits)
    vd = AT.dequantized_cache(vb, v_bits)
    ref = AT.attention(qv, kd, vd, H_kv, scale)
    # componentwise scale sum_t p_t |v_t[d]|
    H, D = qv.shape
    G = H // H_kv
    mag = np.zeros((H, D))
    for h in range(H):
        c = (h // G) * D
        s = scale * (kd[:, c:c + D] @ qv[h])
        p = np.exp(s - s.max())
        p /= p.sum()
        mag[h] = p @ np.abs(vd[:, c:c + D])
    return ref, mag


def check(got, ref, mag):
    err = np.abs(got - ref)
    assert np.all(err <= TOL * mag + 1e-30), f"max err/scale {np.max(err / np.maximum(mag, 1e-30)):.3g}"


@pytest.mark.parametrize("T", [1, 127, 128, 129, 1000, 4096])
def test_llama3_8b_heads(torch, T):
    """LLaMA-3-8B attention: 32 query heads over 8 KV heads of 128 dims."""
    H, H_kv, D = 32, 8, 128
    qb, kb, vb, kbits, vbits = make_case(T, H, H_kv, D, seed=T)
    scale = 1.0 / np.sqrt(D)
    got = run_gpu(torch, qb, kb, vb, kbits, vbits, H_kv, scale)
    ref, mag = oracle(qb, kb, vb, kbits, vbits, H_kv, scale)
    check(got, ref, mag)


@pytest.mark.parametrize("H,H_kv,D,T", [(8, 8, 64, 300), (64, 8, 128, 513), (4, 1, 128, 77), (16, 2, 64, 2048)])
def test_head_layouts_and_six_bit_blocks(torch, H, H_kv, D, T):
    qb, kb, vb, kbits, vbits = make_case(T, H, H_kv, D, seed=H, six=True)
    scale = 0.3 / np.sqrt(D)
    got = run_gpu(torch, qb, kb, vb, kbits, vbits, H_kv, scale)
    ref, mag = oracle(qb, kb, vb, kbits, vbits, H_kv, scale)
    check(got, ref, mag)


def test_cache_appended_token_by_token(torch):
    """Appending token t is one quantizer call of one row into row t: the cache
    built that way equals the one quantized in bulk, byte for byte."""
    T, K = 40, 1024
    g = I.rng(32)
    bits = kv_map(K // 32, g, six=True)
    xb = I.f32_to_bf16_bits(g.standard_normal((T, K)).astype(np.float32))
    bulk_c, bulk_s, _ = mxs.quantize_act(U.to_dev_bf16(torch, xb), bits)
    codes = torch.zeros_like(bulk_c)
    scales = torch.zeros_like(bulk_s)
    for t in range(T):
        mxs.quantize_act(U.to_dev_bf16(torch, xb[t:t + 1]), bits, codes=codes[t:t + 1], scales=scales[t:t + 1])
    torch.cuda.synchronize()
    assert torch.equal(codes, bulk_c) and torch.equal(scales, bulk_s)


def test_non_finite_cache_block(torch):
    """A cached Inf gives its block scale 255; the heads reading that KV head are NaN, the others are not."""
    H, H_kv, D, T = 8, 2, 128, 50
    qb, kb, vb, kbits, vbits = make_case(T, H, H_kv, D, seed=5)
    kb = kb.copy()
    kb[7, 3] = 0x7F80  # +Inf in KV head 0
    got = run_gpu(torch, qb, kb, vb, kbits, vbits, H_kv, 0.1)
    assert np.all(np.isnan(got[:4])) and np.all(np.isfinite(got[4:]))
