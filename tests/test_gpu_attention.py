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


# ---------------------------------------------------------------- batches of sequences
def batch_oracle(qb, kd, vd, lengths, T_cap, H_kv, scale):
    """Oracle output and the componentwise scale sum_t p_t |v_t[d]| per sequence."""
    qv = (qb.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    B, H, D = qv.shape
    ref = AT.attention_batch(qv, kd, vd, lengths, T_cap, H_kv, scale)
    mag = np.zeros((B, H, D))
    G = H // H_kv
    for b in range(B):
        T = int(lengths[b])
        if T == 0:
            continue
        rows = slice(b * T_cap, b * T_cap + T)
        for h in range(H):
            c = (h // G) * D
            s = scale * (kd[rows, c:c + D] @ qv[b, h])
            p = np.exp(s - s.max())
            p /= p.sum()
            mag[b, h] = p @ np.abs(vd[rows, c:c + D])
    return ref, mag


def make_batch(B, T_cap, lengths, H, H_kv, D, seed, six=False, pad_inf=True):
    g = I.rng(33, B, T_cap, H, H_kv, D, seed)
    K = H_kv * D
    kbits, vbits = kv_map(K // 32, g, six), kv_map(K // 32, g, six)
    k = g.standard_normal((B * T_cap, K)).astype(np.float32)
    k[:, g.choice(K, size=max(1, K // 100), replace=False)] *= 20.0
    v = g.standard_normal((B * T_cap, K)).astype(np.float32)
    q = g.standard_normal((B, H, D)).astype(np.float32)
    kb, vb = I.f32_to_bf16_bits(k), I.f32_to_bf16_bits(v)
    if pad_inf:  # rows past a sequence's length hold Inf: scale 255, NaN if they were ever read
        for b, T in enumerate(lengths):
            kb[b * T_cap + T:(b + 1) * T_cap] = 0x7F80
            vb[b * T_cap + T:(b + 1) * T_cap] = 0x7F80
    return I.f32_to_bf16_bits(q), kb, vb, kbits, vbits


def run_batch(torch, qb, kb, vb, kbits, vbits, H_kv, T_cap, lengths, scale, workspace=None):
    kc, ks, _ = mxs.quantize_act(U.to_dev_bf16(torch, kb), kbits)
    vc, vs, _ = mxs.quantize_act(U.to_dev_bf16(torch, vb), vbits)
    ln = None if lengths is None else torch.tensor(np.asarray(lengths, np.int32), device="cuda")
    out = mxs.attention_decode_batch(U.to_dev_bf16(torch, qb), H_kv, kc, ks, kbits, vc, vs, vbits, T_cap, scale,
                                     lengths=ln, workspace=workspace)
    torch.cuda.synchronize()
    return out.cpu().numpy().astype(np.float64)


@pytest.mark.parametrize("B,T_cap,lengths", [
    (5, 300, [300, 0, 1, 64, 129]),
    (16, 1000, [1000, 999, 7, 500, 63, 65, 128, 1, 0, 1000, 257, 640, 3, 31, 900, 100]),
    (2, 4096, [4096, 2049]),
])
def test_batch_ragged_lengths(torch, B, T_cap, lengths):
    """LLaMA-3-8B heads, B sequences of their own lengths in one launch; the
    rows past each length hold Inf (NaN if read), an empty sequence gives 0."""
    H, H_kv, D = 32, 8, 128
    qb, kb, vb, kbits, vbits = make_batch(B, T_cap, lengths, H, H_kv, D, seed=B)
    scale = 1.0 / np.sqrt(D)
    got = run_batch(torch, qb, kb, vb, kbits, vbits, H_kv, T_cap, lengths, scale)
    ref, mag = batch_oracle(qb, AT.dequantized_cache(kb, kbits), AT.dequantized_cache(vb, vbits), lengths, T_cap,
                            H_kv, scale)
    for b, T in enumerate(lengths):
        if T == 0:
            assert np.all(got[b] == 0.0)
        else:
            check(got[b], ref[b], mag[b])


@pytest.mark.parametrize("H,H_kv,D", [(8, 8, 64), (64, 8, 128), (4, 1, 128), (16, 2, 64), (6, 2, 128)])
def test_batch_head_layouts(torch, H, H_kv, D):
    B, T_cap = 3, 333
    lengths = [333, 190, 5]
    qb, kb, vb, kbits, vbits = make_batch(B, T_cap, lengths, H, H_kv, D, seed=H + D, six=True)
    scale = 0.3 / np.sqrt(D)
    got = run_batch(torch, qb, kb, vb, kbits, vbits, H_kv, T_cap, lengths, scale)
    ref, mag = batch_oracle(qb, AT.dequantized_cache(kb, kbits), AT.dequantized_cache(vb, vbits), lengths, T_cap,
                            H_kv, scale)
    check(got, ref, mag)


@pytest.mark.parametrize("shift", [-123, -131, 119])
def test_tiny_and_huge_blocks(torch, shift):
    """Blocks whose scale byte falls outside [8, 247] (values near 2^-123, bf16
    subnormals near 2^-131, values near 2^121) take the fp32 route: the values
    of two blocks of KV head 0 are scaled by 2^shift, in V, and in K too for the
    small shifts (huge keys would overflow the fp32 scores)."""
    B, T_cap, H, H_kv, D = 2, 200, 8, 2, 128
    lengths = [200, 77]
    qb, kb, vb, kbits, vbits = make_batch(B, T_cap, lengths, H, H_kv, D, seed=abs(shift), six=True, pad_inf=False)
    f = np.float32(2.0) ** shift
    for arr in ((kb, vb) if shift < 0 else (vb,)):
        x = (arr.astype(np.uint32) << 16).view(np.float32)
        x[:, 32:96] *= f  # blocks 1, 2 of KV head 0
        arr[:] = I.f32_to_bf16_bits(x)
    scale = 0.2
    got = run_batch(torch, qb, kb, vb, kbits, vbits, H_kv, T_cap, lengths, scale)
    ref, mag = batch_oracle(qb, AT.dequantized_cache(kb, kbits), AT.dequantized_cache(vb, vbits), lengths, T_cap,
                            H_kv, scale)
    check(got, ref, mag)


def test_workspace_reuse_and_determinism(torch):
    """The counters are back to zero after a call: the same workspace serves
    the next call, and repeated calls give bit-identical results."""
    B, T_cap, H, H_kv, D = 4, 2000, 32, 8, 128
    lengths = [2000, 1500, 1, 640]
    qb, kb, vb, kbits, vbits = make_batch(B, T_cap, lengths, H, H_kv, D, seed=9)
    ws = torch.zeros(mxs.attention_batch_workspace_bytes(B, T_cap, H, D), dtype=torch.uint8, device="cuda")
    a = run_batch(torch, qb, kb, vb, kbits, vbits, H_kv, T_cap, lengths, 0.1, workspace=ws)
    assert int(ws[:256].count_nonzero()) == 0
    b2 = run_batch(torch, qb, kb, vb, kbits, vbits, H_kv, T_cap, lengths, 0.1, workspace=ws)
    assert np.array_equal(a, b2)
    ref, mag = batch_oracle(qb, AT.dequantized_cache(kb, kbits), AT.dequantized_cache(vb, vbits), lengths, T_cap,
                            H_kv, 0.1)
    check(a, ref, mag)
