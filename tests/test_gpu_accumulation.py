"""How the tensor core adds block terms into its fp32 accumulator.

Every block term 2^(Ea'+Ew') * D of the MXINT product is exact on the tensor
core (Sec. 2: integer MACs under a shared scale); the one rounding left in the
prefill GEMM is the fp32 accumulation in tensor memory.  These tests pin that
rounding: the kernel's result equals, bit for bit, the replay of its MMAs
under the rule in tc_model.py (addends cut toward zero to two bits below the
largest addend's last place, the sum cut toward zero), and differs from
rounding to nearest.  This is why the prefill GEMM can miss a 1e-5 error bar
on inputs whose block scales spread over many binades, while every
LLaMA-shaped configuration comes out exact."""
import numpy as np
import pytest

from oracle import mxo
from paper_2607_17733_gb300 import inputs as I
from paper_2607_17733_gb300 import mxs
import gpu_util as U
import tc_model as T

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch():
    return U.torch_or_skip()


def _bf16(v):
    return I.f32_to_bf16_bits(np.asarray(v, np.float32))


def _prefill(torch, xb, wb, bits):
    _, _, planes = mxs.quantize_act(U.to_dev_bf16(torch, xb), bits, want_codes=False, want_planes=True)
    packed = mxs.pack_weight(U.to_dev_bf16(torch, wb), bits, layout=mxs.W_COMPACT_AND_PLANES)
    return mxs.gemm_prefill(planes, bits, packed, xb.shape[0], wb.shape[0]).cpu().numpy()


def _rne_sequential(terms: np.ndarray) -> np.ndarray:
    acc = np.zeros(terms.shape[:-1], np.float32)
    for k in range(terms.shape[-1]):
        acc = (acc.astype(np.float64) + terms[..., k]).astype(np.float32)
    return acc


@pytest.mark.parametrize("seed", range(4))
def test_prefill_accumulation_probe(torch, seed):
    """M = 32, N = 16, K = 128 (four 4-bit blocks, one K' stage of four MMAs).
    Block 0 holds 1.0 in every row and column; blocks 1-3 hold one value m/4 *
    2^E (m in 4..7: exact in 4-bit MXINT), signed in the weights, so each MMA
    adds one known product near the accumulator's last place."""
    M, N, K = 32, 16, 128
    rs = np.random.default_rng(seed)
    x = np.zeros((M, K), np.float32)
    w = np.zeros((N, K), np.float32)
    x[:, 0] = 1.0
    w[:, 0] = 1.0
    for k in (1, 2, 3):
        x[:, 32 * k] = rs.integers(4, 8, M) / 4.0 * 2.0 ** rs.integers(-14, -9, M)
        w[:, 32 * k] = rs.choice([-1.0, 1.0], N) * rs.integers(4, 8, N) / 4.0 * 2.0 ** rs.integers(-15, -9, N)
    bits = np.full(K // 32, 4, np.uint8)
    xb, wb = _bf16(x), _bf16(w)
    a_s, a_c = mxo.quantize_bf16(xb, bits)
    w_s, w_c = mxo.quantize_bf16(wb, bits)
    assert np.array_equal(mxo.dequantize(a_c, a_s, bits), x.astype(np.float64))
    assert np.array_equal(mxo.dequantize(w_c, w_s, bits), w.astype(np.float64))
    y = _prefill(torch, xb, wb, bits)
    model = T.prefill_model(bits, a_c, a_s, w_c, w_s)
    terms = np.stack([x[:, None, 32 * k].astype(np.float64) * w[None, :, 32 * k] for k in range(4)], axis=-1)
    rne = _rne_sequential(terms)
    print(f"seed {seed}: model matches {np.mean(y == model):.4f}, sequential round-to-nearest "
          f"{np.mean(y == rne):.4f} of {y.size} outputs")
    assert np.array_equal(y, model)
    assert not np.array_equal(y, rne)


@pytest.mark.parametrize("M,N,nb,p", [(48, 64, 128, (0.8, 0.15, 0.05)), (40, 48, 96, (0.5, 0.3, 0.2)),
                                      (33, 40, 40, (0, 0.5, 0.5)), (64, 64, 64, (1, 0, 0))])
def test_prefill_matches_the_accumulation_model(torch, M, N, nb, p):
    """Blocks scaled over +-20 binades (exact results do not fit fp32): every
    output of the kernel equals the replay of its MMAs under the rule; the
    model's distance to the exact oracle is printed beside it."""
    from test_gpu_gemm_decode import wide_range_layer
    g = I.rng(44, M, nb)
    bits = I.width_map(nb, *p, g)
    xb, wb = wide_range_layer(M, N, nb, bits, g)
    y = _prefill(torch, xb, wb, bits)
    a_s, a_c = mxo.quantize_bf16(xb, bits)
    w_s, w_c = mxo.quantize_bf16(wb, bits)
    model = T.prefill_model(bits, a_c, a_s, w_c, w_s)
    ref, ab = mxo.gemm(bits, a_c, a_s, w_c, w_s)
    dev = np.max(np.abs(model.astype(np.float64) - ref) / ab)
    print(f"M={M} N={N} K={32 * nb}: model matches {np.mean(y == model):.4f}; model vs exact {dev:.2e}")
    assert np.array_equal(y, model)
