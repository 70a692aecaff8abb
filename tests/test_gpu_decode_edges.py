"""Decode (mxs_linear_decode, 1 <= M <= 16) against the exact oracle at the
edges of the scale range and of the shapes: activation blocks up to 2^127
(scale byte 254) against weights near 2^-110, weight blocks below 2^-126
(scale byte 0) and near 2^127, one-block layers, a second 8-token tile that
holds a few tokens, a last row group of one row, and K long enough for every
cluster size.  M = 1 runs the CUDA-core kernel, M > 1 the tensor-core one."""
import numpy as np
import pytest

from oracle import mxo
from paper_2607_17733_gb300 import inputs as I
from paper_2607_17733_gb300 import mxs
import gpu_util as U

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch():
    return U.torch_or_skip()


def _ref(xb, wb, bits):
    a_s, a_c = mxo.quantize_bf16(xb, bits, mxo.RNE)
    w_s, w_c = mxo.quantize_bf16(wb, bits, mxo.RNE)
    return mxo.gemm(bits, a_c, a_s, w_c, w_s)


def _run(torch, xb, wb, bits, N):
    packed = mxs.pack_weight(U.to_dev_bf16(torch, wb), bits)
    torch.cuda.synchronize()
    return mxs.linear_decode(U.to_dev_bf16(torch, xb), bits, packed, N).cpu().numpy()


@pytest.mark.parametrize("M", [1, 7, 16])
def test_huge_activation_blocks(torch, M):
    """Activation blocks scaled to 2^118..2^125, one element at 1.5 * 2^127
    (scale bytes 245..254), against weight blocks scaled to 2^-110: every
    term is an ordinary fp32 number and comes out exact."""
    g = I.rng(91, M)
    nb, N = 96, 300
    bits = I.width_map(nb, 0.5, 0.25, 0.25, g)
    xf = I.bf16_bits_to_f32(I.activations_bf16(M, bits, g, 0.0)).copy()
    wf = I.bf16_bits_to_f32(I.normal_bf16((N, 32 * nb), 0.02, g)).copy()
    huge = [k for k in range(nb) if k % 7 == 3]
    for j, k in enumerate(huge):
        xf[:, 32 * k:32 * k + 32] *= np.float32(2.0 ** (118 + j % 8))
        wf[:, 32 * k:32 * k + 32] *= np.float32(2.0 ** -110)
    xf[0, 32 * huge[-1]] = np.float32(1.5 * 2.0 ** 127)
    xb, wb = I.f32_to_bf16_bits(xf), I.f32_to_bf16_bits(wf)
    a_s, _ = mxo.quantize_bf16(xb, bits, mxo.RNE)
    assert a_s[:, huge].max() == 254
    y = _run(torch, xb, wb, bits, N)
    ref, ab = _ref(xb, wb, bits)
    assert np.isfinite(ref).all()
    err = U.check_gemm(y, ref, ab)
    print(f"huge activation blocks M={M}: max err/abssum {err:.2e}")


@pytest.mark.parametrize("M,top", [(1, 131), (4, 120)])
def test_weight_scale_extremes(torch, M, top):
    """Weight blocks below 2^-126 (subnormal bf16: scale byte 0) against
    activations near 2^100, and weight blocks scaled by 2^top against
    activations near 2^-100: every term is an ordinary number and comes out
    exact.  The CUDA-core path (M = 1) takes weight scale bytes up to 254; the
    tensor-core path is exact up to 245 (|w| < 2^118; above, the scale of a
    shifted digit saturates), so M = 4 stays there."""
    nb, N = 40, 160
    g = I.rng(92, M)
    bits = I.width_map(nb, 0.6, 0.2, 0.2, g)
    xf = I.bf16_bits_to_f32(I.activations_bf16(M, bits, g, 0.0)).copy()
    wf = I.bf16_bits_to_f32(I.normal_bf16((N, 32 * nb), 0.02, g)).copy()
    for k in range(0, nb, 5):
        wf[:, 32 * k:32 * k + 32] *= np.float32(2.0 ** -124)
        xf[:, 32 * k:32 * k + 32] *= np.float32(2.0 ** 100)
    for k in range(2, nb, 5):
        wf[:, 32 * k:32 * k + 32] = (wf[:, 32 * k:32 * k + 32].astype(np.float64) * 2.0 ** top).astype(np.float32)
        xf[:, 32 * k:32 * k + 32] *= np.float32(2.0 ** -100)
    xb, wb = I.f32_to_bf16_bits(xf), I.f32_to_bf16_bits(wf)
    w_s, _ = mxo.quantize_bf16(wb, bits, mxo.RNE)
    assert (w_s == 0).any() and w_s.max() == (254 if M == 1 else 243)
    y = _run(torch, xb, wb, bits, N)
    ref, ab = _ref(xb, wb, bits)
    U.check_gemm(y, ref, ab)


@pytest.mark.parametrize("M,N,nb,p", [(1, 5, 1, (1, 0, 0)), (9, 130, 1, (0, 0, 1)), (16, 129, 3, (0, 1, 0)),
                                      (9, 1000, 640, (0.7, 0.2, 0.1)), (12, 8192, 256, (0.9, 0.05, 0.05)),
                                      (2, 3000, 896, (0.6, 0.3, 0.1)), (1, 3000, 896, (0.6, 0.3, 0.1))])
def test_edge_shapes(torch, M, N, nb, p):
    """One-block layers, a second token tile holding one or a few tokens, a
    last row group of one row, and K long enough for every cluster size."""
    g = I.rng(93, M, N, nb)
    bits = I.width_map(nb, *p, g)
    xb = I.activations_bf16(M, bits, g, 0.01, outlier_scale=30.0)
    wb = I.normal_bf16((N, 32 * nb), 0.02, g)
    y = _run(torch, xb, wb, bits, N)
    ref, ab = _ref(xb, wb, bits)
    U.check_gemm(y, ref, ab)
