"""Decode with one to four tokens through mxs_linear_decode and
mxs_linear_decode_group (M = 1: the activations' quantization fused into the
CUDA-core GEMM; M = 2..4: quantizer + tensor-core GEMM) against the exact
oracle; ragged shapes, row groups shared by several CTAs (their partial sums
added by the last to arrive), NaN blocks, ties-away rounding, block scales
over +-20 binades, grouped problems, shallow weight rings."""
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


def _run(torch, xb, wb, bits, N, rounding=mxs.RNE):
    packed = mxs.pack_weight(U.to_dev_bf16(torch, wb), bits, rounding=rounding)
    torch.cuda.synchronize()  # weights are static before the first decode call
    return mxs.linear_decode(U.to_dev_bf16(torch, xb), bits, packed, N, rounding=rounding).cpu().numpy()


def _ref(xb, wb, bits, rounding=mxo.RNE):
    a_s, a_c = mxo.quantize_bf16(xb, bits, rounding)
    w_s, w_c = mxo.quantize_bf16(wb, bits, rounding)
    return mxo.gemm(bits, a_c, a_s, w_c, w_s)


@pytest.mark.parametrize("M", [1, 2, 3, 4])
@pytest.mark.parametrize("N,nb,p", [(37, 5, (0.6, 0.2, 0.2)), (1000, 128, (0.8, 0.15, 0.05)),
                                    (300, 448, (0.5, 0.3, 0.2)), (128, 896, (0.85, 0.1, 0.05)),
                                    (640, 61, (1, 0, 0)), (200, 33, (0, 0.5, 0.5))])
def test_gemv_against_oracle(torch, M, N, nb, p):
    g = I.rng(80, M, N, nb)
    bits = I.width_map(nb, *p, g)
    xb = I.activations_bf16(M, bits, g, 0.01, outlier_scale=30.0)
    wb = I.normal_bf16((N, 32 * nb), 0.02, g)
    y = _run(torch, xb, wb, bits, N)
    ref, ab = _ref(xb, wb, bits)
    U.check_gemm(y, ref, ab)


@pytest.mark.parametrize("M", [1, 4])
def test_gemv_nan_rhaz_and_wide_range(torch, M):
    from test_gpu_gemm_decode import wide_range_layer
    g = I.rng(81, M)
    nb, N = 160, 260
    bits = I.width_map(nb, 0.7, 0.2, 0.1, g)
    xb, wb = wide_range_layer(M, N, nb, bits, g)
    xb[0, 45] = 0x7FC0  # NaN in block 1 of token 0
    wb[7, 32 * 9 + 2] = 0xFF80  # -Inf in block 9 of output 7
    y = _run(torch, xb, wb, bits, N, rounding=mxs.RHAZ)
    ref, ab = _ref(xb, wb, bits, rounding=mxo.RHAZ)
    assert np.all(np.isnan(y[0])) and np.all(np.isnan(y[:, 7]))
    err = U.check_gemm(y, ref, ab)
    print(f"gemv wide range M={M}: max err/abssum {err:.2e}")


def test_gemv_group_and_repeat(torch):
    """Three problems in one launch (q/k/v shapes), twice: identical results,
    each within the bar of the oracle."""
    M = 1
    probs, refs = [], []
    for i, (K, N) in enumerate([(4096, 4096), (4096, 1024), (4096, 1024)]):
        g = I.rng(82, K, N, i)
        bits = I.width_map(K // 32, 0.85, 0.10, 0.05, g)
        xb = I.activations_bf16(M, bits, g, 0.01, outlier_scale=30.0)
        wb = I.normal_bf16((N, K), 0.02, g)
        packed = mxs.pack_weight(U.to_dev_bf16(torch, wb), bits)
        y = torch.full((M, N), float("nan"), device="cuda")
        ws = torch.empty(mxs.linear_decode_workspace_bytes(M, K, N, bits), dtype=torch.uint8, device="cuda")
        probs.append((U.to_dev_bf16(torch, xb), bits, packed, N, y, ws))
        refs.append(_ref(xb, wb, bits))
    torch.cuda.synchronize()
    mxs.linear_decode_group(probs)
    first = [p[4].cpu().numpy().copy() for p in probs]
    mxs.linear_decode_group(probs)
    for (x, bits, packed, N, y, ws), (ref, ab), y0 in zip(probs, refs, first):
        got = y.cpu().numpy()
        assert np.array_equal(got, y0)
        U.check_gemm(got, ref, ab)


@pytest.mark.parametrize("stages", [2, 3])
def test_gemv_shallow_ring(torch, stages):
    """The one-token kernel with two or three weight stages in its ring (what
    it falls back to when a CTA's token codes need the shared memory): same
    results, bit for bit, as with four, and within the bar of the oracle."""
    L = mxs.lib()
    M, N, nb = 1, 3000, 448
    g = I.rng(84, stages)
    bits = I.width_map(nb, 0.6, 0.3, 0.1, g)
    xb = I.activations_bf16(M, bits, g, 0.01, outlier_scale=30.0)
    wb = I.normal_bf16((N, 32 * nb), 0.02, g)
    packed = mxs.pack_weight(U.to_dev_bf16(torch, wb), bits)
    torch.cuda.synchronize()
    x = U.to_dev_bf16(torch, xb)
    y4 = mxs.linear_decode(x, bits, packed, N).cpu().numpy()
    assert L.mxs_test_gemv_ring(stages) == 0
    try:
        ys = mxs.linear_decode(x, bits, packed, N).cpu().numpy()
    finally:
        assert L.mxs_test_gemv_ring(0) == 0
    assert np.array_equal(ys, y4)
    ref, ab = _ref(xb, wb, bits)
    U.check_gemm(ys, ref, ab)
    assert L.mxs_test_gemv_ring(1) == 1 and L.mxs_test_gemv_ring(5) == 1

