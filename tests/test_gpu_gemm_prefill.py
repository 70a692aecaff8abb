"""A3 parity: the tcgen05 prefill GEMM (e4m3 digit planes, block-scaled MMA,
fp32 TMEM accumulation) against the exact CPU oracle."""
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


def prep(torch, xb, wb, bits):
    _, _, planes = mxs.quantize_act(U.to_dev_bf16(torch, xb), bits, want_codes=False, want_planes=True)
    packed = mxs.pack_weight(U.to_dev_bf16(torch, wb), bits, layout=mxs.W_COMPACT_AND_PLANES)
    return planes, packed


def oracle_entries(xb, wb, bits, rows=None, cols=None):
    if rows is not None:
        xb = xb[rows]
    if cols is not None:
        wb = wb[cols]
    a_s, a_c = mxo.quantize_bf16(xb, bits)
    w_s, w_c = mxo.quantize_bf16(wb, bits)
    return mxo.gemm(bits, a_c, a_s, w_c, w_s)


MAPS = {"u4": (1, 0, 0), "u6": (0, 1, 0), "u8": (0, 0, 1), "mix": (0.8, 0.15, 0.05), "heavy": (0.5, 0.3, 0.2)}


@pytest.mark.parametrize("M,N,nb", [(128, 256, 4), (17, 16, 1), (130, 300, 9), (300, 520, 40), (256, 1024, 128)])
@pytest.mark.parametrize("mp", list(MAPS))
def test_prefill_small(torch, M, N, nb, mp):
    g = I.rng(M, N, nb, len(mp))
    bits = I.width_map(nb, *MAPS[mp], g)
    xb = I.activations_bf16(M, bits, g, 0.01, outlier_scale=50.0)
    wb = I.normal_bf16((N, 32 * nb), 0.02, g)
    planes, packed = prep(torch, xb, wb, bits)
    y = mxs.gemm_prefill(planes, bits, packed, M, N).cpu().numpy()
    ref, ab = oracle_entries(xb, wb, bits)
    err = U.check_gemm(y, ref, ab)
    print(f"prefill M={M} N={N} K={32 * nb} map={mp}: max err/abssum {err:.2e}")


def test_prefill_special_blocks(torch):
    """NaN and Inf in 4-, 6- and 8-bit blocks of activations and weights: the
    outputs that read such a block are NaN (R5: scale byte 255, zero codes;
    the bf16 form of a 6/8-bit block holds NaN), all others match the oracle;
    all-zero and subnormal blocks quantize like any other."""
    bits = np.array([4, 6, 8, 4, 6, 8, 4, 4], np.uint8)
    g = I.rng(33)
    M, N = 40, 150
    xb = I.activations_bf16(M, bits, g, 0.0)
    wb = I.normal_bf16((N, 32 * len(bits)), 0.02, g)
    xb[3, 40] = 0x7FC0    # NaN in the 6-bit block of token 3
    xb[7, 70] = 0x7F80    # +Inf in the 8-bit block of token 7
    xb[11, 5] = 0xFF80    # -Inf in a 4-bit block of token 11
    xb[20, 32 * 4:32 * 5] = 0        # an all-zero 6-bit block
    xb[21, 32 * 2:32 * 3] = 0x0003   # a subnormal 8-bit block
    wb[9, 32 * 5 + 3] = 0x7FC0       # NaN in the 8-bit block of output 9
    planes, packed = prep(torch, xb, wb, bits)
    y = mxs.gemm_prefill(planes, bits, packed, M, N).cpu().numpy()
    ref, ab = oracle_entries(xb, wb, bits)
    for r in (3, 7, 11):
        assert np.all(np.isnan(y[r]))
    assert np.all(np.isnan(y[:, 9]))
    U.check_gemm(y, ref, ab)


@pytest.mark.parametrize("pad", [64, 3])
def test_prefill_through_mxs_gemm_and_stride(torch, pad):
    """Ragged M and N, y a view with row stride N + pad: rows of 16-byte
    multiples go out through TMA stores (clipped at N and M), other strides
    through plain stores; the padding columns stay untouched."""
    g = I.rng(21)
    bits = I.width_map(32, 0.8, 0.15, 0.05, g)
    M, N = 200, 384 - 40
    xb = I.activations_bf16(M, bits, g, 0.01, outlier_scale=50.0)
    wb = I.normal_bf16((N, 1024), 0.02, g)
    planes, packed = prep(torch, xb, wb, bits)
    y = torch.full((M, N + pad), -3.0, device="cuda")
    mxs.gemm(None, None, planes, bits, packed, N, w_layout=mxs.W_COMPACT_AND_PLANES, y=y[:, :N], M=M)
    yh = y.cpu().numpy()
    assert np.all(yh[:, N:] == -3.0)
    ref, ab = oracle_entries(xb, wb, bits)
    U.check_gemm(yh[:, :N], ref, ab)


@pytest.mark.parametrize("shape", [("llama3-8b-gate", 2048, 4096, 14336, (0.8, 0.15, 0.05)),
                                   ("llama3-8b-down", 2048, 14336, 4096, (0.8, 0.15, 0.05)),
                                   ("single-layer", 128, 4096, 4096, (0.8, 0.15, 0.05))])
def test_prefill_full_size_sampled(torch, shape):
    name, M, K, N, p = shape
    g = I.rng(2, M, K, N)
    bits = I.width_map(K // 32, *p, g)
    xb = I.activations_bf16(M, bits, g, 0.005, student_t=True)
    wb = I.normal_bf16((N, K), 0.02, g)
    planes, packed = prep(torch, xb, wb, bits)
    y = mxs.gemm_prefill(planes, bits, packed, M, N).cpu().numpy()
    rs = np.random.default_rng(0)
    rows = np.sort(rs.choice(M, min(M, 96), replace=False))
    cols = np.sort(rs.choice(N, min(N, 512), replace=False))
    ref, ab = oracle_entries(xb, wb, bits, rows, cols)
    err = U.check_gemm(y[np.ix_(rows, cols)], ref, ab)
    print(f"prefill {name}: max err/abssum {err:.2e}")


@pytest.mark.parametrize("maps", ["u6", "u8", "50/30/20-clustered"])
def test_prefill_sweep_shape_sampled(torch, maps):
    """Bitwidth-sweep shape K=8192, N=28672, M=4096 with the maps that are all
    (or mostly) bf16-form 6/8-bit blocks, 1% outlier columns x50: 96 sampled
    rows x 512 sampled columns against the oracle."""
    K, N, M = 8192, 28672, 4096
    g = I.rng(5, len(maps))
    p = {"u6": (0, 1, 0), "u8": (0, 0, 1), "50/30/20-clustered": (0.5, 0.3, 0.2)}[maps]
    bits = I.width_map(K // 32, *p, g, clustered=maps.endswith("clustered"))
    xb = I.activations_bf16(M, bits, g, 0.01, outlier_scale=50.0)
    wb = I.normal_bf16((N, K), 0.02, g)
    planes, packed = prep(torch, xb, wb, bits)
    y = mxs.gemm_prefill(planes, bits, packed, M, N).cpu().numpy()
    rs = np.random.default_rng(3)
    rows = np.sort(rs.choice(M, 96, replace=False))
    cols = np.sort(rs.choice(N, 512, replace=False))
    ref, ab = oracle_entries(xb, wb, bits, rows, cols)
    err = U.check_gemm(y[np.ix_(rows, cols)], ref, ab)
    print(f"prefill sweep {maps}: max err/abssum {err:.2e}")


def test_prefill_bounded_wait_reports_timeout(torch):
    """A stage that is never loaded: the kernel gives up after its wait bound,
    records MXS_ERR_TIMEOUT, frees its tensor memory and the context stays usable."""
    g = I.rng(31)
    bits = I.width_map(16, 1, 0, 0, g)
    M, N = 128, 256
    xb = I.activations_bf16(M, bits, g, 0.0)
    wb = I.normal_bf16((N, 512), 0.02, g)
    planes, packed = prep(torch, xb, wb, bits)
    assert mxs.device_status(reset=True) in (0, mxs.MXS_OK, 7)
    mxs.test_prefill_starve(planes, bits, packed, M, N, stage=2)
    assert mxs.device_status(reset=True) == 7
    assert mxs.device_status() == 0
    y = mxs.gemm_prefill(planes, bits, packed, M, N).cpu().numpy()  # the context still works
    ref, ab = oracle_entries(xb, wb, bits)
    U.check_gemm(y, ref, ab)


@pytest.mark.parametrize("M,nb,p", [(256, 128, (0.8, 0.15, 0.05)), (130, 448, (0.5, 0.3, 0.2))])
def test_prefill_wide_dynamic_range(torch, M, nb, p):
    """Block scales spread over +-20 binades, so the exact results do not fit
    fp32 and the tensor core's accumulation rounding shows.  Sampled outputs
    equal, bit for bit, the replay of the kernel's MMAs under the measured
    accumulation rule (tc_model.py), and every output is within that rule's
    bound of the exact oracle.  Per MMA, each of at most 33 addends loses
    less than 2^(e-25) <= 2^-25 * (largest addend) and the final cut less
    than 2^-23 * |sum|; both are at most the dot product's sum|a_i w_i| = P
    (the accumulator holds a partial sum), so the error is below
    n_mma * (33 * 2^-25 + 2^-23) * P."""
    import tc_model as T
    from test_gpu_gemm_decode import wide_range_layer
    g = I.rng(41, M, nb)
    bits = I.width_map(nb, *p, g)
    N = 384
    xb, wb = wide_range_layer(M, N, nb, bits, g)
    planes, packed = prep(torch, xb, wb, bits)
    y = mxs.gemm_prefill(planes, bits, packed, M, N).cpu().numpy()
    a_s, a_c = mxo.quantize_bf16(xb, bits)
    w_s, w_c = mxo.quantize_bf16(wb, bits)
    ref, ab = mxo.gemm(bits, a_c, a_s, w_c, w_s)
    assert np.mean(ref.astype(np.float32).astype(np.float64) == ref) < 0.5
    rs = np.random.default_rng(nb)
    rows = np.sort(rs.choice(M, 64, replace=False))
    cols = np.sort(rs.choice(N, 64, replace=False))
    model = T.prefill_model(bits, a_c[rows], a_s[rows], w_c[cols], w_s[cols])
    assert np.array_equal(y[np.ix_(rows, cols)], model)
    n4 = int(np.sum(bits == 4))
    n_mma = 4 * ((n4 + 3) // 4) + 4 * ((bits.size - n4 + 1) // 2)
    A = np.abs(mxo.dequantize(a_c, a_s, bits))
    W = np.abs(mxo.dequantize(w_c, w_s, bits))
    pabs = A @ W.T  # sum |a_i w_i| (a bound's scale: fp64 rounding here is immaterial)
    err = np.abs(y.astype(np.float64) - ref)
    assert np.all(err <= n_mma * (33 * 2.0 ** -25 + 2.0 ** -23) * pabs * 1.001)
    print(f"prefill wide range M={M} K={32 * nb}: max err/abssum {np.max(err / ab):.2e}, "
          f"max err/sum|a w| {np.max(err / pabs):.2e} (bound {n_mma * (33 * 2.0 ** -25 + 2.0 ** -23):.2e})")
