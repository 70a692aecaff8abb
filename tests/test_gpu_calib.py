"""Offline allocation on the GPU against the oracle: column sensitivity
(Alg. 1) componentwise, the column order of Alg. 3 exactly on identical keys,
the block widths exactly, and an end-to-end allocation checked for validity
against the oracle's sensitivities.

Tolerance of the column sums: a lane adds 16 rows of exact squares in fp32
(at most 16 roundings of a sum of positive terms: relative error <= 16 *
2^-24 = 2^-20 ~ 9.5e-7) and adds the runs in fp64, so every column is within
2^-20 (+ fp64 noise) of the exact sum; the tests use 1e-6.

The permuted quantizer and packer (the allocation's column order applied on
the inference path) are compared byte for byte with the oracle's
quantization of x[:, perm] and w[:, perm], and one layer runs end to end:
calibration sums, allocation, permuted packing and quantization, GEMM."""
import numpy as np
import pytest

from oracle import alloc as A
from oracle import mxo
from paper_2607_17733_gb300 import inputs as I
from paper_2607_17733_gb300 import mxs
import gpu_util as U

pytestmark = pytest.mark.gpu
REL = 1e-6


@pytest.fixture(scope="module")
def torch():
    return U.torch_or_skip()


def calib_activations(T, K, seed, outlier_frac=0.01, scale=50.0):
    """Synthetic calibration batch: N(0,1) with a random 1 % of the columns x50
    (systematic outlier channels, Sec. 3.1), rounded once to bf16."""
    g = I.rng(11, T, K, seed)
    x = g.standard_normal((T, K)).astype(np.float32)
    cols = g.choice(K, size=max(1, int(round(outlier_frac * K))), replace=False)
    x[:, cols] *= scale
    return I.f32_to_bf16_bits(x)


def gpu_sensitivity(torch, xb, ld=None, s=None, accumulate=False):
    T, K = xb.shape
    if ld is not None:
        wide = np.zeros((T, ld), np.uint16)
        wide[:, :K] = xb
        x = U.to_dev_bf16(torch, wide)[:, :K]
    else:
        x = U.to_dev_bf16(torch, xb) if T > 0 else torch.empty((0, K), dtype=torch.bfloat16, device="cuda")
    s = mxs.column_sensitivity(x, s=s, accumulate=accumulate)
    torch.cuda.synchronize()
    return s


def check_close(got, want):
    got = np.asarray(got, np.float64)
    err = np.abs(got - want)
    assert np.all(err <= REL * np.abs(want)), f"max rel err {np.max(err / np.maximum(np.abs(want), 1e-300)):.3g}"


@pytest.mark.parametrize("T,K,ld", [(1, 32, None), (7, 96, None), (33, 64, 72), (1000, 4096, None),
                                    (257, 14336, 14336 + 64), (4099, 1024, None)])
def test_column_sensitivity_matches_oracle(torch, T, K, ld):
    xb = calib_activations(T, K, seed=T)
    check_close(gpu_sensitivity(torch, xb, ld).cpu().numpy(), A.column_sensitivity(xb))


def test_empty_batch_writes_zeros_or_keeps_the_sum(torch):
    K = 128
    s = gpu_sensitivity(torch, np.zeros((0, K), np.uint16))
    assert np.array_equal(s.cpu().numpy(), np.zeros(K))
    s.fill_(3.0)
    s = gpu_sensitivity(torch, np.zeros((0, K), np.uint16), s=s, accumulate=True)
    assert np.array_equal(s.cpu().numpy(), np.full(K, 3.0))


def test_accumulates_over_calibration_samples(torch):
    """Alg. 1: H += X^T X for every sample."""
    batches = [calib_activations(T, 4096, seed=100 + T) for T in (512, 3, 1031)]
    s = None
    for i, xb in enumerate(batches):
        s = gpu_sensitivity(torch, xb, s=s, accumulate=i > 0)
    check_close(s.cpu().numpy(), sum(A.column_sensitivity(xb) for xb in batches))


def test_tiny_huge_and_zero_columns(torch):
    """Squares that under- or overflow fp32 (|x| < 2^-63 or >= 2^64) are added in fp64."""
    T, K = 300, 256
    g = np.random.default_rng(9)
    x = g.standard_normal((T, K)).astype(np.float32)
    x[:, 0] = 0.0
    x[:, 1] *= 2.0 ** -100
    x[:, 2] *= 2.0 ** 70
    x[:, 3] = np.ldexp(np.float32(1), -133) * (np.arange(T) % 7)  # bf16 subnormals
    x[:5, 4] = 2.0 ** 70  # a few huge rows in an ordinary column
    xb = I.f32_to_bf16_bits(x)
    got = gpu_sensitivity(torch, xb).cpu().numpy()
    want = A.column_sensitivity(xb)
    assert got[0] == 0.0
    check_close(got[1:], want[1:])


@pytest.mark.parametrize("K", [32, 96, 4096, 65536])
def test_column_order_is_exact_on_identical_keys(torch, K):
    """The GPU order of the same fp64 keys equals the oracle's stable descending argsort."""
    g = np.random.default_rng(K)
    keys = g.integers(0, max(4, K // 8), size=K).astype(np.float64) * 0.5  # many ties
    keys[g.choice(K, size=min(K, 8), replace=False)] = -0.0
    keys[g.choice(K, size=min(K, 8), replace=False)] = 0.0
    s = torch.from_numpy(keys).cuda()
    perm, bits, n6 = mxs.allocate_layer(s, R=0.5, s_layer=0.5)
    torch.cuda.synchronize()
    want_perm, want_bits, want_n6 = A.allocate_layer(keys, 0.5, 0.5)
    assert np.array_equal(perm.cpu().numpy(), want_perm)
    assert np.array_equal(bits, want_bits) and n6 == want_n6


@pytest.mark.parametrize("K,R,sl", [(256, 0.5, 0.5), (256, 3.0, 1.0), (4096, 0.11, 0.8), (14336, 0.0, 0.3),
                                    (32, 1.0, 1.0)])
def test_block_widths_match_oracle(torch, K, R, sl):
    s = torch.rand(K, dtype=torch.float64, device="cuda")
    perm, bits, n6 = mxs.allocate_layer(s, R, sl)
    torch.cuda.synchronize()
    _, want_bits, want_n6 = A.allocate_layer(s.cpu().numpy(), R, sl)
    assert np.array_equal(bits, want_bits) and n6 == want_n6


def test_end_to_end_allocation_is_valid(torch):
    """Sensitivities and order both on the GPU, for four LLaMA-shaped layers at
    B = 4.5: the order is a permutation that sorts the oracle's sensitivities
    (within the sum tolerance), the 8-bit block is the oracle's top 32 where
    the gap at rank 32 exceeds it, and the average width is at most B."""
    d_in = [4096, 4096, 14336, 1024]
    s_layer = [1.0, 0.4, 0.7, 0.1]
    R = mxs.allocation_r(d_in, s_layer, 4.5)
    maps = []
    for li, (K, sl) in enumerate(zip(d_in, s_layer)):
        xb = calib_activations(768, K, seed=li)
        s = gpu_sensitivity(torch, xb)
        perm, bits, _ = mxs.allocate_layer(s, R, sl)
        torch.cuda.synchronize()
        perm = perm.cpu().numpy()
        ref = A.column_sensitivity(xb)
        assert np.array_equal(np.sort(perm), np.arange(K))
        ordered = ref[perm]
        assert np.all(ordered[1:] <= ordered[:-1] * (1 + 2 * REL))
        top = np.sort(ref)[::-1]
        if top[31] > top[32] * (1 + 2 * REL):
            assert set(perm[:32]) == set(A.column_order(ref)[:32])
        maps.append(bits)
    assert A.average_width(maps, d_in) <= 4.5 + 1e-12


# ---------------------------------------------------------------- the allocation on the inference path

def _random_perm(torch, K, seed):
    g = np.random.default_rng(seed)
    p = g.permutation(K).astype(np.int32)
    return p, torch.from_numpy(p).cuda()


@pytest.mark.parametrize("M,nb,p", [(1, 4, (0.5, 0.25, 0.25)), (7, 37, (0.7, 0.2, 0.1)), (129, 128, (0.8, 0.15, 0.05))])
@pytest.mark.parametrize("rounding", [mxs.RNE, mxs.RHAZ])
def test_permuted_quantize_matches_oracle_of_permuted_x(torch, M, nb, p, rounding):
    """mxs_quantize_act_permuted(x, perm) is byte for byte the quantization of x[:, perm]."""
    g = I.rng(21, M, nb)
    bits = I.width_map(nb, *p, g)
    K = 32 * nb
    xb = calib_activations(M, K, seed=nb)
    perm, perm_d = _random_perm(torch, K, seed=M)
    codes, scales, planes = mxs.quantize_act(U.to_dev_bf16(torch, xb), bits, rounding=rounding, want_planes=True,
                                             perm=perm_d)
    torch.cuda.synchronize()
    a_s, a_c = mxo.quantize_bf16(np.ascontiguousarray(xb[:, perm]), bits, rounding)
    pc, ps = mxo.pack_act(bits, a_s, a_c)
    assert np.array_equal(codes.cpu().numpy(), pc) and np.array_equal(scales.cpu().numpy(), ps)
    pl, sf = mxo.planes(bits, a_s, a_c, bf16_68=True)
    kp = pl.shape[1]
    got = planes.cpu().numpy()
    assert np.array_equal(got[:M * kp].reshape(M, kp), pl)
    # scale tiles [tile][stage][i<32][w<4][q<4] = row 128*tile + 32w + i; rows >= M are not written
    off = (M * kp + 255) // 256 * 256
    tiles = got[off:off + sf.size].reshape(-1, kp // 128, 32, 4, 4)
    rows = 128 * np.arange(tiles.shape[0])[:, None, None, None, None] + 32 * np.arange(4)[None, None, None, :, None] \
        + np.arange(32)[None, None, :, None, None]
    valid = np.broadcast_to(rows < M, tiles.shape)
    assert np.array_equal(tiles[valid], sf.reshape(tiles.shape)[valid])


@pytest.mark.parametrize("N,nb", [(200, 40), (37, 5)])
@pytest.mark.parametrize("layout", [mxs.W_COMPACT, mxs.W_COMPACT_AND_PLANES])
def test_permuted_pack_matches_oracle_of_permuted_w(torch, N, nb, layout):
    g = I.rng(22, N, nb)
    bits = I.width_map(nb, 0.6, 0.25, 0.15, g)
    K = 32 * nb
    wb = I.normal_bf16((N, K), 0.02, g)
    perm, perm_d = _random_perm(torch, K, seed=N)
    got = mxs.pack_weight(U.to_dev_bf16(torch, wb), bits, layout=layout, perm=perm_d)
    torch.cuda.synchronize()
    w_s, w_c = mxo.quantize_bf16(np.ascontiguousarray(wb[:, perm]), bits)
    want = mxo.pack_weight(bits, w_s, w_c, with_planes=layout == mxs.W_COMPACT_AND_PLANES)
    assert np.array_equal(got.cpu().numpy()[:want.size], want)


@pytest.mark.parametrize("M", [1, 16, 256])
def test_mxsens_layer_end_to_end(torch, M):
    """The method on one layer: calibration sums (Alg. 1), the allocation (Alg.
    3, Theorem 1's R at B = 4.5 for this layer alone) giving the column order
    and block widths, weights packed and activations quantized in that order,
    and the GEMM (decode for M <= 16, tensor-core prefill above) -- against the
    oracle computing the same allocation from its own sums and the exact GEMM
    of the permuted, quantized operands.  The allocation is taken from the GPU
    and checked valid against the oracle's sums (near-ties may order
    differently within the sum tolerance); the GEMM is then compared for that
    allocation."""
    K, N = 4096, 1024
    calib = calib_activations(2048, K, seed=77)
    s = gpu_sensitivity(torch, calib)
    R = mxs.allocation_r([K], [1.0], 4.5)
    perm_d, bits, n6 = mxs.allocate_layer(s, R, 1.0)
    torch.cuda.synchronize()
    perm = perm_d.cpu().numpy()
    ref = A.column_sensitivity(calib)
    ordered = ref[perm]
    assert np.all(ordered[1:] <= ordered[:-1] * (1 + 2 * REL))
    _, want_bits, want_n6 = A.allocate_layer(ref, A.allocation_r([K], [1.0], 4.5), 1.0)
    assert np.array_equal(bits, want_bits) and n6 == want_n6

    g = I.rng(23, M)
    x = g.standard_normal((M, K)).astype(np.float32)
    x[:, np.argsort(-ref)[:16]] *= 50.0  # the calibration's outlier channels stay outliers
    xb = I.f32_to_bf16_bits(x)
    wb = I.normal_bf16((N, K), 0.02, g)
    layout = mxs.W_COMPACT if M <= 16 else mxs.W_COMPACT_AND_PLANES
    packed = mxs.pack_weight(U.to_dev_bf16(torch, wb), bits, layout=layout, perm=perm_d)
    _, _, planes = mxs.quantize_act(U.to_dev_bf16(torch, xb), bits, want_codes=False, want_planes=True, perm=perm_d)
    torch.cuda.synchronize()
    if M <= 16:
        y = mxs.gemm_decode(None, None, bits, packed, N, planes=planes, M=M)
    else:
        y = mxs.gemm_prefill(planes, bits, packed, M, N)
    a_s, a_c = mxo.quantize_bf16(np.ascontiguousarray(xb[:, perm]), bits)
    w_s, w_c = mxo.quantize_bf16(np.ascontiguousarray(wb[:, perm]), bits)
    yr, abssum = mxo.gemm(bits, a_c, a_s, w_c, w_s)
    U.check_gemm(y.cpu().numpy(), yr, abssum)
