"""A1/A2 parity: the CUDA quantizer and weight packer against the CPU oracle,
byte for byte (codes, scales, MMA planes, scale tiles, packed weights)."""
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


def run_quantize(torch, xb, bits, rounding=mxs.RNE, planes=True, ld=None):
    M, K = xb.shape
    if ld is not None:  # strided source rows
        wide = np.zeros((M, ld), np.uint16)
        wide[:, :K] = xb
        xd = U.to_dev_bf16(torch, wide)[:, :K]
    else:
        xd = U.to_dev_bf16(torch, xb)
    codes, scales, pl = mxs.quantize_act(xd, bits, rounding=rounding, want_planes=planes)
    torch.cuda.synchronize()
    return codes.cpu().numpy(), scales.cpu().numpy(), None if pl is None else pl.cpu().numpy()


def oracle_quantize(xb, bits, rounding=mxo.RNE):
    s, c = mxo.quantize_bf16(xb, bits, rounding)
    pc, ps = mxo.pack_act(bits, s, c)
    pl, sf = mxo.planes(bits, s, c, bf16_68=True)  # 6/8-bit blocks as bf16 values, the operand of both GEMMs
    return pc, ps, pl, sf


def compare(torch, xb, bits, rounding=mxs.RNE, ld=None):
    codes, scales, planes = run_quantize(torch, xb, bits, rounding, True, ld)
    pc, ps, pl, sf = oracle_quantize(xb, bits, rounding)
    assert np.array_equal(codes, pc), "codes"
    assert np.array_equal(scales, ps), "scales"
    M = xb.shape[0]
    kp = pl.shape[1]
    off = (M * kp + 255) // 256 * 256
    assert np.array_equal(planes[:M * kp].reshape(M, kp), pl), "planes"
    # scale tiles: [tile][stage][i<32][w<4][q<4] = row 128*tile + 32w + i; rows >= M are not written
    got = planes[off:off + sf.size].reshape(-1, kp // 128, 32, 4, 4)
    want = sf.reshape(got.shape)
    rows = 128 * np.arange(got.shape[0])[:, None, None, None, None] + 32 * np.arange(4)[None, None, None, :, None] \
        + np.arange(32)[None, None, :, None, None]
    valid = np.broadcast_to(rows < M, got.shape)
    assert np.array_equal(got[valid], want[valid]), "scale tiles"
    # the alignment gaps between and after the two sections are not written


@pytest.mark.parametrize("rounding", [mxs.RNE, mxs.RHAZ])
def test_single_layer_config(torch, rounding):
    """M=128, K=4096, map 80/15/5, 0.5% outlier columns x50."""
    g = I.rng(0, 0)
    bits = I.width_map(128, 0.80, 0.15, 0.05, g)
    xb = I.activations_bf16(128, bits, g, 0.005, outlier_scale=50.0)
    compare(torch, xb, bits, rounding)


@pytest.mark.parametrize("M,nb,p", [(1, 1, (1, 0, 0)), (3, 5, (0.4, 0.3, 0.3)), (37, 70, (0.7, 0.2, 0.1)),
                                    (129, 33, (0.5, 0.25, 0.25)), (200, 9, (0, 0, 1)), (17, 12, (0, 1, 0))])
@pytest.mark.parametrize("rounding", [mxs.RNE, mxs.RHAZ])
def test_ragged_shapes_and_maps(torch, M, nb, p, rounding):
    g = I.rng(M, nb)
    bits = I.width_map(nb, *p, g)
    xb = I.activations_bf16(M, bits, g, 0.02, student_t=True)
    compare(torch, xb, bits, rounding)


def test_strided_rows(torch):
    g = I.rng(3, 3)
    bits = I.width_map(16, 0.6, 0.2, 0.2, g)
    xb = I.activations_bf16(9, bits, g, 0.03, outlier_scale=30.0)
    compare(torch, xb, bits, ld=512 + 8)


def test_special_blocks(torch):
    """zero, subnormal, huge, Inf/NaN and tie-heavy blocks."""
    nb = 8
    bits = np.array([4, 6, 8, 4, 6, 8, 4, 8], np.uint8)
    rows = []
    f = np.float32
    z = np.zeros(32 * nb, f)
    rows.append(z.copy())
    sub = z.copy()
    sub[:] = np.ldexp(f(1), -133) * (np.arange(32 * nb) % 7)
    rows.append(sub)
    big = z.copy()
    big[::5] = f(3.3e38)
    big[1::5] = f(-1e38)
    rows.append(big)
    spec = np.linspace(-3, 3, 32 * nb).astype(f)
    spec[3], spec[40], spec[70], spec[200] = np.inf, -np.inf, np.nan, np.nan
    rows.append(spec)
    ties = np.tile((np.arange(32) - 16 + 0.5).astype(f) * f(0.25), nb)
    rows.append(ties)
    xb = I.f32_to_bf16_bits(np.stack([np.nan_to_num(r, nan=0.0, posinf=0, neginf=0) for r in rows]))
    # put the exact non-finite bit patterns back (the generator rounds finite values only)
    xb[3, 3], xb[3, 40], xb[3, 70], xb[3, 200] = 0x7F80, 0xFF80, 0x7FC0, 0xFFC1
    for rounding in (mxs.RNE, mxs.RHAZ):
        compare(torch, xb, bits, rounding)


@pytest.mark.parametrize("M,K", [(2048, 4096), (2048, 14336), (4096, 28672)])
def test_prefill_shapes_full_size(torch, M, K):
    g = I.rng(2, K)
    bits = I.width_map(K // 32, 0.80, 0.15, 0.05, g)
    xb = I.activations_bf16(M, bits, g, 0.005, student_t=True)
    compare(torch, xb, bits)


@pytest.mark.parametrize("M,K", [(1219, 4096), (601, 8192), (153, 17408), (157, 28672), (4871, 1024)])
@pytest.mark.parametrize("rounding", [mxs.RNE, mxs.RHAZ])
def test_many_rows_with_special_blocks(torch, M, K, rounding):
    """Many rows (several CTAs per row and rows per grid column, ragged last
    scale tile) with Inf/NaN, all-zero, subnormal and tie blocks planted among
    ordinary ones; odd M also reads strided source rows."""
    g = I.rng(7, K, M)
    bits = I.width_map(K // 32, 0.7, 0.2, 0.1, g)
    xb = I.activations_bf16(M, bits, g, 0.01, student_t=True)
    xb[1] = 0
    xb[2, :] = I.f32_to_bf16_bits((np.ldexp(np.float32(1), -133) * (np.arange(K) % 5)).astype(np.float32))
    xb[M - 1, 7], xb[M - 1, 300] = 0x7F80, 0xFFC1
    xb[M // 2] = I.f32_to_bf16_bits(np.tile((np.arange(32) - 16 + 0.5).astype(np.float32) * 0.25, K // 32))
    compare(torch, xb, bits, rounding, ld=K + 64 if M % 2 else None)


# ---------------------------------------------------------------- weights
@pytest.mark.parametrize("N,nb,p", [(16, 4, (0.5, 0.25, 0.25)), (37, 11, (0.6, 0.2, 0.2)),
                                    (200, 128, (0.8, 0.15, 0.05)), (1, 3, (0, 0, 1)), (300, 7, (1, 0, 0))])
@pytest.mark.parametrize("layout", [mxs.W_COMPACT, mxs.W_COMPACT_AND_PLANES])
def test_pack_weight_bit_exact(torch, N, nb, p, layout):
    g = I.rng(N, nb, 5)
    bits = I.width_map(nb, *p, g)
    wb = I.normal_bf16((N, 32 * nb), 0.02, g)
    packed = mxs.pack_weight(U.to_dev_bf16(torch, wb), bits, layout=layout)
    torch.cuda.synchronize()
    s, c = mxo.quantize_bf16(wb, bits)
    assert np.array_equal(packed.cpu().numpy(), mxo.pack_weight(bits, s, c, layout == mxs.W_COMPACT_AND_PLANES))


def test_pack_weight_full_size_sampled(torch):
    """gate/up of the 8B shapes: every byte of the packed buffer."""
    g = I.rng(1, 14336)
    bits = I.width_map(128, 0.85, 0.10, 0.05, g)
    wb = I.normal_bf16((14336, 4096), 0.02, g)
    packed = mxs.pack_weight(U.to_dev_bf16(torch, wb), bits, layout=mxs.W_COMPACT_AND_PLANES)
    torch.cuda.synchronize()
    s, c = mxo.quantize_bf16(wb, bits)
    assert np.array_equal(packed.cpu().numpy(), mxo.pack_weight(bits, s, c, True))


@pytest.mark.parametrize("M,rounding", [(5, mxs.RNE), (300, mxs.RNE), (300, mxs.RHAZ)])
def test_quantize_group_matches_single_launches(torch, M, rounding):
    """mxs_quantize_act_group writes, for every problem, the same planes and
    scale tiles as mxs_quantize_act of that problem alone (three widths maps
    and K's)."""
    shapes = [(4096, (0.8, 0.15, 0.05)), (1024, (0.5, 0.3, 0.2)), (2080, (0.9, 0.05, 0.05))]
    probs, singles, xbs = [], [], []
    for i, (K, p) in enumerate(shapes):
        g = I.rng(90, M, K, i)
        bits = I.width_map(K // 32, *p, g)
        xb = I.activations_bf16(M, bits, g, 0.01, outlier_scale=40.0)
        x = U.to_dev_bf16(torch, xb)
        pl = torch.full((mxs.act_planes_bytes(M, K, bits),), 0xAB, dtype=torch.uint8, device="cuda")
        probs.append((x, bits, pl))
        xbs.append(xb)
        _, _, one = mxs.quantize_act(x, bits, rounding=rounding, want_codes=False, want_planes=True)
        singles.append(one)
    mxs.quantize_act_group(probs, rounding=rounding)
    torch.cuda.synchronize()
    for (x, bits, pl), one, xb in zip(probs, singles, xbs):
        K = x.shape[1]
        kp = mxo.plane_shape(bits)[0]
        got, want = pl.cpu().numpy(), one.cpu().numpy()
        assert np.array_equal(got[:M * kp], want[:M * kp])
        off = (M * kp + 255) // 256 * 256
        nst = kp // 128
        tiles_g = got[off:off + ((M + 127) // 128) * nst * 512].reshape(-1, nst, 32, 4, 4)
        tiles_w = want[off:off + ((M + 127) // 128) * nst * 512].reshape(-1, nst, 32, 4, 4)
        rows = 128 * np.arange(tiles_g.shape[0])[:, None, None, None, None] + 32 * np.arange(4)[None, None, None, :, None] \
            + np.arange(32)[None, None, :, None, None]
        valid = np.broadcast_to(rows < M, tiles_g.shape)
        assert np.array_equal(tiles_g[valid], tiles_w[valid])
        # and the oracle agrees
        s_, c_ = mxo.quantize_bf16(xb, bits, mxo.RHAZ if rounding == mxs.RHAZ else mxo.RNE)
        pl_o, _ = mxo.planes(bits, s_, c_, bf16_68=True)
        assert np.array_equal(got[:M * kp].reshape(M, kp), pl_o)
