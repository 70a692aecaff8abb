"""Parity on the single-layer configuration and the bitwidth-mix sweep.

Single layer: activations M=128 x K=4096 N(0,1) with 0.5 % of the columns x50,
weights 4096 x 4096 N(0,0.02), map 80/15/5 (outlier blocks 8-bit), seed 0:
codes and scales bit-exact, and the whole 128 x 4096 result element by element
against the exact oracle.

Sweep: K=8192, N=28672, M in {16, 4096}; maps uniform 4 / 6 / 8 bits and
90/5/5, 70/20/10, 50/30/20 (4/6/8 %) with the 8-bit blocks placed at random or
as one clustered run; activations N(0,1) with 1 % outlier columns x50 (inside
the 8-bit blocks, the paper's top-32-columns rule of Alg. 3), weights
N(0,0.02).  Decode (M=16, through mxs_linear_decode): every token, 1024
sampled columns.  Prefill (M=4096): 128 sampled rows x 512 sampled columns."""
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


def test_single_layer_config_full_result(torch):
    M, K, N = 128, 4096, 4096
    g = I.rng(0)
    bits = I.width_map(K // 32, 0.80, 0.15, 0.05, g)
    assert (int(np.sum(bits == 4)), int(np.sum(bits == 6)), int(np.sum(bits == 8))) == (103, 19, 6)
    xb = I.activations_bf16(M, bits, g, 0.005, outlier_scale=50.0)
    wb = I.normal_bf16((N, K), 0.02, g)
    x, w = U.to_dev_bf16(torch, xb), U.to_dev_bf16(torch, wb)
    codes, scales, planes = mxs.quantize_act(x, bits, want_planes=True)
    packed = mxs.pack_weight(w, bits, layout=mxs.W_COMPACT_AND_PLANES)
    y = mxs.gemm(codes, scales, planes, bits, packed, N, w_layout=mxs.W_COMPACT_AND_PLANES).cpu().numpy()
    a_s, a_c = mxo.quantize_bf16(xb, bits)
    w_s, w_c = mxo.quantize_bf16(wb, bits)
    pc, ps = mxo.pack_act(bits, a_s, a_c)
    assert np.array_equal(codes.cpu().numpy(), pc)
    assert np.array_equal(scales.cpu().numpy(), ps)
    assert np.array_equal(packed.cpu().numpy(), mxo.pack_weight(bits, w_s, w_c, with_planes=True))
    ref, ab = mxo.gemm(bits, a_c, a_s, w_c, w_s)
    err = U.check_gemm(y, ref, ab)
    print(f"single layer 128x4096x4096: max err/abssum {err:.2e}, "
          f"{np.mean(y.astype(np.float64) == ref):.4f} of outputs equal to the rounded exact result")


SWEEP_K, SWEEP_N = 8192, 28672
SWEEP_MAPS = {"u4": ((1, 0, 0), False), "u6": ((0, 1, 0), False), "u8": ((0, 0, 1), False),
              "90/5/5-random": ((0.9, 0.05, 0.05), False), "90/5/5-clustered": ((0.9, 0.05, 0.05), True),
              "70/20/10-random": ((0.7, 0.2, 0.1), False), "70/20/10-clustered": ((0.7, 0.2, 0.1), True),
              "50/30/20-random": ((0.5, 0.3, 0.2), False), "50/30/20-clustered": ((0.5, 0.3, 0.2), True)}


@pytest.fixture(scope="module")
def sweep_weights(torch):
    """One weight matrix for the whole sweep (the map only changes its quantization)."""
    wb = I.normal_bf16((SWEEP_N, SWEEP_K), 0.02, I.rng(4, 0))
    return wb, U.to_dev_bf16(torch, wb)


@pytest.mark.parametrize("M", [16, 4096])
@pytest.mark.parametrize("name", list(SWEEP_MAPS))
def test_bitwidth_sweep(torch, sweep_weights, name, M):
    wb, w = sweep_weights
    p, clustered = SWEEP_MAPS[name]
    g = I.rng(4, 1, list(SWEEP_MAPS).index(name), M)
    bits = I.width_map(SWEEP_K // 32, *p, g, clustered=clustered)
    if clustered:
        idx8 = np.flatnonzero(bits == 8)
        assert idx8.size > 1 and np.all(np.diff(idx8) == 1)
    xb = I.activations_bf16(M, bits, g, 0.01, outlier_scale=50.0)
    x = U.to_dev_bf16(torch, xb)
    rs = np.random.default_rng(M)
    if M <= 16:
        packed = mxs.pack_weight(w, bits)
        torch.cuda.synchronize()  # weights are static before the first decode call
        y = mxs.linear_decode(x, bits, packed, SWEEP_N).cpu().numpy()
        rows = np.arange(M)
        cols = np.sort(rs.choice(SWEEP_N, 1024, replace=False))
    else:
        packed = mxs.pack_weight(w, bits, layout=mxs.W_COMPACT_AND_PLANES)
        _, _, planes = mxs.quantize_act(x, bits, want_codes=False, want_planes=True)
        y = mxs.gemm_prefill(planes, bits, packed, M, SWEEP_N).cpu().numpy()
        rows = np.sort(rs.choice(M, 128, replace=False))
        cols = np.sort(rs.choice(SWEEP_N, 512, replace=False))
    del packed
    a_s, a_c = mxo.quantize_bf16(xb[rows], bits)
    w_s, w_c = mxo.quantize_bf16(wb[cols], bits)
    ref, ab = mxo.gemm(bits, a_c, a_s, w_c, w_s)
    err = U.check_gemm(y[np.ix_(rows, cols)], ref, ab)
    print(f"sweep {name} M={M}: max err/abssum {err:.2e}")
