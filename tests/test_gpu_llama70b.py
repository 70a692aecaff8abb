"""Config 3 parity: LLaMA-2-70B shapes with the per-layer width maps (4-bit
share 60 % at layer 0 rising to 95 % at layer 79, 8-bit blocks over the 1 %
outlier columns), decode (M = 1, 16) and prefill (M = 4096), on the sampled
layers 0, 40 and 79; outputs sampled so that the exact oracle stays fast."""
import numpy as np
import pytest

from oracle import mxo
from paper_2607_17733_gb300 import inputs as I
from paper_2607_17733_gb300 import mxs
import gpu_util as U

pytestmark = pytest.mark.gpu

SHAPES = {name: (K, N) for name, K, N in I.LLAMA2_70B}


@pytest.fixture(scope="module")
def torch():
    return U.torch_or_skip()


def _layer(torch, M, proj, layer, layout):
    K, N = SHAPES[proj]
    g = I.rng(3, layer, K, N, M)
    bits = I.llama70b_layer_map(K, layer, 80, g)
    xb = I.activations_bf16(M, bits, g, 0.01, outlier_scale=50.0)
    wb = I.normal_bf16((N, K), 0.015, g)
    packed = mxs.pack_weight(U.to_dev_bf16(torch, wb), bits, layout=layout)
    torch.cuda.synchronize()
    return bits, xb, wb, packed


def _check(y, xb, wb, bits, rows, cols):
    a_s, a_c = mxo.quantize_bf16(xb[rows], bits)
    w_s, w_c = mxo.quantize_bf16(wb[cols], bits)
    ref, ab = mxo.gemm(bits, a_c, a_s, w_c, w_s)
    return U.check_gemm(y[np.ix_(rows, cols)], ref, ab)


@pytest.mark.parametrize("layer", [0, 40, 79])
@pytest.mark.parametrize("proj", ["q", "k", "down"])
@pytest.mark.parametrize("M", [1, 16])
def test_decode_70b_layers(torch, M, proj, layer):
    bits, xb, wb, packed = _layer(torch, M, proj, layer, mxs.W_COMPACT)
    N = SHAPES[proj][1]
    y = mxs.linear_decode(U.to_dev_bf16(torch, xb), bits, packed, N).cpu().numpy()
    cols = np.sort(np.random.default_rng(layer).choice(N, min(N, 512), replace=False))
    _check(y, xb, wb, bits, np.arange(M), cols)


@pytest.mark.parametrize("layer", [0, 79])
@pytest.mark.parametrize("proj", ["q", "down"])
def test_prefill_70b_layers(torch, proj, layer):
    M = 4096
    bits, xb, wb, packed = _layer(torch, M, proj, layer, mxs.W_COMPACT_AND_PLANES)
    N = SHAPES[proj][1]
    _, _, planes = mxs.quantize_act(U.to_dev_bf16(torch, xb), bits, want_codes=False, want_planes=True)
    y = mxs.gemm_prefill(planes, bits, packed, M, N).cpu().numpy()
    rs = np.random.default_rng(layer + 1)
    rows = np.sort(rs.choice(M, 64, replace=False))
    cols = np.sort(rs.choice(N, 256, replace=False))
    _check(y, xb, wb, bits, rows, cols)
