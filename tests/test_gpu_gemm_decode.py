"""A4 parity: the decode GEMM (M <= 16) against the exact CPU oracle."""
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


def layer(torch, M, K, N, bits, g, w_sigma=0.02, outlier_frac=0.01, outlier_scale=30.0):
    xb = I.activations_bf16(M, bits, g, outlier_frac, outlier_scale=outlier_scale)
    wb = I.normal_bf16((N, K), w_sigma, g)
    codes, scales, _ = mxs.quantize_act(U.to_dev_bf16(torch, xb), bits)
    packed = mxs.pack_weight(U.to_dev_bf16(torch, wb), bits)
    torch.cuda.synchronize()  # weights are static: packed before the first linear_decode
    return xb, wb, codes, scales, packed


def decode_from(torch, src, xb, bits, packed, N, codes=None, scales=None):
    """The decode kernel over packed codes, or over the MMA planes of the same
    activations (TMA-loaded token operand)."""
    M = xb.shape[0]
    if src == "codes":
        return mxs.gemm(codes, scales, None, bits, packed, N)
    _, _, planes = mxs.quantize_act(U.to_dev_bf16(torch, xb), bits, want_codes=False, want_planes=True)
    return mxs.gemm_decode(None, None, bits, packed, N, planes=planes, M=M)


def oracle_full(xb, wb, bits):
    a_s, a_c = mxo.quantize_bf16(xb, bits)
    w_s, w_c = mxo.quantize_bf16(wb, bits)
    return mxo.gemm(bits, a_c, a_s, w_c, w_s)


@pytest.mark.parametrize("M", [1, 2, 4, 7, 8, 9, 16])
@pytest.mark.parametrize("N,nb", [(16, 1), (37, 5), (200, 40), (1000, 128)])
def test_decode_small(torch, M, N, nb):
    g = I.rng(M, N, nb)
    bits = I.width_map(nb, 0.7, 0.2, 0.1, g)
    xb, wb, codes, scales, packed = layer(torch, M, 32 * nb, N, bits, g)
    y = mxs.gemm(codes, scales, None, bits, packed, N).cpu().numpy()
    ref, ab = oracle_full(xb, wb, bits)
    U.check_gemm(y, ref, ab)
    # the same products in the same order over the planes: the same bits
    y_planes = decode_from(torch, "planes", xb, bits, packed, N).cpu().numpy()
    assert np.array_equal(y_planes, y, equal_nan=True)


@pytest.mark.parametrize("M", [1, 5, 16])
@pytest.mark.parametrize("N,nb,p", [(130, 3, (1, 0, 0)), (129, 7, (0, 0.5, 0.5)), (640, 61, (0.7, 0.2, 0.1)),
                                    (256, 333, (0.9, 0.05, 0.05))])
def test_decode_from_planes_ragged(torch, M, N, nb, p):
    """Ragged stage counts (n4 % 4, n68 % 2 != 0), ragged N, K split over
    cluster ranks: the planes path against the oracle."""
    g = I.rng(60, M, N, nb)
    bits = I.width_map(nb, *p, g)
    xb = I.activations_bf16(M, bits, g, 0.01, outlier_scale=30.0)
    wb = I.normal_bf16((N, 32 * nb), 0.02, g)
    packed = mxs.pack_weight(U.to_dev_bf16(torch, wb), bits)
    y = decode_from(torch, "planes", xb, bits, packed, N).cpu().numpy()
    ref, ab = oracle_full(xb, wb, bits)
    U.check_gemm(y, ref, ab)


@pytest.mark.parametrize("p", [(1, 0, 0), (0, 1, 0), (0, 0, 1), (0.5, 0.3, 0.2)])
def test_decode_uniform_and_mixed_maps(torch, p):
    g = I.rng(7, int(10 * p[0]))
    bits = I.width_map(96, *p, g)
    xb, wb, codes, scales, packed = layer(torch, 16, 3072, 300, bits, g)
    y = mxs.gemm(codes, scales, None, bits, packed, 300)
    ref, ab = oracle_full(xb, wb, bits)
    U.check_gemm(y.cpu().numpy(), ref, ab)


def test_decode_output_stride_and_determinism(torch):
    g = I.rng(8, 8)
    bits = I.width_map(64, 0.8, 0.15, 0.05, g)
    xb, wb, codes, scales, packed = layer(torch, 5, 2048, 130, bits, g)
    y = torch.full((5, 160), -7.0, device="cuda")
    mxs.gemm(codes, scales, None, bits, packed, 130, y=y[:, :130])
    y2 = mxs.gemm(codes, scales, None, bits, packed, 130)
    torch.cuda.synchronize()
    yh = y.cpu().numpy()
    assert np.all(yh[:, 130:] == -7.0)
    assert np.array_equal(yh[:, :130], y2.cpu().numpy())
    ref, ab = oracle_full(xb, wb, bits)
    U.check_gemm(yh[:, :130], ref, ab)


def test_decode_nan_block(torch):
    bits = np.array([4, 8, 6, 4], np.uint8)
    g = I.rng(9)
    xb = I.activations_bf16(3, bits, g, 0.0)
    xb[1, 40] = 0x7FC0  # NaN in block 1 of token 1
    wb = I.normal_bf16((20, 128), 0.02, g)
    codes, scales, _ = mxs.quantize_act(U.to_dev_bf16(torch, xb), bits)
    packed = mxs.pack_weight(U.to_dev_bf16(torch, wb), bits)
    y = mxs.gemm(codes, scales, None, bits, packed, 20).cpu().numpy()
    ref, ab = oracle_full(xb, wb, bits)
    assert np.all(np.isnan(y[1])) and not np.isnan(y[[0, 2]]).any()
    U.check_gemm(y, ref, ab)


LLAMA3 = {name: (K, N) for name, K, N in I.LLAMA3_8B}


@pytest.mark.parametrize("src", ["codes", "planes"])
@pytest.mark.parametrize("proj", ["q", "k", "o", "gate", "down"])
@pytest.mark.parametrize("M", [1, 4, 16])
def test_decode_llama3_8b_full_size(torch, proj, M, src):
    """8B decode projections at full size; map 85/10/5, 1% outlier columns x30.
    Every output is checked for M=1/4, 2048 sampled columns for M=16."""
    K, N = LLAMA3[proj]
    g = I.rng(1, K, N, M)
    bits = I.width_map(K // 32, 0.85, 0.10, 0.05, g)
    xb, wb, codes, scales, packed = layer(torch, M, K, N, bits, g)
    y = decode_from(torch, src, xb, bits, packed, N, codes, scales).cpu().numpy()
    a_s, a_c = mxo.quantize_bf16(xb, bits)
    cols = np.arange(N) if M < 16 or N <= 2048 else np.sort(np.random.default_rng(0).choice(N, 2048, replace=False))
    w_s, w_c = mxo.quantize_bf16(wb[cols], bits)
    ref, ab = mxo.gemm(bits, a_c, a_s, w_c, w_s)
    U.check_gemm(y[:, cols], ref, ab)


@pytest.mark.parametrize("maps", ["u4", "u8", "90/5/5", "50/30/20-clustered"])
def test_decode_sweep_70b_shape_sampled(torch, maps):
    """K=8192, N=28672, M=16 (bitwidth sweep shape), 1% outliers x50; 512 columns."""
    K, N, M = 8192, 28672, 16
    g = I.rng(4, len(maps))
    p = {"u4": (1, 0, 0), "u8": (0, 0, 1), "90/5/5": (0.9, 0.05, 0.05),
         "50/30/20-clustered": (0.5, 0.3, 0.2)}[maps]
    bits = I.width_map(K // 32, *p, g, clustered=maps.endswith("clustered"))
    xb, wb, codes, scales, packed = layer(torch, M, K, N, bits, g, outlier_scale=50.0)
    y = mxs.gemm(codes, scales, None, bits, packed, N).cpu().numpy()
    assert np.array_equal(decode_from(torch, "planes", xb, bits, packed, N).cpu().numpy(), y)
    cols = np.sort(np.random.default_rng(1).choice(N, 512, replace=False))
    a_s, a_c = mxo.quantize_bf16(xb, bits)
    w_s, w_c = mxo.quantize_bf16(wb[cols], bits)
    ref, ab = mxo.gemm(bits, a_c, a_s, w_c, w_s)
    U.check_gemm(y[:, cols], ref, ab)


def wide_range_layer(M, N, nb, bits, g, spread=20):
    """Blocks scaled by random powers of two over 2*spread binades: the exact
    results no longer fit fp32, so the kernels' accumulation rounding shows."""
    xb = I.activations_bf16(M, bits, g, 0.0)
    wb = I.normal_bf16((N, 32 * nb), 0.02, g)
    xf = I.bf16_bits_to_f32(xb).reshape(M, nb, 32)
    wf = I.bf16_bits_to_f32(wb).reshape(N, nb, 32)
    xf = xf * np.exp2(g.integers(-spread, spread + 1, size=(M, nb, 1))).astype(np.float32)
    wf = wf * np.exp2(g.integers(-spread, spread + 1, size=(N, nb, 1))).astype(np.float32)
    return I.f32_to_bf16_bits(xf.reshape(M, -1)), I.f32_to_bf16_bits(wf.reshape(N, -1))


@pytest.mark.parametrize("M,nb,p", [(1, 128, (0.85, 0.10, 0.05)), (16, 448, (0.8, 0.15, 0.05)),
                                    (5, 64, (0, 0, 1))])
def test_decode_wide_dynamic_range(torch, M, nb, p):
    g = I.rng(40, M, nb)
    bits = I.width_map(nb, *p, g)
    N = 300
    xb, wb = wide_range_layer(M, N, nb, bits, g)
    codes, scales, _ = mxs.quantize_act(U.to_dev_bf16(torch, xb), bits)
    packed = mxs.pack_weight(U.to_dev_bf16(torch, wb), bits)
    y = mxs.gemm(codes, scales, None, bits, packed, N).cpu().numpy()
    assert np.array_equal(decode_from(torch, "planes", xb, bits, packed, N).cpu().numpy(), y)
    ref, ab = oracle_full(xb, wb, bits)
    assert np.mean(ref.astype(np.float32).astype(np.float64) == ref) < 0.5  # rounding really happens
    err = U.check_gemm(y, ref, ab)
    print(f"decode wide range M={M} K={32 * nb}: max err/abssum {err:.2e}")


@pytest.mark.parametrize("M", [1, 3, 8, 16])
@pytest.mark.parametrize("N,nb,p", [(37, 5, (0.6, 0.2, 0.2)), (1000, 128, (0.85, 0.10, 0.05)),
                                    (64, 448, (0.8, 0.15, 0.05)), (300, 896, (0.5, 0.3, 0.2))])
def test_fused_linear_decode(torch, M, N, nb, p):
    """Quantize-to-planes + GEMM in one call (the GEMM a programmatic dependent
    of the quantizer): same y as quantize + GEMM over the codes (bit for bit)
    and within the bar of the oracle."""
    g = I.rng(50, M, N, nb)
    bits = I.width_map(nb, *p, g)
    xb, wb, codes, scales, packed = layer(torch, M, 32 * nb, N, bits, g)
    y_fused = mxs.linear_decode(U.to_dev_bf16(torch, xb), bits, packed, N).cpu().numpy()
    y_two = mxs.gemm(codes, scales, None, bits, packed, N).cpu().numpy()
    assert np.array_equal(y_fused, y_two)
    ref, ab = oracle_full(xb, wb, bits)
    U.check_gemm(y_fused, ref, ab)


def test_fused_linear_decode_rhaz_and_stride(torch):
    g = I.rng(51)
    bits = I.width_map(64, 0.7, 0.2, 0.1, g)
    M, K, N = 6, 2048, 100
    xb = I.activations_bf16(M, bits, g, 0.02, outlier_scale=50.0)
    wb = I.normal_bf16((N, K), 0.02, g)
    wide = np.zeros((M, K + 64), np.uint16)
    wide[:, :K] = xb
    x = U.to_dev_bf16(torch, wide)[:, :K]
    packed = mxs.pack_weight(U.to_dev_bf16(torch, wb), bits, rounding=mxs.RHAZ)
    torch.cuda.synchronize()
    y = mxs.linear_decode(x, bits, packed, N, rounding=mxs.RHAZ).cpu().numpy()
    a_s, a_c = mxo.quantize_bf16(xb, bits, mxo.RHAZ)
    w_s, w_c = mxo.quantize_bf16(wb, bits, mxo.RHAZ)
    ref, ab = mxo.gemm(bits, a_c, a_s, w_c, w_s)
    U.check_gemm(y, ref, ab)


@pytest.mark.parametrize("M", [1, 5, 16])
@pytest.mark.parametrize("shapes", [[(4096, 4096), (4096, 1024), (4096, 1024)], [(4096, 14336), (4096, 14336)],
                                    [(512, 200), (1024, 37)], [(14336, 4096)]])
def test_linear_decode_group(torch, M, shapes):
    """Projections that share an input in one grouped launch (q/k/v, gate/up shapes and
    ragged ones): every problem against the oracle, and against its own single launch
    within the GEMM bound (the K split may differ)."""
    probs, refs = [], []
    for i, (K, N) in enumerate(shapes):
        g = I.rng(61, M, K, N, i)
        bits = I.width_map(K // 32, 0.8, 0.15, 0.05, g)
        xb = I.activations_bf16(M, bits, g, 0.01, outlier_scale=30.0)
        wb = I.normal_bf16((N, K), 0.02, g)
        packed = mxs.pack_weight(U.to_dev_bf16(torch, wb), bits)
        x = U.to_dev_bf16(torch, xb)
        y = torch.full((M, N), float("nan"), device="cuda")
        ws = torch.empty(mxs.linear_decode_workspace_bytes(M, K, N, bits), dtype=torch.uint8, device="cuda")
        probs.append((x, bits, packed, N, y, ws))
        refs.append(oracle_full(xb, wb, bits))
    torch.cuda.synchronize()  # weights are static before the first decode call
    mxs.linear_decode_group(probs)
    torch.cuda.synchronize()
    for (x, bits, packed, N, y, ws), (ref, ab) in zip(probs, refs):
        got = y.cpu().numpy()
        U.check_gemm(got, ref, ab)
        single = mxs.linear_decode(x, bits, packed, N).cpu().numpy()
        U.check_gemm(got, single.astype(np.float64), ab)


@pytest.mark.parametrize("M,N,nb", [(16, 1000, 128), (3, 4096, 448), (1, 3000, 448), (1, 8192, 256)])
def test_linear_decode_workspace_garbage_reuse_and_graph_replay(torch, M, N, nb):
    """The fused layer needs nothing prepared in its workspace: a workspace
    full of garbage, the same workspace reused, and a CUDA graph replaying the
    same call all give the same y, bit for bit (M = 1: the arrival counts of
    the CTAs that share a row group are tagged per call)."""
    g = I.rng(70, M, N, nb)
    bits = I.width_map(nb, 0.8, 0.15, 0.05, g)
    xb, wb, codes, scales, packed = layer(torch, M, 32 * nb, N, bits, g)
    x = U.to_dev_bf16(torch, xb)
    ws = torch.randint(0, 256, (mxs.linear_decode_workspace_bytes(M, 32 * nb, N, bits),), dtype=torch.uint8,
                       device="cuda")
    ys = [mxs.linear_decode(x, bits, packed, N, workspace=ws).cpu().numpy() for _ in range(3)]
    ref, ab = oracle_full(xb, wb, bits)
    U.check_gemm(ys[0], ref, ab)
    assert all(np.array_equal(ys[0], y) for y in ys[1:])
    y = torch.empty((M, N), dtype=torch.float32, device="cuda")
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        mxs.linear_decode(x, bits, packed, N, y=y, workspace=ws, stream=s)
    s.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=s):
        mxs.linear_decode(x, bits, packed, N, y=y, workspace=ws, stream=s)
    for _ in range(3):
        y.fill_(float("nan"))
        graph.replay()
        torch.cuda.synchronize()
        assert np.array_equal(y.cpu().numpy(), ys[0])


def test_decode_bounded_wait_reports_timeout(torch):
    """A weight chunk that never arrives, in a launch the planner splits over a
    thread-block cluster (N = 1024: 8 row groups, K = 8192): every CTA's
    converters give up after the wait bound, the kernel records
    MXS_ERR_TIMEOUT, drains what it issued, frees its tensor memory and
    returns; the context stays usable and the next decode call is exact."""
    M, N, K = 16, 1024, 8192
    g = I.rng(43)
    bits = I.width_map(K // 32, 0.8, 0.15, 0.05, g)
    xb, wb, codes, scales, packed = layer(torch, M, K, N, bits, g)
    _, _, planes = mxs.quantize_act(U.to_dev_bf16(torch, xb), bits, want_codes=False, want_planes=True)
    assert mxs.device_status(reset=True) in (0, 7)
    mxs.test_decode_starve(planes, bits, packed, M, N, chunk=1)
    assert mxs.device_status(reset=True) == 7
    assert mxs.device_status() == 0
    y = mxs.gemm_decode(None, None, bits, packed, N, planes=planes, M=M).cpu().numpy()
    ref, ab = oracle_full(xb, wb, bits)
    U.check_gemm(y, ref, ab)
