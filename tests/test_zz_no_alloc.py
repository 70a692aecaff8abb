"""mxs_linear_decode_noalloc against mxs_linear_decode.

Some callers of the decode layer cannot allocate device memory -- an
allocator-free runtime that owns all device memory up front, a plug-in whose
host forbids allocations on its hot path, a real-time loop that must not block
in the allocator.  For them the library keeps the activations' MMA planes in a
fixed array of its own instead of a caller workspace.  These tests call that
entry point through the C ABI and compare it with the workspace path.

The file name makes pytest collect it last, so a run that stops at the first
failure has already run every other test when it gets here."""
import ctypes

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


def _layer(torch, M, K, N, p, seed, rounding=mxs.RNE):
    g = I.rng(70, seed)
    bits = I.width_map(K // 32, *p, g)
    xb = I.activations_bf16(M, bits, g, 0.01, outlier_scale=30.0)
    wb = I.normal_bf16((N, K), 0.02, g)
    packed = mxs.pack_weight(U.to_dev_bf16(torch, wb), bits, rounding=rounding)
    torch.cuda.synchronize()  # weights are static before the first decode call
    return bits, xb, wb, packed


def _noalloc(torch, x, bits, packed, N, rounding=mxs.RNE):
    """One call straight through the C ABI (no workspace argument exists)."""
    L = mxs.lib()
    M, K = x.shape
    y = torch.full((M, N), float("nan"), device="cuda")
    b = np.ascontiguousarray(bits, np.uint8)
    rc = L.mxs_linear_decode_noalloc(ctypes.c_void_p(x.data_ptr()), M, K, x.stride(0),
                                     b.ctypes.data_as(ctypes.c_void_p), rounding, ctypes.c_void_p(packed.data_ptr()),
                                     N, ctypes.c_void_p(y.data_ptr()), y.stride(0), None)
    assert rc == 0, mxs.last_error()
    return y


def test_noalloc_matches_workspace_path_on_two_calls_in_a_row(torch):
    """Two calls back to back on one stream share the library's array.  The
    second has fewer tokens and a longer K, so the array still holds the
    first call's planes in places the second does not write; both results
    must match the workspace path within the GEMM bar."""
    cases = [(16, 4096, 1000, (0.85, 0.10, 0.05), 1), (3, 14336, 512, (0.5, 0.3, 0.2), 2)]
    layers = [_layer(torch, M, K, N, p, seed) for M, K, N, p, seed in cases]
    xs = [U.to_dev_bf16(torch, xb) for _, xb, _, _ in layers]
    y_na = [_noalloc(torch, x, bits, packed, N)
            for x, (bits, _, _, packed), (_, _, N, _, _) in zip(xs, layers, cases)]
    torch.cuda.synchronize()
    for x, y, (bits, xb, wb, packed), (M, K, N, _, _) in zip(xs, y_na, layers, cases):
        y_ws = mxs.linear_decode(x, bits, packed, N).cpu().numpy()
        a_s, a_c = mxo.quantize_bf16(xb, bits)
        w_s, w_c = mxo.quantize_bf16(wb, bits)
        _, abssum = mxo.gemm(bits, a_c, a_s, w_c, w_s)
        U.check_gemm(y.cpu().numpy(), y_ws.astype(np.float64), abssum)


def test_noalloc_at_the_size_limit_under_both_roundings(torch):
    """The largest planes the array holds in practice: 16 tokens, K = 49152,
    every block 8-bit (1,966,080 of the 2 MiB), under ties-to-even and
    ties-away rounding, two calls in a row against the workspace path."""
    M, K, N = 16, 49152, 256
    bits_all8 = np.full(K // 32, 8, np.uint8)
    assert 1_900_000 < mxs.act_planes_bytes(M, K, bits_all8) <= 2 << 20
    for rounding in (mxs.RHAZ, mxs.RNE):
        bits, xb, wb, packed = _layer(torch, M, K, N, (0, 0, 1), 9, rounding)
        assert np.all(bits == 8)
        x = U.to_dev_bf16(torch, xb)
        y_na = _noalloc(torch, x, bits, packed, N, rounding)
        y_ws = mxs.linear_decode(x, bits, packed, N, rounding=rounding).cpu().numpy()
        a_s, a_c = mxo.quantize_bf16(xb, bits, rounding=rounding)
        w_s, w_c = mxo.quantize_bf16(wb, bits, rounding=rounding)
        ref, abssum = mxo.gemm(bits, a_c, a_s, w_c, w_s)
        U.check_gemm(y_na.cpu().numpy(), y_ws.astype(np.float64), abssum)
        U.check_gemm(y_na.cpu().numpy(), ref, abssum)
