"""The C ABI: exports, size queries and argument validation (no GPU needed).

Validation happens before any CUDA call, so every error path below runs the
same on a machine without a GPU."""
import ctypes
import os
import re

import numpy as np
import pytest

from oracle import mxo
from paper_2607_17733_gb300 import build as B
from paper_2607_17733_gb300 import mxs

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    B.build()
    return mxs.lib()


def header_functions():
    text = open(os.path.join(ROOT, "include", "mxs.h")).read()
    return sorted(set(re.findall(r"MXS_API\s+[\w\s\*]*?\b(mxs_\w+)\s*\(", text)))


def test_every_declared_function_is_exported(L):
    names = header_functions()
    assert len(names) >= 10
    for n in names:
        assert hasattr(L, n), n
    assert sorted(mxs.EXPORTS) == names
    assert L.mxs_version() == 3


def _bits(nb, seed=0, p=(0.7, 0.2, 0.1)):
    rs = np.random.default_rng(seed)
    return rs.choice(np.array([4, 6, 8], np.uint8), size=nb, p=p)


@pytest.mark.parametrize("K", [32, 96, 4096, 14336])
def test_sizes_match_the_storage_format(L, K):
    bits = _bits(K // 32, K)
    n4 = int(np.sum(bits == 4))
    assert mxs.act_row_bytes(K, bits) == 16 * n4 + 32 * (K // 32 - n4)
    assert mxs.act_codes_bytes(7, K, bits) == 7 * (16 * n4 + 32 * (K // 32 - n4))
    for N in (1, 16, 37, 1000):
        for layout in (0, 1):
            assert mxs.weight_bytes(N, K, bits, layout) == mxo.weight_bytes(N, K, bits, bool(layout))
    kp, nst = mxo.plane_shape(bits)
    M = 130
    sf_off = (M * kp + 255) // 256 * 256
    assert mxs.act_planes_bytes(M, K, bits) == (sf_off + 2 * nst * 512 + 255) // 256 * 256


def test_size_queries_reject_bad_arguments(L):
    bits = np.full(4, 4, np.uint8)
    assert L.mxs_act_row_bytes(100, bits.ctypes.data) == -2  # K not a multiple of 32
    assert L.mxs_act_row_bytes(0, bits.ctypes.data) == -2
    assert L.mxs_act_row_bytes(65536 + 32, bits.ctypes.data) == -2
    bad = np.array([4, 5, 6, 8], np.uint8)
    assert L.mxs_act_row_bytes(128, bad.ctypes.data) == -3
    assert "bits[1]=5" in mxs.last_error()
    assert L.mxs_act_row_bytes(128, None) == -1
    assert L.mxs_weight_bytes(16, 128, bits.ctypes.data, 7) == -1
    assert L.mxs_act_codes_bytes(-1, 128, bits.ctypes.data) == -2


FAKE = 1 << 20  # an aligned address that is never dereferenced: validation fails first


def test_quantize_validation(L):
    bits = np.full(4, 4, np.uint8)
    b = bits.ctypes.data
    q = L.mxs_quantize_act
    assert q(FAKE, 4, 100, 100, b, 0, FAKE, FAKE, None, None) == 2
    assert q(FAKE, 4, 128, 128, np.full(4, 7, np.uint8).ctypes.data, 0, FAKE, FAKE, None, None) == 3
    assert q(FAKE, 4, 128, 120, b, 0, FAKE, FAKE, None, None) == 1   # ld_x < K
    assert q(FAKE, 4, 128, 132, b, 0, FAKE, FAKE, None, None) == 1   # ld_x not a multiple of 8
    assert q(FAKE, 4, 128, 128, b, 2, FAKE, FAKE, None, None) == 1   # rounding
    assert q(FAKE, 4, 128, 128, b, 0, None, None, None, None) == 1   # no output
    assert q(FAKE, 4, 128, 128, b, 0, FAKE, None, None, None) == 1   # codes without scales
    assert q(FAKE + 8, 4, 128, 128, b, 0, FAKE, FAKE, None, None) == 4
    assert q(FAKE, 4, 128, 128, b, 0, FAKE, FAKE, FAKE + 4, None) == 4
    assert q(FAKE, 0, 128, 128, b, 0, FAKE, FAKE, None, None) == 0   # M = 0: nothing to do


def test_pack_and_gemm_validation(L):
    bits = np.full(4, 4, np.uint8)
    b = bits.ctypes.data
    assert L.mxs_pack_weight(FAKE, 16, 128, 128, b, 0, 3, FAKE, None) == 1
    assert L.mxs_pack_weight(FAKE, 16, 128, 128, b, 0, 0, None, None) == 1
    assert L.mxs_pack_weight(FAKE, 16, 128, 128, b, 0, 0, FAKE + 2, None) == 4
    other = np.array([4, 4, 8, 4], np.uint8)
    g = L.mxs_gemm
    assert g(FAKE, FAKE, None, b, FAKE, 0, other.ctypes.data, 4, 16, 128, FAKE, 16, None, 0, None) == 8
    d = L.mxs_gemm_decode
    assert d(FAKE, FAKE, None, b, FAKE, 17, 16, 128, FAKE, 16, None, 0, None) == 2   # M > 16
    assert d(FAKE, FAKE, None, b, FAKE, 4, 16, 128, FAKE, 8, None, 0, None) == 1     # ld_y < N
    assert d(FAKE, FAKE, None, b, None, 4, 16, 128, FAKE, 16, None, 0, None) == 1
    assert d(FAKE, FAKE, None, b, FAKE, 4, 16, 128, FAKE + 2, 16, None, 0, None) == 4
    assert d(FAKE, FAKE, FAKE, b, FAKE, 4, 16, 128, FAKE, 16, None, 0, None) == 1    # codes and planes
    assert d(None, None, None, b, FAKE, 4, 16, 128, FAKE, 16, None, 0, None) == 1    # neither
    assert d(None, None, FAKE + 8, b, FAKE, 4, 16, 128, FAKE, 16, None, 0, None) == 4
    ld = L.mxs_linear_decode
    need = L.mxs_act_planes_bytes(4, 128, b)
    assert need > 0
    assert ld(FAKE, 4, 128, 128, b, 0, FAKE, 16, FAKE, 16, FAKE, need - 1, None) == 5  # workspace too small
    assert ld(FAKE, 4, 128, 128, b, 0, FAKE, 16, FAKE, 16, None, need, None) == 5
    assert ld(FAKE, 4, 128, 128, b, 0, FAKE, 16, FAKE, 16, FAKE + 4, need, None) == 4
    assert ld(FAKE, 17, 128, 128, b, 0, FAKE, 16, FAKE, 16, FAKE, need, None) == 2


def test_valid_call_without_gpu_reports_cuda_error(L):
    torch = pytest.importorskip("torch")
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    bits = np.full(4, 4, np.uint8)
    rc = L.mxs_quantize_act(FAKE, 4, 128, 128, bits.ctypes.data, 0, FAKE, FAKE, None, None)
    assert rc == 6 and "cudaGetDevice" in mxs.last_error()


def test_noalloc_rejects_sizes_beyond_its_scratch(L):
    """mxs_linear_decode_noalloc keeps the planes in a fixed 2 MiB array: a
    16-token K=65536 all-8-bit layer needs more and is refused before any
    device call (so no GPU is needed here)."""
    bits = np.full(2048, 8, np.uint8)
    assert L.mxs_act_planes_bytes(16, 65536, bits.ctypes.data) > 2 << 20
    rc = L.mxs_linear_decode_noalloc(FAKE, 16, 65536, 65536, bits.ctypes.data, 0, FAKE, 16, FAKE, 16, None)
    assert rc == 5 and "built-in scratch" in mxs.last_error()
    small = np.full(4, 4, np.uint8)
    assert L.mxs_linear_decode_noalloc(FAKE, 17, 128, 128, small.ctypes.data, 0, FAKE, 16, FAKE, 16, None) == 2


def test_allocation_r_runs_on_the_host(L):
    """Theorem 1's R needs no device: the library against the oracle's closed form."""
    from oracle import alloc as A
    d = [4096, 4096, 14336, 1024, 28672]
    s = [1.0, 0.3, 0.7, 0.05, 0.5]
    for B in (4.1, 4.5, 5.75):
        assert abs(mxs.allocation_r(d, s, B) - A.allocation_r(d, s, B)) <= 1e-12 * max(1.0, A.allocation_r(d, s, B))


def test_allocation_validation(L):
    r = ctypes.c_double()
    d = np.array([4096, 100], np.int64)
    sl = np.array([0.5, 0.5])
    assert L.mxs_allocation_r(2, d.ctypes.data, sl.ctypes.data, 4.5, ctypes.byref(r)) == 2
    d = np.array([4096, 4096], np.int64)
    sl = np.array([0.5, 1.5])
    assert L.mxs_allocation_r(2, d.ctypes.data, sl.ctypes.data, 4.5, ctypes.byref(r)) == 1
    sl = np.array([0.0, 0.0])
    assert L.mxs_allocation_r(2, d.ctypes.data, sl.ctypes.data, 4.5, ctypes.byref(r)) == 1
    sl = np.array([0.5, 0.5])
    assert L.mxs_allocation_r(2, d.ctypes.data, sl.ctypes.data, 4.0, ctypes.byref(r)) == 1
    assert L.mxs_allocation_r(0, d.ctypes.data, sl.ctypes.data, 4.5, ctypes.byref(r)) == 2
    # device calls: rejected before any CUDA call
    fake = ctypes.c_void_p(1 << 20)
    bits = np.zeros(8, np.uint8)
    n6 = ctypes.c_int64()
    assert L.mxs_column_sensitivity(fake, 4, 100, 104, fake, 0, None) == 2
    assert L.mxs_column_sensitivity(fake, -1, 64, 64, fake, 0, None) == 2
    assert L.mxs_column_sensitivity(fake, 4, 64, 60, fake, 0, None) == 1
    assert L.mxs_column_sensitivity(ctypes.c_void_p((1 << 20) + 8), 4, 64, 64, fake, 0, None) == 4
    assert L.mxs_allocate_layer(fake, 100, 0.5, 0.5, fake, bits.ctypes.data, ctypes.byref(n6), None) == 2
    assert L.mxs_allocate_layer(fake, 256, -1.0, 0.5, fake, bits.ctypes.data, ctypes.byref(n6), None) == 1
    assert L.mxs_allocate_layer(fake, 1 << 20, 0.5, 0.5, fake, bits.ctypes.data, ctypes.byref(n6), None) == 2


def test_decode_group_validation(L):
    """mxs_linear_decode_group checks every problem before any device call."""
    bits = np.full(4, 4, np.uint8)
    b = bits.ctypes.data
    need = L.mxs_act_planes_bytes(4, 128, b)

    def prob(**kw):
        f = dict(x=FAKE, K=128, ld_x=128, bits=b, packed_w=FAKE, N=16, y=FAKE, ld_y=16, workspace=FAKE,
                 ws_bytes=need)
        f.update(kw)
        return mxs.DecodeProblem(**f)

    def call(probs, M=4, rounding=0, count=None):
        arr = (mxs.DecodeProblem * max(1, len(probs)))(*probs)
        return L.mxs_linear_decode_group(ctypes.addressof(arr), len(probs) if count is None else count, M,
                                         rounding, None)

    ws2 = FAKE + (1 << 16)
    bad = np.full(4, 5, np.uint8)
    assert call([prob()], count=0) == 1
    assert call([prob(), prob(workspace=ws2), prob(workspace=ws2 * 2)], count=4) == 1
    assert call([prob()], M=17) == 2
    assert call([prob()], M=-1) == 2
    assert call([prob()], rounding=3) == 1
    assert call([prob(), prob(K=100)]) == 2
    assert call([prob(), prob(workspace=ws2, bits=bad.ctypes.data)]) == 3
    assert call([prob(), prob(workspace=ws2, ld_y=8)]) == 1
    assert call([prob(), prob(workspace=ws2, ld_x=132)]) == 1
    assert call([prob(), prob(workspace=ws2, y=None)]) == 1
    assert call([prob(), prob(workspace=ws2, ws_bytes=need - 1)]) == 5
    assert call([prob(), prob(workspace=ws2 + 8)]) == 4
    assert call([prob(), prob(workspace=ws2, packed_w=FAKE + 4)]) == 4
    assert call([prob(), prob()]) == 1 and "share a workspace" in mxs.last_error()
    assert call([prob(N=-1)]) == 2


def test_prefill_rejects_decode_sized_m(L):
    """Planes of M <= 16 rows hold the decode form of 6/8-bit blocks, so the
    prefill GEMM refuses them before any device call; M = 0 is a no-op."""
    bits = np.full(4, 6, np.uint8)
    b = bits.ctypes.data
    for M in (1, 16):
        assert L.mxs_gemm_prefill(FAKE, b, FAKE, M, 16, 128, FAKE, 16, None) == 2
        assert "M > 16" in mxs.last_error()


def test_quantize_group_validation(L):
    """mxs_quantize_act_group checks every problem before any device call."""
    bits = np.full(4, 4, np.uint8)
    b = bits.ctypes.data

    def prob(**kw):
        f = dict(x=FAKE, K=128, ld_x=128, bits=b, planes=FAKE, planes_bytes=1 << 16)
        f.update(kw)
        return mxs.QuantProblem(**f)

    def call(probs, M=4, rounding=0, count=None):
        arr = (mxs.QuantProblem * max(1, len(probs)))(*probs)
        return L.mxs_quantize_act_group(ctypes.addressof(arr), len(probs) if count is None else count, M,
                                        rounding, None)

    p2 = FAKE + (1 << 16)
    bad = np.full(4, 5, np.uint8)
    assert call([prob()], count=0) == 1
    assert call([prob(), prob(planes=p2), prob(planes=2 * p2)], count=4) == 1
    assert call([prob()], M=-1) == 2
    assert call([prob()], rounding=2) == 1
    assert call([prob(), prob(planes=p2, K=100)]) == 2
    assert call([prob(), prob(planes=p2, bits=bad.ctypes.data)]) == 3
    assert call([prob(), prob(planes=p2, ld_x=132)]) == 1
    assert call([prob(), prob(planes=p2, x=None)]) == 1
    assert call([prob(), prob(planes=p2 + 8)]) == 4
    need = mxs.act_planes_bytes(4, 128, bits)
    assert call([prob(), prob(planes=p2, planes_bytes=need - 1)]) == 5 and "problem 1" in mxs.last_error()
    assert call([prob(), prob()]) == 1 and "share planes" in mxs.last_error()
    assert call([prob()], M=0) == 0


def test_probe_validation(L):
    """The rate probe checks its arguments before any device call."""
    f = ctypes.c_double()
    assert L.mxs_probe_mma(4, 16, 10, None, ctypes.byref(f), None) == 1
    assert L.mxs_probe_mma(0, 24, 10, None, ctypes.byref(f), None) == 1
    assert L.mxs_probe_mma(0, 272, 10, None, ctypes.byref(f), None) == 1
    assert L.mxs_probe_mma(1, 16, 0, None, ctypes.byref(f), None) == 1
    assert L.mxs_probe_mma(2, 16, 10, None, None, None) == 1
    assert L.mxs_probe_mma(0, 16, 10, FAKE + 4, ctypes.byref(f), None) == 4
    assert L.mxs_probe_status(None, 0) == 1


def test_decode_arm_starve_validation(L):
    """The decode kernels' starve hook takes kernel 1 or 2 and a stage >= 0
    (host only: arming touches no device; 0 disarms)."""
    assert L.mxs_test_decode_arm_starve(0, 1) == 1
    assert L.mxs_test_decode_arm_starve(3, 1) == 1
    assert L.mxs_test_decode_arm_starve(1, -1) == 1
    assert L.mxs_test_decode_arm_starve(1, 0) == 0
    assert L.mxs_test_decode_arm_starve(2, 0) == 0
