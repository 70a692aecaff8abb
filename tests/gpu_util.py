"""Helpers shared by the GPU parity tests (host side only)."""
import numpy as np
import pytest

# The MXINT GEMM result y[m,n] = sum_kb t_kb (each t_kb exact in fp32 on both
# sides) is accumulated in fp32 by the kernels and summed exactly by the
# oracle.  A recursive fp32 sum of n terms errs by at most (n-1) * 2^-24 *
# sum|t_kb|, and by ~sqrt(n) * 2^-24 * sum|t_kb| in practice; 1e-5 of
# sum|t_kb| (Higham's componentwise measure for dot products) is the stated
# bar, checked alongside the normwise max|y - r| / max|r| <= 1e-5.
GEMM_RTOL = 1e-5


def torch_or_skip():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    return torch


def to_dev_bf16(torch, bits16):
    return torch.from_numpy(np.ascontiguousarray(bits16).view(np.int16)).view(torch.bfloat16).cuda()


def check_gemm(y, ref, abssum, rtol=GEMM_RTOL):
    y = np.asarray(y, np.float64)
    ref = np.asarray(ref, np.float64)
    assert y.shape == ref.shape
    nan_ref = np.isnan(ref)
    assert np.array_equal(np.isnan(y), nan_ref), "NaN pattern differs"
    ok = ~nan_ref
    err = np.abs(y[ok] - ref[ok])
    comp = err / np.maximum(abssum[ok], 1e-300)
    assert np.all(err <= rtol * abssum[ok] + 1e-38), f"componentwise error {comp.max():.3e}"
    if ok.any() and np.max(np.abs(ref[ok])) > 0:
        norm = err.max() / np.max(np.abs(ref[ok]))
        assert norm <= rtol, f"normwise error {norm:.3e}"
    return float(comp.max()) if comp.size else 0.0
