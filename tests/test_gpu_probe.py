"""The MMA issue-rate probe behind the decode kernels' design: an N = 16
tcgen05 MMA costs its issuing thread a few tens of cycles, and several
issuing warps on one SM each keep that rate (the tensor pipe is far from
busy), which is why decode_tc.cu spreads its MMAs over four issuers."""
import ctypes

import numpy as np
import pytest

from paper_2607_17733_gb300 import mxs
import gpu_util as U

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch():
    return U.torch_or_skip()


def _cycles_per_mma(torch, kind, issuers, iters=4096):
    L = mxs.lib()
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    cyc = torch.zeros(sms, dtype=torch.int64, device="cuda")
    assert L.mxs_probe_mma_issue(kind, issuers, iters, ctypes.c_void_p(cyc.data_ptr()), None) == 0, mxs.last_error()
    torch.cuda.synchronize()
    st = ctypes.c_int(0)
    assert L.mxs_probe_status(ctypes.byref(st), 1) == 0 and st.value == 0
    return float(cyc.double().mean().item()) / iters


@pytest.mark.parametrize("kind", [0, 1, 2])
def test_issuers_keep_their_rate(torch, kind):
    one = _cycles_per_mma(torch, kind, 1)
    four = _cycles_per_mma(torch, kind, 4)
    print(f"kind {kind}: {one:.1f} cycles per MMA with one issuer, {four:.1f} per issuer with four")
    assert 5 < one < 1000
    assert four < 1.5 * one  # four issuers: about four times the MMAs per SM


def test_probe_rejects_bad_arguments(torch):
    L = mxs.lib()
    assert L.mxs_probe_mma_issue(3, 1, 4096, None, None) == 1
    assert L.mxs_probe_mma_issue(0, 3, 4096, None, None) == 1
    assert L.mxs_probe_mma_issue(0, 1, 4097, None, None) == 1
