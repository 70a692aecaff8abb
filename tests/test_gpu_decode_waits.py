"""Failure handling of the two kernels behind mxs_linear_decode: a weight
stage that never arrives (mxs_test_decode_arm_starve makes every CTA of the
next launch skip that copy).  The consumers' bounded wait for it runs out;
each starved CTA records MXS_ERR_TIMEOUT, stops its arithmetic, waits for the
copies it did issue, frees its tensor memory and returns.  The host reads the
status through mxs_device_status, the context stays usable, and the next
call on the same workspace (its arrival counters left mid-count by the
aborted launch) is exact against the oracle.  No device fault, trap or hang
is involved: the failure is a copy the producer does not issue."""
import pytest

from oracle import mxo
from paper_2607_17733_gb300 import inputs as I
from paper_2607_17733_gb300 import mxs
import gpu_util as U

pytestmark = pytest.mark.gpu

TIMEOUT = 7  # MXS_ERR_TIMEOUT


@pytest.fixture(scope="module")
def torch():
    return U.torch_or_skip()


def _ref(xb, wb, bits):
    a_s, a_c = mxo.quantize_bf16(xb, bits, mxo.RNE)
    w_s, w_c = mxo.quantize_bf16(wb, bits, mxo.RNE)
    return mxo.gemm(bits, a_c, a_s, w_c, w_s)


# a 70B o projection: 64 row groups over 152 CTAs, ~7 weight stages per CTA
# in either kernel, so stage 1 starves every CTA at its first copy and stage 4
# in mid-stream with copies in flight
@pytest.mark.parametrize("M,kernel", [(1, 1), (5, 2), (16, 2)])
@pytest.mark.parametrize("stage", [1, 4])
def test_decode_starved_stage_reports_timeout(torch, M, kernel, stage):
    K, N = 8192, 8192
    g = I.rng(44, M, stage)
    bits = I.width_map(K // 32, 0.8, 0.15, 0.05, g)
    xb = I.activations_bf16(M, bits, g, 0.01, outlier_scale=30.0)
    wb = I.normal_bf16((N, K), 0.02, g)
    x = U.to_dev_bf16(torch, xb)
    packed = mxs.pack_weight(U.to_dev_bf16(torch, wb), bits)
    ws = torch.empty(mxs.linear_decode_workspace_bytes(M, K, N, bits), dtype=torch.uint8, device="cuda")
    y = torch.zeros((M, N), dtype=torch.float32, device="cuda")
    torch.cuda.synchronize()
    assert mxs.device_status(reset=True) in (0, TIMEOUT)

    mxs.test_decode_arm_starve(kernel, stage)
    mxs.linear_decode(x, bits, packed, N, y=y, workspace=ws)
    torch.cuda.synchronize()
    assert mxs.device_status(reset=True) == TIMEOUT
    assert mxs.device_status() == 0

    # the arming was taken by that one launch: the next call, on the same
    # workspace, runs whole and exact
    y.fill_(float("nan"))
    mxs.linear_decode(x, bits, packed, N, y=y, workspace=ws)
    ref, ab = _ref(xb, wb, bits)
    U.check_gemm(y.cpu().numpy(), ref, ab)
    assert mxs.device_status() == 0


def test_decode_starve_in_a_group(torch):
    """A grouped launch (q/k/v shapes at M = 16) with one stage starved: the
    status is the timeout, and the same three problems then run exactly."""
    M = 16
    probs, refs = [], []
    for i, (K, N) in enumerate([(4096, 4096), (4096, 1024), (4096, 1024)]):
        g = I.rng(45, K, N, i)
        bits = I.width_map(K // 32, 0.85, 0.10, 0.05, g)
        xb = I.activations_bf16(M, bits, g, 0.01, outlier_scale=30.0)
        wb = I.normal_bf16((N, K), 0.02, g)
        packed = mxs.pack_weight(U.to_dev_bf16(torch, wb), bits)
        y = torch.zeros((M, N), dtype=torch.float32, device="cuda")
        ws = torch.empty(mxs.linear_decode_workspace_bytes(M, K, N, bits), dtype=torch.uint8, device="cuda")
        probs.append((U.to_dev_bf16(torch, xb), bits, packed, N, y, ws))
        refs.append(_ref(xb, wb, bits))
    torch.cuda.synchronize()
    assert mxs.device_status(reset=True) in (0, TIMEOUT)
    mxs.test_decode_arm_starve(2, 1)
    mxs.linear_decode_group(probs)
    torch.cuda.synchronize()
    assert mxs.device_status(reset=True) == TIMEOUT
    for p in probs:
        p[4].fill_(float("nan"))
    mxs.linear_decode_group(probs)
    for p, (ref, ab) in zip(probs, refs):
        U.check_gemm(p[4].cpu().numpy(), ref, ab)
    assert mxs.device_status() == 0
