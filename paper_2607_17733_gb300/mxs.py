"""Thin ctypes binding of libmxs (include/mxs.h).

Argument marshalling only: every step of the quantize / pack / GEMM path runs
in the library's CUDA kernels.  torch supplies device memory and the current
stream.  There is no fallback: if libmxs.so is missing or the device is not
sm_103a, the calls raise.
"""
from __future__ import annotations

import ctypes
import os
import threading

import numpy as np

MXS_OK = 0
ERRORS = {1: "INVALID_ARG", 2: "SHAPE", 3: "BITS", 4: "ALIGN", 5: "BUFFER", 6: "CUDA",
          7: "TIMEOUT", 8: "UNSUPPORTED"}
RNE, RHAZ = 0, 1
W_COMPACT, W_COMPACT_AND_PLANES = 0, 1
MAX_K = 65536

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libmxs.so")
EXPORTS = ["mxs_last_error", "mxs_version", "mxs_act_row_bytes", "mxs_act_codes_bytes",
           "mxs_act_planes_bytes", "mxs_weight_bytes", "mxs_gemm_workspace_bytes",
           "mxs_quantize_act", "mxs_pack_weight", "mxs_gemm", "mxs_gemm_decode",
           "mxs_gemm_prefill", "mxs_device_status", "mxs_test_prefill_starve", "mxs_test_decode_starve",
           "mxs_linear_decode",
           "mxs_linear_decode_noalloc", "mxs_column_sensitivity", "mxs_allocation_r", "mxs_allocate_layer",
           "mxs_quantize_act_permuted", "mxs_pack_weight_permuted", "mxs_attention_decode_workspace_bytes",
           "mxs_attention_decode", "mxs_linear_decode_group", "mxs_quantize_act_group",
           "mxs_attention_decode_batch_workspace_bytes", "mxs_attention_decode_batch", "mxs_probe_mma",
           "mxs_probe_status", "mxs_linear_decode_workspace_bytes", "mxs_test_gemv_split",
           "mxs_test_gemv_ring", "mxs_probe_mma_issue",
           "mxs_test_decode_arm_starve", "mxs_test_dtc_split", "mxs_test_dtc_split_weight"]

_lock = threading.Lock()
_lib = None


class MxsError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"MXS_ERR_{ERRORS.get(code, code)}: {msg}")
        self.code = code


def lib() -> ctypes.CDLL:
    """Load libmxs.so (built by paper_2607_17733_gb300.build)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: run `python -c 'import __graft_entry__ as g; g.build()'`")
        L = ctypes.CDLL(LIB_PATH)
        P, I64, I, SZ = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_size_t
        L.mxs_last_error.restype = ctypes.c_char_p
        L.mxs_last_error.argtypes = []
        L.mxs_version.restype = I
        for name in ("mxs_act_row_bytes",):
            getattr(L, name).argtypes = [I64, P]
            getattr(L, name).restype = I64
        for name in ("mxs_act_codes_bytes", "mxs_act_planes_bytes"):
            getattr(L, name).argtypes = [I64, I64, P]
            getattr(L, name).restype = I64
        L.mxs_weight_bytes.argtypes = [I64, I64, P, I]
        L.mxs_weight_bytes.restype = I64
        L.mxs_gemm_workspace_bytes.argtypes = [I64, I64, I64, P]
        L.mxs_gemm_workspace_bytes.restype = I64
        L.mxs_quantize_act.argtypes = [P, I64, I64, I64, P, I, P, P, P, P]
        L.mxs_quantize_act.restype = I
        L.mxs_pack_weight.argtypes = [P, I64, I64, I64, P, I, I, P, P]
        L.mxs_pack_weight.restype = I
        L.mxs_quantize_act_permuted.argtypes = [P, I64, I64, I64, P, P, I, P, P, P, P]
        L.mxs_quantize_act_permuted.restype = I
        L.mxs_pack_weight_permuted.argtypes = [P, I64, I64, I64, P, P, I, I, P, P]
        L.mxs_pack_weight_permuted.restype = I
        L.mxs_gemm.argtypes = [P, P, P, P, P, I, P, I64, I64, I64, P, I64, P, SZ, P]
        L.mxs_gemm.restype = I
        L.mxs_gemm_decode.argtypes = [P, P, P, P, P, I64, I64, I64, P, I64, P, SZ, P]
        L.mxs_gemm_decode.restype = I
        L.mxs_linear_decode.argtypes = [P, I64, I64, I64, P, I, P, I64, P, I64, P, SZ, P]
        L.mxs_linear_decode.restype = I
        L.mxs_linear_decode_noalloc.argtypes = [P, I64, I64, I64, P, I, P, I64, P, I64, P]
        L.mxs_linear_decode_noalloc.restype = I
        L.mxs_gemm_prefill.argtypes = [P, P, P, I64, I64, I64, P, I64, P]
        L.mxs_gemm_prefill.restype = I
        L.mxs_test_prefill_starve.argtypes = [P, P, P, I64, I64, I64, P, I64, I, P]
        L.mxs_test_prefill_starve.restype = I
        L.mxs_test_decode_starve.argtypes = [P, P, P, I64, I64, I64, P, I64, I, P]
        L.mxs_test_decode_starve.restype = I
        L.mxs_device_status.argtypes = [ctypes.POINTER(ctypes.c_int), I, P]
        L.mxs_device_status.restype = I
        D = ctypes.c_double
        L.mxs_column_sensitivity.argtypes = [P, I64, I64, I64, P, I, P]
        L.mxs_column_sensitivity.restype = I
        L.mxs_allocation_r.argtypes = [I64, P, P, D, ctypes.POINTER(D)]
        L.mxs_allocation_r.restype = I
        L.mxs_allocate_layer.argtypes = [P, I64, D, D, P, P, ctypes.POINTER(I64), P]
        L.mxs_allocate_layer.restype = I
        L.mxs_linear_decode_group.argtypes = [P, I, I64, I, P]
        L.mxs_linear_decode_group.restype = I
        L.mxs_quantize_act_group.argtypes = [P, I, I64, I, P]
        L.mxs_quantize_act_group.restype = I
        L.mxs_attention_decode_workspace_bytes.argtypes = [I64, I64, I64]
        L.mxs_attention_decode_workspace_bytes.restype = I64
        L.mxs_attention_decode.argtypes = [P, I64, I64, I64, P, P, P, P, P, P, I64, ctypes.c_float, P, P, SZ, P]
        L.mxs_attention_decode.restype = I
        L.mxs_attention_decode_batch_workspace_bytes.argtypes = [I64, I64, I64, I64]
        L.mxs_attention_decode_batch_workspace_bytes.restype = I64
        L.mxs_attention_decode_batch.argtypes = [P, I64, I64, I64, I64, P, P, P, P, P, P, P, I64, ctypes.c_float, P, P,
                                                 SZ, P]
        L.mxs_attention_decode_batch.restype = I
        L.mxs_probe_mma.argtypes = [I, I, I64, P, ctypes.POINTER(ctypes.c_double), P]
        L.mxs_probe_mma.restype = I
        L.mxs_probe_status.argtypes = [ctypes.POINTER(ctypes.c_int), I]
        L.mxs_probe_status.restype = I
        L.mxs_linear_decode_workspace_bytes.argtypes = [I64, I64, I64, P]
        L.mxs_linear_decode_workspace_bytes.restype = I64
        L.mxs_test_gemv_split.argtypes = [P, P, P, I, I, P, P]
        L.mxs_test_gemv_split.restype = I
        L.mxs_test_dtc_split.argtypes = [P, P, P, I, I, P, P]
        L.mxs_test_dtc_split.restype = I
        L.mxs_test_dtc_split_weight.argtypes = [P]
        L.mxs_test_dtc_split_weight.restype = I
        L.mxs_test_gemv_ring.argtypes = [I]
        L.mxs_test_gemv_ring.restype = I
        L.mxs_test_decode_arm_starve.argtypes = [I, I]
        L.mxs_test_decode_arm_starve.restype = I
        L.mxs_probe_mma_issue.argtypes = [I, I, I64, P, P]
        L.mxs_probe_mma_issue.restype = I
        _lib = L
        return L


def last_error() -> str:
    return lib().mxs_last_error().decode()


def check(rc: int) -> None:
    if rc != MXS_OK:
        raise MxsError(rc, last_error())


def _size(v: int) -> int:
    if v < 0:
        raise MxsError(-v, last_error())
    return int(v)


class _Bits:
    """Host copy of a width map, kept alive for the duration of a call."""

    def __init__(self, bits):
        self.arr = np.ascontiguousarray(np.asarray(bits, dtype=np.uint8))
        self.ptr = self.arr.ctypes.data

    def __len__(self):
        return self.arr.size


def _ld(t) -> int:
    """Row stride in elements of a 2-D tensor; a single row has no meaningful
    stride (torch may report anything), so its row length is used."""
    return int(t.shape[1]) if t.shape[0] <= 1 else int(t.stride(0))


def _ptr(t) -> int | None:
    return None if t is None else t.data_ptr()


def _stream(stream) -> int | None:
    import torch
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


# ------------------------------------------------------------------ sizes
def act_row_bytes(K: int, bits) -> int:
    b = _Bits(bits)
    return _size(lib().mxs_act_row_bytes(K, b.ptr))


def act_codes_bytes(M: int, K: int, bits) -> int:
    b = _Bits(bits)
    return _size(lib().mxs_act_codes_bytes(M, K, b.ptr))


def act_planes_bytes(M: int, K: int, bits) -> int:
    b = _Bits(bits)
    return _size(lib().mxs_act_planes_bytes(M, K, b.ptr))


def linear_decode_workspace_bytes(M: int, K: int, N: int, bits) -> int:
    """Workspace bytes of linear_decode / each problem of linear_decode_group
    (mxs_linear_decode_workspace_bytes)."""
    b = _Bits(bits)
    return _size(lib().mxs_linear_decode_workspace_bytes(M, K, N, b.ptr))


def weight_bytes(N: int, K: int, bits, layout: int = W_COMPACT) -> int:
    b = _Bits(bits)
    return _size(lib().mxs_weight_bytes(N, K, b.ptr, layout))


def gemm_workspace_bytes(M: int, N: int, K: int, bits) -> int:
    b = _Bits(bits)
    return _size(lib().mxs_gemm_workspace_bytes(M, N, K, b.ptr))


# ------------------------------------------------------------------ calls
def quantize_act(x, bits, rounding: int = RNE, codes=None, scales=None, planes=None,
                 want_codes: bool = True, want_planes: bool = False, stream=None, perm=None):
    """x: bf16 [M, K] CUDA tensor (row stride may exceed K).  Returns
    (codes uint8 [M, row_bytes] | None, scales uint8 [M, K/32] | None, planes uint8 | None).
    perm (int32 [K] CUDA tensor): quantize x[:, perm] (mxs_quantize_act_permuted)."""
    import torch
    M, K = x.shape
    b = _Bits(bits)
    if want_codes and codes is None:
        codes = torch.empty((M, act_row_bytes(K, b.arr)), dtype=torch.uint8, device=x.device)
        scales = torch.empty((M, K // 32), dtype=torch.uint8, device=x.device)
    if want_planes and planes is None:
        planes = torch.empty(act_planes_bytes(M, K, b.arr), dtype=torch.uint8, device=x.device)
    if perm is not None:
        check(lib().mxs_quantize_act_permuted(_ptr(x), M, K, _ld(x), _ptr(perm), b.ptr, rounding, _ptr(codes),
                                              _ptr(scales), _ptr(planes), _stream(stream)))
    else:
        check(lib().mxs_quantize_act(_ptr(x), M, K, _ld(x), b.ptr, rounding, _ptr(codes), _ptr(scales),
                                     _ptr(planes), _stream(stream)))
    return codes, scales, planes


def pack_weight(w, bits, layout: int = W_COMPACT, rounding: int = RNE, out=None, stream=None, perm=None):
    """w: bf16 [N, K] CUDA tensor -> packed uint8 buffer (of w[:, perm] when perm is given)."""
    import torch
    N, K = w.shape
    b = _Bits(bits)
    if out is None:
        out = torch.empty(weight_bytes(N, K, b.arr, layout), dtype=torch.uint8, device=w.device)
    if perm is not None:
        check(lib().mxs_pack_weight_permuted(_ptr(w), N, K, _ld(w), _ptr(perm), b.ptr, rounding, layout,
                                             _ptr(out), _stream(stream)))
    else:
        check(lib().mxs_pack_weight(_ptr(w), N, K, _ld(w), b.ptr, rounding, layout, _ptr(out),
                                    _stream(stream)))
    return out


def gemm(codes, scales, planes, bits, packed_w, N: int, w_layout: int = W_COMPACT, y=None,
         workspace=None, M: int | None = None, K: int | None = None, stream=None):
    """y [M, N] fp32 = x W^T on quantized operands (decode kernel for M <= 16)."""
    import torch
    b = _Bits(bits)
    K = 32 * len(b) if K is None else K
    if M is None:
        if codes is None:
            raise ValueError("gemm over activation planes needs M= (a planes buffer is flat)")
        M = codes.shape[0]
    dev = packed_w.device
    if y is None:
        y = torch.empty((M, N), dtype=torch.float32, device=dev)
    ws_need = gemm_workspace_bytes(M, N, K, b.arr)
    if workspace is None and ws_need > 0:
        workspace = torch.empty(ws_need, dtype=torch.uint8, device=dev)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    check(lib().mxs_gemm(_ptr(codes), _ptr(scales), _ptr(planes), b.ptr, _ptr(packed_w), w_layout, b.ptr,
                         M, N, K, _ptr(y), _ld(y), _ptr(workspace), ws_bytes, _stream(stream)))
    return y


def gemm_decode(codes, scales, bits, packed_w, N: int, y=None, workspace=None, stream=None, planes=None,
                M: int | None = None):
    """Decode kernel (M <= 16) over packed codes + scales, or over the MMA
    planes of quantize_act (pass planes=..., M=... and codes = scales = None)."""
    import torch
    b = _Bits(bits)
    if M is None:
        M = codes.shape[0]
    K = 32 * len(b)
    if y is None:
        y = torch.empty((M, N), dtype=torch.float32, device=packed_w.device)
    ws_need = gemm_workspace_bytes(M, N, K, b.arr)
    if workspace is None and ws_need > 0:
        workspace = torch.empty(ws_need, dtype=torch.uint8, device=packed_w.device)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    check(lib().mxs_gemm_decode(_ptr(codes), _ptr(scales), _ptr(planes), b.ptr, _ptr(packed_w), M, N, K, _ptr(y),
                                _ld(y), _ptr(workspace), ws_bytes, _stream(stream)))
    return y


def linear_decode(x, bits, packed_w, N: int, rounding: int = RNE, y=None, workspace=None, stream=None):
    """Activation quantization + decode GEMM (M <= 16) in one call: y [M, N]
    fp32.  workspace: uint8 of at least linear_decode_workspace_bytes(M, K, N,
    bits) bytes (allocated when None)."""
    import torch
    b = _Bits(bits)
    M, K = x.shape
    if y is None:
        y = torch.empty((M, N), dtype=torch.float32, device=packed_w.device)
    if workspace is None:
        workspace = torch.empty(max(linear_decode_workspace_bytes(M, K, N, b.arr), 16), dtype=torch.uint8,
                                device=packed_w.device)
    ws_bytes = workspace.numel() * workspace.element_size()
    check(lib().mxs_linear_decode(_ptr(x), M, K, _ld(x), b.ptr, rounding, _ptr(packed_w), N, _ptr(y),
                                  _ld(y), _ptr(workspace), ws_bytes, _stream(stream)))
    return y


class DecodeProblem(ctypes.Structure):
    """ctypes mirror of mxs_decode_problem (include/mxs.h)."""
    _fields_ = [("x", ctypes.c_void_p), ("K", ctypes.c_int64), ("ld_x", ctypes.c_int64), ("bits", ctypes.c_void_p),
                ("packed_w", ctypes.c_void_p), ("N", ctypes.c_int64), ("y", ctypes.c_void_p), ("ld_y", ctypes.c_int64),
                ("workspace", ctypes.c_void_p), ("ws_bytes", ctypes.c_size_t)]


def linear_decode_group(problems, rounding: int = RNE, stream=None):
    """Up to three decode layers in one grouped launch (mxs_linear_decode_group).
    problems: sequence of (x [M, K] bf16, bits, packed_w, N, y [M, N] fp32, workspace uint8)."""
    arr = (DecodeProblem * len(problems))()
    keep = []
    M = problems[0][0].shape[0]
    for i, (x, bits, packed_w, N, y, ws) in enumerate(problems):
        b = _Bits(bits)
        keep.append(b)
        if x.shape[0] != M:
            raise ValueError("every problem of a group has the same M")
        arr[i] = DecodeProblem(_ptr(x), x.shape[1], _ld(x), b.ptr, _ptr(packed_w), N, _ptr(y), _ld(y), _ptr(ws),
                               ws.numel() * ws.element_size())
    check(lib().mxs_linear_decode_group(ctypes.addressof(arr), len(problems), M, rounding, _stream(stream)))


class QuantProblem(ctypes.Structure):
    """ctypes mirror of mxs_quant_problem (include/mxs.h)."""
    _fields_ = [("x", ctypes.c_void_p), ("K", ctypes.c_int64), ("ld_x", ctypes.c_int64), ("bits", ctypes.c_void_p),
                ("planes", ctypes.c_void_p), ("planes_bytes", ctypes.c_size_t)]


def quantize_act_group(problems, rounding: int = RNE, stream=None):
    """MMA planes of up to three activations in one launch (mxs_quantize_act_group).
    problems: sequence of (x [M, K] bf16, bits, planes uint8 of act_planes_bytes(M, K, bits)).
    Returns the planes tensors."""
    arr = (QuantProblem * len(problems))()
    keep = []
    M = problems[0][0].shape[0]
    for i, (x, bits, planes) in enumerate(problems):
        b = _Bits(bits)
        keep.append(b)
        if x.shape[0] != M:
            raise ValueError("every problem of a group has the same M")
        arr[i] = QuantProblem(_ptr(x), x.shape[1], _ld(x), b.ptr, _ptr(planes), planes.numel() * planes.element_size())
    check(lib().mxs_quantize_act_group(ctypes.addressof(arr), len(problems), M, rounding, _stream(stream)))
    return [p[2] for p in problems]


def linear_decode_noalloc(x, bits, packed_w, N: int, rounding: int = RNE, y=None, stream=None):
    """linear_decode without a workspace: the planes go to the library's own
    2 MiB device array (for callers that cannot allocate; see the header)."""
    import torch
    b = _Bits(bits)
    M, K = x.shape
    if y is None:
        y = torch.empty((M, N), dtype=torch.float32, device=packed_w.device)
    check(lib().mxs_linear_decode_noalloc(_ptr(x), M, K, _ld(x), b.ptr, rounding, _ptr(packed_w), N, _ptr(y),
                                          _ld(y), _stream(stream)))
    return y


def gemm_prefill(planes, bits, packed_w, M: int, N: int, y=None, stream=None):
    """Tensor-core path: planes from quantize_act(want_planes=True), weights
    packed with W_COMPACT_AND_PLANES."""
    import torch
    b = _Bits(bits)
    K = 32 * len(b)
    if y is None:
        y = torch.empty((M, N), dtype=torch.float32, device=packed_w.device)
    check(lib().mxs_gemm_prefill(_ptr(planes), b.ptr, _ptr(packed_w), M, N, K, _ptr(y), _ld(y),
                                 _stream(stream)))
    return y


def test_prefill_starve(planes, bits, packed_w, M: int, N: int, stage: int, y=None, stream=None):
    """Test hook: the prefill kernel with K' stage `stage` never loaded."""
    import torch
    b = _Bits(bits)
    K = 32 * len(b)
    if y is None:
        y = torch.zeros((M, N), dtype=torch.float32, device=packed_w.device)
    check(lib().mxs_test_prefill_starve(_ptr(planes), b.ptr, _ptr(packed_w), M, N, K, _ptr(y), _ld(y),
                                        int(stage), _stream(stream)))
    return y


def test_decode_starve(planes, bits, packed_w, M: int, N: int, chunk: int, y=None, stream=None):
    """Test hook: the decode kernel over activation planes with every CTA's
    copy chunk `chunk` (1-based) never loaded."""
    import torch
    b = _Bits(bits)
    K = 32 * len(b)
    if y is None:
        y = torch.zeros((M, N), dtype=torch.float32, device=packed_w.device)
    check(lib().mxs_test_decode_starve(_ptr(planes), b.ptr, _ptr(packed_w), M, N, K, _ptr(y), _ld(y),
                                       int(chunk), _stream(stream)))
    return y


def test_decode_arm_starve(kernel: int, stage: int):
    """Test hook: the next launch of decode kernel `kernel` (1: one token,
    2: tensor-core, 2..16 tokens) skips every CTA's weight stage `stage`."""
    check(lib().mxs_test_decode_arm_starve(int(kernel), int(stage)))


def device_status(reset: bool = False, stream=None) -> int:
    st = ctypes.c_int(0)
    check(lib().mxs_device_status(ctypes.byref(st), int(reset), _stream(stream)))
    return st.value


# ---------------------------------------------------------------- offline allocation
def column_sensitivity(x, s=None, accumulate: bool = False, stream=None):
    """Alg. 1: s[j] (fp64, device) = (accumulate ? s[j] : 0) + sum over the rows of x[:, j]^2
    for a bf16 x [T, K] on the GPU (mxs_column_sensitivity)."""
    import torch
    T, K = x.shape
    if s is None:
        s = torch.zeros(K, dtype=torch.float64, device=x.device)
    check(lib().mxs_column_sensitivity(_ptr(x), T, K, _ld(x), _ptr(s), int(bool(accumulate)), _stream(stream)))
    return s


def allocation_r(d_in, s_layer, B: float) -> float:
    """Theorem 1: the control parameter R for an average of B bits (host only)."""
    d = np.ascontiguousarray(np.asarray(d_in, dtype=np.int64))
    sl = np.ascontiguousarray(np.asarray(s_layer, dtype=np.float64))
    if d.size != sl.size:
        raise ValueError("d_in and s_layer differ in length")
    r = ctypes.c_double()
    check(lib().mxs_allocation_r(d.size, d.ctypes.data, sl.ctypes.data, float(B), ctypes.byref(r)))
    return r.value


def allocate_layer(s, R: float, s_layer: float, perm=None, stream=None):
    """Alg. 3 for one layer: (perm [K] int32 on the device, bits [K/32] uint8 on the host, N6)."""
    import torch
    K = s.numel()
    if perm is None:
        perm = torch.empty(K, dtype=torch.int32, device=s.device)
    bits = np.zeros(max(K // 32, 1), dtype=np.uint8)
    n6 = ctypes.c_int64()
    check(lib().mxs_allocate_layer(_ptr(s), K, float(R), float(s_layer), _ptr(perm), bits.ctypes.data,
                                   ctypes.byref(n6), _stream(stream)))
    return perm, bits, n6.value


# ---------------------------------------------------------------- KV cache
def attention_decode(q, H_kv: int, k_codes, k_scales, k_bits, v_codes, v_scales, v_bits, T: int, scale: float,
                     out=None, workspace=None, stream=None):
    """One decode step over an MXINT KV cache (mxs_attention_decode).  q: bf16 [H, D];
    the caches as written by quantize_act (codes [T_max, row bytes], scales [T_max, nb])."""
    import torch
    H, D = q.shape
    kb, vb = _Bits(k_bits), _Bits(v_bits)
    if out is None:
        out = torch.empty((H, D), dtype=torch.float32, device=q.device)
    need = _size(lib().mxs_attention_decode_workspace_bytes(T, H, D))
    if workspace is None:  # its counters must start at zero; the call leaves them zero
        workspace = torch.zeros(need, dtype=torch.uint8, device=q.device)
    check(lib().mxs_attention_decode(_ptr(q), H, H_kv, D, _ptr(k_codes), _ptr(k_scales), kb.ptr, _ptr(v_codes),
                                     _ptr(v_scales), vb.ptr, T, float(scale), _ptr(out), _ptr(workspace),
                                     workspace.numel() * workspace.element_size(), _stream(stream)))
    return out


def attention_decode_batch(q, H_kv: int, k_codes, k_scales, k_bits, v_codes, v_scales, v_bits, T_cap: int,
                           scale: float, lengths=None, out=None, workspace=None, stream=None):
    """One decode step of B sequences over an MXINT KV cache
    (mxs_attention_decode_batch).  q: bf16 [B, H, D]; sequence b owns cache rows
    [b * T_cap, b * T_cap + lengths[b]); lengths: device int32 [B] or None
    (every sequence T_cap tokens).  workspace: zero-initialised uint8 of
    attention_batch_workspace_bytes(...) bytes (allocated zeroed when None)."""
    import torch
    B, H, D = q.shape
    kb, vb = _Bits(k_bits), _Bits(v_bits)
    if out is None:
        out = torch.empty((B, H, D), dtype=torch.float32, device=q.device)
    if workspace is None:
        workspace = torch.zeros(attention_batch_workspace_bytes(B, T_cap, H, D), dtype=torch.uint8, device=q.device)
    check(lib().mxs_attention_decode_batch(_ptr(q), B, H, H_kv, D, _ptr(k_codes), _ptr(k_scales), kb.ptr,
                                           _ptr(v_codes), _ptr(v_scales), vb.ptr,
                                           None if lengths is None else _ptr(lengths), T_cap, float(scale),
                                           _ptr(out), _ptr(workspace), workspace.numel() * workspace.element_size(),
                                           _stream(stream)))
    return out


def attention_batch_workspace_bytes(B: int, T_cap: int, H: int, D: int) -> int:
    return _size(lib().mxs_attention_decode_batch_workspace_bytes(B, T_cap, H, D))


# ---------------------------------------------------------------- tensor-core rate probes
PROBE_FP8, PROBE_FP8_TMEM_A, PROBE_BF16, PROBE_S8_MMA_SYNC = 0, 1, 2, 3


def probe_mma(kind: int, n: int, iters: int, cycles=None, stream=None) -> float:
    """Launch the rate probe (mxs_probe_mma); returns the launch's FLOPs."""
    flop = ctypes.c_double()
    check(lib().mxs_probe_mma(int(kind), int(n), int(iters), _ptr(cycles), ctypes.byref(flop), _stream(stream)))
    return flop.value


def probe_status(reset: bool = False) -> int:
    st = ctypes.c_int(0)
    check(lib().mxs_probe_status(ctypes.byref(st), int(reset)))
    return st.value
