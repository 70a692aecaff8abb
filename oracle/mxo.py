"""ctypes front end of the CPU oracle (oracle/mxo.c).

TEST INFRASTRUCTURE ONLY: imported by tests/, __graft_entry__.smoke() and the
cpu_baseline / reference legs of bench.py.  The CUDA library never imports it
and it never imports the CUDA library.

Every function takes and returns numpy arrays in the oracle's natural layouts:
  codes  int8  [R, K]    one element per byte, natural K order
  scales uint8 [R, K/32] E8M0 byte of each block, natural block order
plus the packed library layouts (pack_act / pack_weight / planes) written from
the storage-format description.  See mxo.c for the rules (R1-R5) and their
source in the paper.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

RNE = 0
RHAZ = 1

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "mxo.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "libmxo.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile mxo.c with gcc (plain -O2, IEEE semantics, OpenMP over rows).
    MXO_LIB names an already built copy instead (the planted-mistake tests
    load altered copies of mxo.c this way)."""
    if os.environ.get("MXO_LIB"):
        return os.environ["MXO_LIB"]
    os.makedirs(_BUILD, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-fno-fast-math",
           "-ffp-contract=off", _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = ctypes.CDLL(build())
        P = ctypes.c_void_p
        I64 = ctypes.c_int64
        I = ctypes.c_int
        lib.mxo_quantize_block.argtypes = [P, I, I, P, P]
        lib.mxo_quantize_block.restype = I
        lib.mxo_element_value.argtypes = [ctypes.c_int8, ctypes.c_uint8, I]
        lib.mxo_element_value.restype = ctypes.c_double
        lib.mxo_quantize_bf16.argtypes = [P, I64, I64, I64, P, I, P, P]
        lib.mxo_quantize_bf16.restype = I
        lib.mxo_fsum.argtypes = [P, I64]
        lib.mxo_fsum.restype = ctypes.c_double
        lib.mxo_gemm.argtypes = [I64, I64, I64, P, P, P, P, P, P, P]
        lib.mxo_gemm.restype = I
        lib.mxo_gemm_entries.argtypes = [I64, P, P, P, P, P, I64, P, P, P, P]
        lib.mxo_gemm_entries.restype = I
        lib.mxo_slots.argtypes = [P, I64, P, P]
        lib.mxo_slots.restype = I
        lib.mxo_pack_act.argtypes = [I64, I64, P, P, P, P, P]
        lib.mxo_pack_act.restype = I
        lib.mxo_weight_bytes.argtypes = [I64, I64, P, I]
        lib.mxo_weight_bytes.restype = I64
        lib.mxo_e4m3_encode.argtypes = [ctypes.c_double]
        lib.mxo_e4m3_encode.restype = I
        lib.mxo_planes.argtypes = [I64, I64, P, P, P, P, P, I]
        lib.mxo_planes.restype = I
        lib.mxo_pack_weight.argtypes = [I64, I64, P, P, P, I, P]
        lib.mxo_pack_weight.restype = I
        _lib = lib
        return lib


def _p(a: np.ndarray) -> int:
    return a.ctypes.data


def _c(a, dtype) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=dtype))


# ---------------------------------------------------------------- quantize
def quantize_block(x, b: int, rounding: int = RNE):
    """One block of 32 real values -> (scale byte, int8 codes[32])."""
    x = _c(x, np.float64)
    assert x.shape == (32,)
    codes = np.zeros(32, np.int8)
    s = np.zeros(1, np.uint8)
    rc = _load().mxo_quantize_block(_p(x), int(b), int(rounding), _p(s), _p(codes))
    if rc != 0:
        raise ValueError(f"mxo_quantize_block rc={rc}")
    return int(s[0]), codes


def element_value(m: int, scale: int, b: int) -> float:
    return _load().mxo_element_value(int(m), int(scale), int(b))


def dequantize(codes: np.ndarray, scales: np.ndarray, bits: np.ndarray) -> np.ndarray:
    """codes [R,K], scales [R,nb] natural order -> fp64 values (NaN for S=255)."""
    codes = np.asarray(codes)
    R, K = codes.shape
    nb = K // 32
    widths = np.repeat(np.asarray(bits, np.int64), 32)[None, :]
    s = np.repeat(np.asarray(scales, np.int64).reshape(R, nb), 32, axis=1)
    out = np.ldexp(codes.astype(np.float64), (s - 127 - (widths - 2)).astype(np.int32))
    out[s == 255] = np.nan
    return out


def quantize_bf16(x_bits: np.ndarray, bits, rounding: int = RNE):
    """x_bits: uint16 [R, K] bf16 bit patterns -> (scales [R,nb], codes [R,K])."""
    x_bits = _c(x_bits, np.uint16)
    R, K = x_bits.shape
    bits = _c(bits, np.uint8)
    assert K % 32 == 0 and bits.shape == (K // 32,)
    scales = np.zeros((R, K // 32), np.uint8)
    codes = np.zeros((R, K), np.int8)
    rc = _load().mxo_quantize_bf16(_p(x_bits), R, K, K, _p(bits), int(rounding), _p(scales), _p(codes))
    if rc != 0:
        raise ValueError("mxo_quantize_bf16 failed")
    return scales, codes


# ---------------------------------------------------------------- sums / GEMM
def fsum(v) -> float:
    v = _c(v, np.float64).ravel()
    return _load().mxo_fsum(_p(v), v.size)


def gemm(bits, a_codes, a_scales, w_codes, w_scales):
    """Exact MXINT GEMM: returns (y [M,N] fp64 correctly rounded, abssum [M,N])."""
    bits = _c(bits, np.uint8)
    a_codes = _c(a_codes, np.int8)
    w_codes = _c(w_codes, np.int8)
    a_scales = _c(a_scales, np.uint8)
    w_scales = _c(w_scales, np.uint8)
    M, K = a_codes.shape
    N = w_codes.shape[0]
    y = np.zeros((M, N), np.float64)
    ab = np.zeros((M, N), np.float64)
    rc = _load().mxo_gemm(M, N, K, _p(bits), _p(a_codes), _p(a_scales), _p(w_codes),
                          _p(w_scales), _p(y), _p(ab))
    if rc != 0:
        raise ValueError("mxo_gemm failed")
    return y, ab


def gemm_entries(bits, a_codes, a_scales, w_codes, w_scales, rows, cols):
    """y and abssum for the listed (rows[i], cols[i]) entries only."""
    bits = _c(bits, np.uint8)
    a_codes = _c(a_codes, np.int8)
    w_codes = _c(w_codes, np.int8)
    a_scales = _c(a_scales, np.uint8)
    w_scales = _c(w_scales, np.uint8)
    rows = _c(rows, np.int64)
    cols = _c(cols, np.int64)
    K = a_codes.shape[1]
    y = np.zeros(rows.size, np.float64)
    ab = np.zeros(rows.size, np.float64)
    rc = _load().mxo_gemm_entries(K, _p(bits), _p(a_codes), _p(a_scales), _p(w_codes),
                                  _p(w_scales), rows.size, _p(rows), _p(cols), _p(y), _p(ab))
    if rc != 0:
        raise ValueError("mxo_gemm_entries failed")
    return y, ab


# ---------------------------------------------------------------- storage format
def slots(bits):
    bits = _c(bits, np.uint8)
    sb = np.zeros(bits.size, np.int32)
    cnt = np.zeros(3, np.int64)
    if _load().mxo_slots(_p(bits), bits.size, _p(sb), _p(cnt)) != 0:
        raise ValueError("width outside {4,6,8}")
    return sb, tuple(int(c) for c in cnt)


def pack_act(bits, scales, codes):
    bits = _c(bits, np.uint8)
    scales = _c(scales, np.uint8)
    codes = _c(codes, np.int8)
    R, K = codes.shape
    _, (n4, n6, n8) = slots(bits)
    pc = np.zeros((R, 16 * n4 + 32 * (n6 + n8)), np.uint8)
    ps = np.zeros((R, K // 32), np.uint8)
    if _load().mxo_pack_act(R, K, _p(bits), _p(scales), _p(codes), _p(pc), _p(ps)) != 0:
        raise ValueError("mxo_pack_act failed")
    return pc, ps


def weight_bytes(N: int, K: int, bits, with_planes: bool) -> int:
    bits = _c(bits, np.uint8)
    return int(_load().mxo_weight_bytes(N, K, _p(bits), int(bool(with_planes))))


def pack_weight(bits, scales, codes, with_planes: bool = False) -> np.ndarray:
    bits = _c(bits, np.uint8)
    scales = _c(scales, np.uint8)
    codes = _c(codes, np.int8)
    N, K = codes.shape
    out = np.zeros(weight_bytes(N, K, bits, with_planes), np.uint8)
    if _load().mxo_pack_weight(N, K, _p(bits), _p(scales), _p(codes), int(bool(with_planes)),
                               _p(out)) != 0:
        raise ValueError("mxo_pack_weight failed")
    return out


def e4m3_encode(v: float) -> int:
    return int(_load().mxo_e4m3_encode(float(v)))


def plane_shape(bits):
    _, (n4, n6, n8) = slots(bits)
    n68 = n6 + n8
    st4 = (n4 + 3) // 4
    nst = st4 + (n68 + 1) // 2
    return 128 * nst, nst


def planes(bits, scales, codes, bf16_68: bool = False):
    """(planes uint8 [R, Kp], scale tiles uint8 [ceil(R/128), nst, 512]).
    6/8-bit blocks as high/low e4m3 digits, or (bf16_68) as bf16 values
    m * 2^(S-127-(b-2)); see mxo.c."""
    bits = _c(bits, np.uint8)
    scales = _c(scales, np.uint8)
    codes = _c(codes, np.int8)
    R, K = codes.shape
    kp, nst = plane_shape(bits)
    pl = np.zeros((R, kp), np.uint8)
    sf = np.zeros(((R + 127) // 128, nst, 512), np.uint8)
    if _load().mxo_planes(R, K, _p(bits), _p(scales), _p(codes), _p(pl), _p(sf), int(bool(bf16_68))) != 0:
        raise ValueError("mxo_planes failed")
    return pl, sf
