"""Pins of the CPU oracle against facts that do not come from the oracle itself.

Each test fixes one part of the oracle by an independent route: brute force
over every grid point, exact rational arithmetic, a library routine that
computes the same thing another way, closed forms, or invariants.  Together
they are chosen so that a dropped term, a wrong sign, an off-by-one exponent,
a transposed operand or a wrong tie rule fails at least one of them.
"""
import math
import random
from fractions import Fraction

import numpy as np
import pytest

from oracle import mxo
from paper_2607_17733_gb300 import inputs as I
import mxformat

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")


# --------------------------------------------------------------- brute force
def brute_block(xs, b, rounding):
    """Nearest point of the b-bit grid (independent of the oracle's formulae).

    E is the largest integer in [-127, 127] with 2^E <= max|x| (found by
    search, not by log2/frexp); the grid is {m * 2^(E-(b-2)) : |m| <= 2^(b-1)-1};
    every element takes the grid point at the smallest exact distance, ties
    going to the even m (RNE) or to the larger |m| (RHAZ)."""
    if any(not math.isfinite(x) for x in xs):
        return 255, [0] * 32
    fx = [Fraction(x) for x in xs]
    amax = max(abs(f) for f in fx)
    E = -127
    for e in range(-127, 128):
        if Fraction(2) ** e <= amax:
            E = e
    step = Fraction(2) ** (E - (b - 2))
    Q = 2 ** (b - 1) - 1
    out = []
    for f in fx:
        best_d, best_m = None, None
        for m in range(-Q, Q + 1):
            d = abs(f - m * step)
            if best_d is None or d < best_d:
                best_d, best_m = d, m
            elif d == best_d:
                if rounding == mxo.RNE and m % 2 == 0:
                    best_m = m
                if rounding == mxo.RHAZ and abs(m) > abs(best_m):
                    best_m = m
        out.append(best_m)
    return E + 127, out


def random_bf16_block(rs, spread):
    """32 bf16-representable values with a random dynamic range."""
    x = np.array([rs.gauss(0, 1) * 2.0 ** rs.randint(-spread, spread) for _ in range(32)], np.float32)
    return [float(v) for v in I.bf16_bits_to_f32(I.f32_to_bf16_bits(x))]


@pytest.mark.parametrize("b", [3, 4, 6, 8])
@pytest.mark.parametrize("rounding", [mxo.RNE, mxo.RHAZ])
def test_quantize_matches_brute_force(b, rounding):
    rs = random.Random(1000 * b + rounding)
    for trial in range(40):
        xs = random_bf16_block(rs, spread=trial % 6)
        if trial % 5 == 0:  # plant exact ties: values halfway between grid points
            E = rs.randint(-3, 3)
            step = 2.0 ** (E - (b - 2))
            xs[0] = 2.0 ** E * 1.5  # fixes amax's exponent at E
            for i in range(1, 32):
                m = rs.randint(-(2 ** (b - 1)) + 1, 2 ** (b - 1) - 2)
                xs[i] = (m + 0.5) * step
        s, codes = mxo.quantize_block(xs, b, rounding)
        bs, bcodes = brute_block(xs, b, rounding)
        assert s == bs
        assert list(codes) == bcodes


def test_tie_rule_hand_cases():
    # b=4, amax in [1,2) -> E = 0, step 2^-2; 0.625 = 2.5 steps, 0.375 = 1.5 steps
    xs = [1.0, 0.625, -0.625, 0.375, -0.375, 0.875, 1.875] + [0.0] * 25
    s, rne = mxo.quantize_block(xs, 4, mxo.RNE)
    _, rhaz = mxo.quantize_block(xs, 4, mxo.RHAZ)
    assert s == 127
    assert list(rne[:7]) == [4, 2, -2, 2, -2, 4, 7]   # 3.5 -> 4 (even); 7.5 -> 8 -> clamp 7
    assert list(rhaz[:7]) == [4, 3, -3, 2, -2, 4, 7]  # 3.5 -> 4 (away); 7.5 -> 8 -> clamp 7


@pytest.mark.parametrize("b", [4, 6, 8])
def test_exact_round_trip(b):
    """Blocks already on the grid (with max|m| >= 2^(b-2)) come back unchanged."""
    rs = random.Random(b)
    Q = 2 ** (b - 1) - 1
    for _ in range(200):
        E = rs.randint(-120, 120)
        m = [rs.randint(-Q, Q) for _ in range(32)]
        m[rs.randrange(32)] = rs.choice([-1, 1]) * rs.randint(2 ** (b - 2), Q)
        xs = [mi * 2.0 ** (E - (b - 2)) for mi in m]
        for rounding in (mxo.RNE, mxo.RHAZ):
            s, codes = mxo.quantize_block(xs, b, rounding)
            assert s == E + 127
            assert list(codes) == m


@pytest.mark.parametrize("b", [4, 6, 8])
def test_idempotence(b):
    """q(dq(q(x))) == q(x) for codes and scales."""
    rs = random.Random(17 + b)
    for trial in range(200):
        xs = random_bf16_block(rs, spread=trial % 8)
        s, codes = mxo.quantize_block(xs, b)
        if not any(codes):
            continue
        xs2 = [mxo.element_value(int(c), s, b) for c in codes]
        s2, codes2 = mxo.quantize_block(xs2, b)
        assert s2 == s and list(codes2) == list(codes)


@pytest.mark.parametrize("b", [4, 6, 8])
def test_all_zero_block(b):
    s, codes = mxo.quantize_block([0.0] * 32, b)
    assert s == 0 and not codes.any()


@pytest.mark.parametrize("b", [4, 6, 8])
def test_single_outlier_block(b):
    """One outlier sets the scale; it lands in [2^(b-2), Q]; values below half
    a step vanish."""
    Q = 2 ** (b - 1) - 1
    xs = [0.01 * (i % 7 - 3) for i in range(32)]
    xs[5] = 50.0  # floor(log2 50) = 5
    s, codes = mxo.quantize_block(xs, b)
    assert s == 127 + 5
    assert 2 ** (b - 2) <= codes[5] <= Q
    half_step = 2.0 ** (5 - (b - 2)) / 2
    for i, x in enumerate(xs):
        if i != 5 and abs(x) < half_step:
            assert codes[i] == 0


def test_subnormal_and_special_blocks():
    tiny = [2.0 ** -133 * (i % 5) for i in range(32)]  # bf16 subnormals
    s, codes = mxo.quantize_block(tiny, 8)
    assert s == 0
    # E clamps at -127: element value m * 2^(-127-6) -> m = x / 2^-133 exactly
    assert list(codes) == [i % 5 for i in range(32)]
    for special in (math.inf, -math.inf, math.nan):
        xs = [1.0] * 32
        xs[3] = special
        s, codes = mxo.quantize_block(xs, 4)
        assert s == 255 and not codes.any()
    big = [3.3e38] + [0.0] * 31  # largest binade of bf16: E = 127, S = 254
    assert mxo.quantize_block(big, 8)[0] == 254


def test_row_quantizer_agrees_with_block_quantizer():
    g = I.rng(5, 1)
    bits = I.width_map(8, 0.5, 0.25, 0.25, g)
    xb = I.activations_bf16(3, bits, g, 0.05, outlier_scale=50.0)
    scales, codes = mxo.quantize_bf16(xb, bits)
    xf = I.bf16_bits_to_f32(xb).astype(np.float64)
    for r in range(3):
        for kb in range(8):
            s, c = mxo.quantize_block(xf[r, 32 * kb:32 * kb + 32], int(bits[kb]))
            assert s == scales[r, kb] and np.array_equal(c, codes[r, 32 * kb:32 * kb + 32])


# --------------------------------------------------------------- summation
def test_fsum_matches_python_math_fsum():
    rs = random.Random(3)
    cases = [[1e100, 1.0, -1e100], [1.0, 1e-16, 1e-16], [0.1] * 10, [2.0 ** 60, 1.0, -(2.0 ** 60)]]
    for _ in range(300):
        n = rs.randint(1, 60)
        cases.append([rs.uniform(-1, 1) * 2.0 ** rs.randint(-60, 60) for _ in range(n)])
    # halfway cases where the deciding bit sits in a far partial
    cases.append([1.0, 2.0 ** -53, 2.0 ** -106])
    cases.append([1.0, 2.0 ** -53, -(2.0 ** -106)])
    cases.append([1.0 + 2.0 ** -52, 2.0 ** -53])
    for c in cases:
        assert mxo.fsum(c) == math.fsum(c)


# --------------------------------------------------------------- GEMM
def exact_gemm(bits, ac, as_, wc, ws):
    """y = sum_k dq(a)[m,k] * dq(w)[n,k] in exact rationals, rounded once."""
    M, K = ac.shape
    N = wc.shape[0]
    y = np.zeros((M, N))
    for m in range(M):
        for n in range(N):
            acc = Fraction(0)
            for k in range(K):
                kb = k // 32
                b = int(bits[kb])
                va = Fraction(int(ac[m, k])) * Fraction(2) ** (int(as_[m, kb]) - 127 - (b - 2))
                vw = Fraction(int(wc[n, k])) * Fraction(2) ** (int(ws[n, kb]) - 127 - (b - 2))
                acc += va * vw
            y[m, n] = float(acc)
    return y


def test_gemm_exact_rational_tiny():
    g = I.rng(11, 2)
    for M, N, nb in [(1, 1, 1), (2, 3, 2), (3, 2, 2)]:
        bits = np.array([[4, 6, 8][i % 3] for i in range(nb)], np.uint8)
        a = I.activations_bf16(M, bits, g, 0.1, outlier_scale=40.0)
        w = I.normal_bf16((N, 32 * nb), 0.02, g)
        as_, ac = mxo.quantize_bf16(a, bits)
        ws, wc = mxo.quantize_bf16(w, bits)
        y, ab = mxo.gemm(bits, ac, as_, wc, ws)
        assert np.array_equal(y, exact_gemm(bits, ac, as_, wc, ws))
        assert np.all(ab >= np.abs(y))


def test_gemm_wide_exponent_spread_is_exact():
    """Terms spanning ~200 binades: only an exact summation survives this."""
    bits = np.array([8, 8, 8], np.uint8)
    a = np.zeros((1, 96), np.float64)
    w = np.zeros((1, 96), np.float64)
    a[0, 0], w[0, 0] = 2.0 ** 100, 1.0
    a[0, 32], w[0, 32] = 1.0, 1.0
    a[0, 64], w[0, 64] = -(2.0 ** 100), 1.0
    ab = I.f32_to_bf16_bits(a.astype(np.float32))
    wb = I.f32_to_bf16_bits(w.astype(np.float32))
    as_, ac = mxo.quantize_bf16(ab, bits)
    ws, wc = mxo.quantize_bf16(wb, bits)
    y, _ = mxo.gemm(bits, ac, as_, wc, ws)
    assert y[0, 0] == 1.0


@pytest.mark.parametrize("b", [4, 6, 8])
def test_gemm_integer_valued_equals_int64_matmul(b):
    """Integer inputs with every block max in [2^(b-2), Q] sit on the grid with
    step 1, so the MXINT product is the plain integer matmul."""
    rs = np.random.default_rng(b)
    Q = 2 ** (b - 1) - 1
    M, N, nb = 5, 7, 4
    K = 32 * nb

    def draw(rows):
        v = rs.integers(-Q, Q + 1, size=(rows, K))
        for r in range(rows):
            for kb in range(nb):
                v[r, 32 * kb + rs.integers(0, 32)] = rs.choice([-1, 1]) * rs.integers(2 ** (b - 2), Q + 1)
        return v

    A, W = draw(M), draw(N)
    bits = np.full(nb, b, np.uint8)
    as_, ac = mxo.quantize_bf16(I.f32_to_bf16_bits(A.astype(np.float32)), bits)
    ws, wc = mxo.quantize_bf16(I.f32_to_bf16_bits(W.astype(np.float32)), bits)
    assert np.array_equal(ac, A) and np.array_equal(wc, W)
    y, _ = mxo.gemm(bits, ac, as_, wc, ws)
    assert np.array_equal(y, (A.astype(np.int64) @ W.T.astype(np.int64)).astype(np.float64))


def test_gemm_entries_match_full_gemm_and_transpose_rule():
    g = I.rng(12, 3)
    bits = I.width_map(6, 0.5, 0.3, 0.2, g)
    a = I.activations_bf16(4, bits, g, 0.02, outlier_scale=50.0)
    w = I.normal_bf16((9, 192), 0.02, g)
    as_, ac = mxo.quantize_bf16(a, bits)
    ws, wc = mxo.quantize_bf16(w, bits)
    y, ab = mxo.gemm(bits, ac, as_, wc, ws)
    rows = np.array([0, 3, 2, 1])
    cols = np.array([8, 0, 4, 4])
    ye, abe = mxo.gemm_entries(bits, ac, as_, wc, ws, rows, cols)
    assert np.array_equal(ye, y[rows, cols]) and np.array_equal(abe, ab[rows, cols])
    # swapping the roles of A and W transposes y (same map on both sides)
    yt, _ = mxo.gemm(bits, wc, ws, ac, as_)
    assert np.array_equal(yt, y.T)


def test_gemm_nan_block_propagates():
    """An Inf or NaN in a block (scale byte 255) makes every output that block
    enters NaN, from either operand: an activation block its row, a weight
    block its column; the other outputs stay finite."""
    bits = np.array([4, 8], np.uint8)
    a = np.ones((2, 64), np.float32)
    a[0, 40] = np.inf
    w = np.ones((3, 64), np.float32)
    w[2, 5] = np.nan
    as_, ac = mxo.quantize_bf16(I.f32_to_bf16_bits(a), bits)
    ws, wc = mxo.quantize_bf16(I.f32_to_bf16_bits(w), bits)
    assert as_[0, 1] == 255 and ws[2, 0] == 255
    y, _ = mxo.gemm(bits, ac, as_, wc, ws)
    assert np.all(np.isnan(y[0])) and np.all(np.isnan(y[:, 2]))
    assert np.all(np.isfinite(y[1, :2]))


# --------------------------------------------------------------- storage format
def test_e4m3_encoder_matches_torch_and_table():
    torch = pytest.importorskip("torch")
    if not hasattr(torch, "float8_e4m3fn"):
        pytest.skip("torch without float8_e4m3fn")
    values = sorted({m / 4 for m in range(-7, 8)} | {h / 2 for h in range(-4, 4)}
                    | {l / 16 for l in range(8)} | {h / 4 for h in range(-8, 8)}
                    | {l / 64 for l in range(16)})
    for v in values:
        code = mxo.e4m3_encode(v)
        assert code >= 0
        ref = torch.tensor([v], dtype=torch.float32).to(torch.float8_e4m3fn).view(torch.uint8).item()
        assert code == ref, v
        assert mxformat.E4M3_TABLE[code] == v
    assert mxo.e4m3_encode(17.0) == -1 and mxo.e4m3_encode(0.3) == -1
    # every finite e4m3 value, subnormals and -0 included, encodes to its own code
    for code in range(256):
        if code in (0x7F, 0xFF):  # the NaN codes
            continue
        v = float(mxformat.E4M3_TABLE[code])
        if code == 0x80:
            v = -0.0
        assert mxo.e4m3_encode(v) == code, hex(code)


@pytest.mark.parametrize("b", [4, 6, 8])
def test_element_value_of_a_nan_block(b):
    """Reading R5: a block holding Inf or NaN has scale byte 255, and every
    element of it reads as NaN, whatever its code."""
    for m in (-(2 ** (b - 1) - 1), -1, 0, 1, 2 ** (b - 1) - 1):
        assert math.isnan(mxo.element_value(m, 255, b))


@pytest.mark.parametrize("b", [6, 8])
def test_plane_digits_cover_every_code(b):
    """Every m in [-Q, Q] splits into two exactly representable e4m3 digits
    whose sum is m * 2^-(b-2)."""
    Q = 2 ** (b - 1) - 1
    bits = np.full(1, b, np.uint8)
    codes = np.zeros((2 * Q + 1, 32), np.int8)
    codes[:, 0] = np.arange(-Q, Q + 1)
    scales = np.full((2 * Q + 1, 1), 127, np.uint8)
    pl, _ = mxo.planes(bits, scales, codes)
    hi = mxformat.E4M3_TABLE[pl[:, 128 * 0 + 0]]
    lo = mxformat.E4M3_TABLE[pl[:, 32]]
    assert np.array_equal((hi + lo) * 2.0 ** (b - 2), np.arange(-Q, Q + 1).astype(np.float64))
    assert np.all(lo >= 0)


@pytest.mark.parametrize("b", [6, 8])
def test_plane_bf16_form_is_the_exact_block_value(b):
    """bf16 form of a 6/8-bit block: every m in [-Q, Q] under scale bytes
    from the bottom (subnormal results) to the top of the range is the bf16
    whose value is exactly m * 2^(S-127-(b-2)) (compared with numpy's exact
    fp64 ldexp), and the NaN scale byte gives bf16 NaN."""
    Q = 2 ** (b - 1) - 1
    bits = np.full(1, b, np.uint8)
    m = np.arange(-Q, Q + 1)
    for S in (0, 1, 7, 100, 127, 200, 254, 255):
        codes = np.zeros((2 * Q + 1, 32), np.int8)
        codes[:, 0] = m
        codes[:, 31] = -m
        scales = np.full((2 * Q + 1, 1), S, np.uint8)
        pl, _ = mxo.planes(bits, scales, codes, bf16_68=True)
        h = pl[:, :64].copy().view(np.uint16)
        got = (h.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
        if S == 255:
            assert np.all(h == 0x7FC0)
            continue
        want = np.ldexp(m.astype(np.float64), S - 127 - (b - 2))
        assert np.array_equal(got[:, 0], want) and np.array_equal(got[:, 31], -want)
        assert np.all(got[:, 1:31] == 0)


def _random_quantized(seed, R, nb, p=(0.6, 0.25, 0.15)):
    g = I.rng(seed, 7)
    bits = I.width_map(nb, *p, g)
    x = I.activations_bf16(R, bits, g, 0.02, outlier_scale=50.0)
    scales, codes = mxo.quantize_bf16(x, bits)
    return bits, scales, codes


def test_pack_act_round_trip_and_size():
    bits, scales, codes = _random_quantized(1, 5, 13)
    pc, ps = mxo.pack_act(bits, scales, codes)
    n4 = int(np.sum(bits == 4))
    assert pc.shape == (5, 16 * n4 + 32 * (13 - n4))
    s2, c2 = mxformat.decode_act(bits, pc, ps)
    assert np.array_equal(s2, scales) and np.array_equal(c2, codes)


@pytest.mark.parametrize("N", [1, 16, 37])
def test_pack_weight_round_trip(N):
    bits, scales, codes = _random_quantized(N, N, 11)
    buf = mxo.pack_weight(bits, scales, codes, with_planes=True)
    s2, c2 = mxformat.decode_weight(N, bits, buf)
    assert np.array_equal(s2, scales) and np.array_equal(c2, codes)
    compact = mxformat.weight_compact(N, bits)
    kp, nst = mxo.plane_shape(bits)
    pl = buf[compact:compact + N * kp].reshape(N, kp)
    sf_off = mxformat.align256(compact + N * kp)
    sf = buf[sf_off:sf_off + ((N + 127) // 128) * nst * 512]
    s3, c3 = mxformat.decode_planes(bits, pl, sf, bf16_68=True)  # weight planes: 6/8-bit blocks as bf16
    assert np.array_equal(s3, scales) and np.array_equal(c3, codes)
    pd, sfd = mxo.planes(bits, scales, codes)  # digit form (the oracle's second encoding; no kernel reads it)
    s4, c4 = mxformat.decode_planes(bits, pd, sfd.reshape(-1))
    assert np.array_equal(s4, scales) and np.array_equal(c4, codes)


def test_storage_accounting_matches_paper_scale_overhead():
    """Sec. 5.1: the 8-bit shared exponent of a 32-element block adds 0.25
    bit per element; a 4-bit block is stored in 16 + 1 bytes (4.25 bit/elem)."""
    N, nb = 4096, 128
    bits = np.full(nb, 4, np.uint8)
    compact = mxo.weight_bytes(N, 32 * nb, bits, with_planes=False)
    assert compact * 8 / (N * 32 * nb) == pytest.approx(4.25, abs=1e-3)
    bits8 = np.full(nb, 8, np.uint8)
    assert mxo.weight_bytes(N, 32 * nb, bits8, False) * 8 / (N * 32 * nb) == pytest.approx(8.25, abs=1e-3)
