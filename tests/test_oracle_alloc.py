"""Pins of the allocation oracle (oracle/alloc.py) to the paper and to
mathematics independent of its code: exact rational sums, an explicit
column-by-column construction of the triplet allocation (the statement of
Theorem 1), a root found by bisection, hand-worked examples of Alg. 3 and a
selection sort with the tie rule written out."""
from fractions import Fraction

import numpy as np
import pytest

from oracle import alloc as A
from paper_2607_17733_gb300 import inputs as I


def _bits(values):
    return I.f32_to_bf16_bits(np.asarray(values, dtype=np.float32))


# ---------------------------------------------------------------- Alg. 1
def test_column_sensitivity_is_the_exact_sum_of_squares():
    """Every bf16 value is a dyadic rational: the exact sum of squares, in
    fractions, against the oracle's fp64 result (which may round once per add)."""
    g = np.random.default_rng(1)
    vals = g.standard_normal((9, 5)).astype(np.float32) * np.array([1, 1e-3, 1e3, 3e-38, 1e18], np.float32)
    xb = _bits(vals)
    got = A.column_sensitivity(xb)
    x = A.bf16_to_f64(xb)
    for j in range(x.shape[1]):
        exact = sum(Fraction(float(v)) ** 2 for v in x[:, j])
        assert abs(Fraction(float(got[j])) - exact) <= exact * Fraction(1, 2 ** 50)


def test_column_sensitivity_is_the_hessian_diagonal():
    """Small integer-valued activations: diag(X^T X) from an integer matrix product is exact."""
    g = np.random.default_rng(2)
    xi = g.integers(-50, 51, size=(64, 96))
    got = A.column_sensitivity(_bits(xi))
    want = np.diag(xi.T.astype(np.int64) @ xi.astype(np.int64)).astype(np.float64)
    assert np.array_equal(got, want)


def test_column_sensitivity_accumulates_over_samples():
    """Alg. 1 adds X^T X of every calibration sample: two batches give the sum of their parts."""
    g = np.random.default_rng(3)
    a = g.integers(-20, 21, size=(30, 64))
    b = g.integers(-20, 21, size=(17, 64))
    assert np.array_equal(A.column_sensitivity(_bits(a)) + A.column_sensitivity(_bits(b)),
                          A.column_sensitivity(_bits(np.vstack([a, b]))))


# ---------------------------------------------------------------- Theorem 1
D_IN = [128, 256, 4096]
S_LAYER = [0.5, 1.0, 0.25]


def _explicit_average(d_in, s_layer, R):
    """Theorem 1's setting built column by column: 32 columns at 8 bits, then
    R * S * (d - 32) columns at 6 bits (here an integer), the rest at 4 bits."""
    widths = []
    for d, s in zip(d_in, s_layer):
        n6 = Fraction(R) * Fraction(s) * (d - 32)
        assert n6.denominator == 1
        widths += [8] * 32 + [6] * int(n6) + [4] * (d - 32 - int(n6))
    return Fraction(sum(widths), len(widths))


def test_allocation_r_reaches_the_average_of_an_explicit_allocation():
    R = Fraction(1, 2)  # R * S * (d - 32) = 24, 112, 508 columns: whole numbers
    B = _explicit_average(D_IN, S_LAYER, R)
    assert abs(A.allocation_r(D_IN, S_LAYER, float(B)) - 0.5) < 1e-12


def test_allocation_r_matches_bisection():
    """The continuous average width as a function of R (fractional column
    counts), solved for B = 4.5 by bisection."""
    d = np.array([4096, 4096, 14336, 1024], float)
    s = np.array([1.0, 0.3, 0.7, 0.05])
    B = 4.5

    def avg(R):
        n6 = R * s * (d - 32)
        return float((8 * 32 * len(d) + np.sum(6 * n6 + 4 * (d - 32 - n6))) / d.sum())

    lo, hi = 0.0, 10.0
    for _ in range(200):
        mid = 0.5 * (lo + hi)
        lo, hi = (mid, hi) if avg(mid) < B else (lo, mid)
    assert abs(A.allocation_r(d, s, B) - lo) < 1e-12


def test_allocation_r_is_zero_at_the_eight_and_four_bit_floor():
    """With no 6-bit columns the average is (8*32*n + 4*sum(d - 32)) / sum(d)."""
    d = [4096, 14336]
    B = (8 * 32 * 2 + 4 * sum(x - 32 for x in d)) / sum(d)
    assert abs(A.allocation_r(d, [0.4, 0.9], B)) < 1e-12


# ---------------------------------------------------------------- Alg. 3
def test_allocate_layer_hand_example():
    """K = 256, R * S = 1/4: N6 = floor(224 / 4) = 56 columns, one whole 6-bit block."""
    s = np.arange(256, dtype=np.float64)[::-1].copy()  # column 0 most sensitive
    perm, bits, n6 = A.allocate_layer(s, R=0.5, s_layer=0.5)
    assert n6 == 56
    assert list(bits) == [8, 6, 4, 4, 4, 4, 4, 4]
    assert np.array_equal(perm, np.arange(256))


def test_allocate_layer_clamps_the_six_bit_count():
    perm, bits, n6 = A.allocate_layer(np.ones(256), R=3.0, s_layer=1.0)
    assert n6 == 224 and list(bits) == [8] + [6] * 7
    perm, bits, n6 = A.allocate_layer(np.ones(256), R=0.0, s_layer=1.0)
    assert n6 == 0 and list(bits) == [8] + [4] * 7


def _selection_order(s):
    """Descending order, ties by index, by repeated selection of the maximum."""
    left = list(range(len(s)))
    out = []
    while left:
        best = left[0]
        for j in left[1:]:
            if s[j] > s[best]:
                best = j
        out.append(best)
        left.remove(best)
    return out


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_column_order_matches_selection_with_ties(seed):
    g = np.random.default_rng(seed)
    s = g.integers(0, 12, size=96).astype(np.float64)  # many equal keys
    assert list(A.column_order(s)) == _selection_order(list(s))


def test_block_flooring_keeps_the_average_at_or_below_b():
    g = np.random.default_rng(5)
    d = [4096, 1024, 14336]
    sl = [1.0, 0.2, 0.6]
    B = 4.4
    R = A.allocation_r(d, sl, B)
    maps = [A.allocate_layer(g.random(k), R, s)[1] for k, s in zip(d, sl)]
    avg = A.average_width(maps, d)
    assert avg <= B + 1e-12
    # each layer loses fewer than 64 columns of 6 bits (column floor + block floor)
    assert B - avg < 2 * 64 * len(d) / sum(d)


def test_n6_is_the_floor_of_the_product():
    """Alg. 3 takes the floor of R * S_layer * (d_in - 32) for the 6-bit column
    count: a fractional part above one half still rounds down."""
    d = 4096  # d - 32 = 4064
    assert A.n6_columns(d, 100.75 / 4064, 1.0) == 100
    assert A.n6_columns(d, 200.6 / 4064, 1.0) == 200
    assert A.n6_columns(d, 0.9 / 4064, 1.0) == 0
    assert A.n6_columns(d, 2 * 301.7 / 4064, 0.5) == 301
