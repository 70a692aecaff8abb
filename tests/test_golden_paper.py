"""The oracles against numbers the paper prints (tests/golden/paper_numbers.txt,
each line with its place in the paper), compared at the precision printed."""
import os

import numpy as np
import pytest

from oracle import alloc as A
from oracle import mxo

HERE = os.path.dirname(os.path.abspath(__file__))


def golden():
    out = {}
    with open(os.path.join(HERE, "golden", "paper_numbers.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            name, value, decimals = line.split("|")[0].split()
            out[name] = (float(value), int(decimals))
    return out


G = golden()


def printed(name, x):
    value, decimals = G[name]
    assert round(x, decimals) == pytest.approx(value), f"{name}: {x} prints as {round(x, decimals)}, not {value}"


def test_scale_overhead_per_element():
    """The compact storage: a 4-bit block is 16 code bytes + 1 scale byte, an
    8-bit block 32 + 1 (6-bit codes take whole bytes, as 8-bit ones do)."""
    N, K = 256, 4096
    for b in (4, 8):
        bits = np.full(K // 32, b, np.uint8)
        per_element = mxo.weight_bytes(N, K, bits, with_planes=False) * 8 / (N * K)
        printed("scale_bits_per_element", per_element - b)


def test_one_eight_bit_block_of_4096_columns_is_the_4_03_budget():
    """Alg. 3 with no 6-bit columns (R = 0): block 0 (the 32 most sensitive
    columns) at 8 bits, the rest at 4: average width and the share of
    operations at the higher precision."""
    s = np.random.default_rng(7).random(4096)
    perm, bits, n6 = A.allocate_layer(s, R=0.0, s_layer=1.0)
    assert n6 == 0 and bits[0] == 8 and np.all(bits[1:] == 4)
    printed("bits_4_8_one_block_d4096", A.average_width([bits], [4096]))
    printed("higher_precision_share_at_4_03", float(np.sum(bits > 4)) * 32 / 4096)
