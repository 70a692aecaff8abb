"""The one-token decode path's work split (host code, no GPU): every CTA of a
launch gets an equal share of its problem's weight bytes, cut at slot
boundaries, the shares tile the weight stream exactly once, and the CTAs
that share a 128-row group are a contiguous run of at most a few.

The split is read through the C ABI's test hook (mxs_test_gemv_split) and
checked here against the packed layout's own arithmetic: a row group of a
map with n4 4-bit blocks out of nb is 2176 * n4 + 4224 * (nb - n4) bytes,
4-bit slots first (128 rows x 16 code bytes + 128 scale bytes each), then
6/8-bit slots (128 x 32 + 128)."""
import ctypes

import numpy as np
import pytest

from paper_2607_17733_gb300 import inputs as I
from paper_2607_17733_gb300 import mxs


def _split(problems, sms, hook="mxs_test_gemv_split"):
    """problems: [(K, bits, N)] -> (ncta list, spans [n, 4])."""
    L = mxs.lib()
    n = len(problems)
    Ks = (ctypes.c_int64 * n)(*[K for K, _, _ in problems])
    Ns = (ctypes.c_int64 * n)(*[N for _, _, N in problems])
    keep = [np.ascontiguousarray(b, np.uint8) for _, b, _ in problems]
    bp = (ctypes.c_void_p * n)(*[b.ctypes.data for b in keep])
    ncta = np.zeros(n, np.int32)
    spans = np.zeros((256, 4), np.int32)
    total = getattr(L, hook)(Ks, bp, Ns, n, sms, ncta.ctypes.data, spans.ctypes.data)
    assert total > 0, mxs.last_error()
    assert total == int(ncta.sum())
    return [int(c) for c in ncta], spans[:total]


def _weights():
    """The build's split weights (percent of a slot's bytes): 4-bit slots in
    the one-token split, 6/8-bit slots in the tensor-core one."""
    c4 = ctypes.c_int(0)
    c8 = mxs.lib().mxs_test_dtc_split_weight(ctypes.byref(c4))
    return c4.value, c8


def _check_problem(K, bits, N, spans, w4=100, w8=100, stage=False):
    """Each CTA's range, in bytes of the weight stream; the ranges tile it.
    Returns their sizes in bytes and weights.  w4, w8: a slot's weight in
    percent of its bytes; the weighted shares are equal up to the rounding of
    each cut to the next slot (stage: to the next plane stage of four 4-bit or
    two 6/8-bit slots, which each cut must then fall on)."""
    nb = K // 32
    n4 = int(np.sum(bits == 4))
    GB = 2176 * n4 + 4224 * (nb - n4)
    G = (N + 127) // 128
    W = G * GB

    def off(s):  # byte offset of slot boundary s within a group
        return 2176 * s if s <= n4 else 2176 * n4 + 4224 * (s - n4)

    def cost(s):  # weight of the group's slots before boundary s
        return 2176 * w4 * min(s, n4) + 4224 * w8 * max(0, s - n4)

    def on_stage(s):  # a plane-stage boundary of the group
        return s in (n4, nb) or (s % 4 == 0 if s < n4 else (s - n4) % 2 == 0)

    pos = 0
    sizes, costs = [], []
    for g0, s0, g1, s1 in spans.tolist():  # Python ints: no fixed-width overflow
        assert 0 <= g0 <= g1 < G and 0 <= s0 < nb and 1 <= s1 <= nb
        if stage:
            assert on_stage(s0) and on_stage(s1)
        a, b = g0 * GB + off(s0), g1 * GB + off(s1)
        assert a == pos and b > a  # contiguous, nonempty
        sizes.append(b - a)
        costs.append(g1 * cost(nb) + cost(s1) - g0 * cost(nb) - cost(s0))
        pos = b
    assert pos == W  # the whole stream, once
    sizes, costs = np.array(sizes), np.array(costs)
    # each share is the ideal weight / n, each cut moved by less than one
    # rounding step
    ideal = G * cost(nb) / len(spans)
    step = max(4 * 2176 * w4, 2 * 4224 * w8) if stage else max(2176 * w4, 4224 * w8)
    assert costs.min() > ideal - step - 1 and costs.max() < ideal + step + 1
    return sizes, costs
    # each CTA meets at most one group partly at either end; the CTAs that
    # share a group are a contiguous run
    for g in range(G):
        who = [k for k, (g0, s0, g1, s1) in enumerate(spans) if g0 <= g <= g1]
        assert who == list(range(who[0], who[-1] + 1))
        assert len(who) < 1 << 16  # the arrival count's field
    return sizes


@pytest.mark.parametrize("K,N,p,sms", [
    (8192, 8192, (0.6, 0.3, 0.1), 152),     # a 70B o projection: 64 groups over 152 SMs
    (28672, 8192, (0.6, 0.3, 0.1), 152),    # 70B down
    (8192, 28672, (0.95, 0.04, 0.01), 152),  # 70B gate, mostly 4-bit
    (4096, 4096, (0.85, 0.1, 0.05), 148),
    (4096, 14336, (0, 0, 1), 152),          # every block 8-bit
    (4096, 14336, (1, 0, 0), 152),          # every block 4-bit
    (32, 5, (1, 0, 0), 152),                # one block, one short group: one CTA
    (96, 300, (0, 1, 0), 152),              # a few small slots
    (65536, 129, (0.5, 0.3, 0.2), 152),     # the longest K, a last group of one row
])
def test_split_single(K, N, p, sms):
    bits = I.width_map(K // 32, *p, I.rng(401, K, N))
    ncta, spans = _split([(K, bits, N)], sms)
    assert 1 <= ncta[0] <= min(sms, 256)
    _check_problem(K, bits, N, spans, w4=_weights()[0])
    nb = K // 32
    n4 = int(np.sum(bits == 4))
    W = ((N + 127) // 128) * (2176 * n4 + 4224 * (nb - n4))
    # as many CTAs as the SMs, unless a share would drop below 32 KB
    assert ncta[0] == min(sms, max(1, min(W // 4225, W // 32768)))


@pytest.mark.parametrize("hook", ["mxs_test_gemv_split", "mxs_test_dtc_split"])
def test_split_groups_share_the_sms_by_bytes(hook):
    """q/k/v and gate/up of a 70B layer: the CTAs go to the problems in
    proportion to their bytes, so the heaviest share per CTA is within a few
    percent of the launch's average."""
    w4, w8 = _weights()
    kw = dict(w4=w4) if hook == "mxs_test_gemv_split" else dict(w8=w8, stage=True)
    for shapes in ([(8192, 8192), (8192, 1024), (8192, 1024)], [(8192, 28672), (8192, 28672)]):
        probs = [(K, I.llama70b_layer_map(K, 7, 80, I.rng(5, 0, i)), N) for i, (K, N) in enumerate(shapes)]
        ncta, spans = _split(probs, 152, hook)
        assert sum(ncta) == 152
        base, worst, total = 0, 0, 0
        for (K, bits, N), c in zip(probs, ncta):
            _, costs = _check_problem(K, bits, N, spans[base:base + c], **kw)
            base += c
            worst = max(worst, costs.max())
            total += costs.sum()
        assert worst <= 1.06 * total / 152


@pytest.mark.parametrize("K,N,p,sms", [
    (8192, 8192, (0.6, 0.3, 0.1), 152),
    (28672, 8192, (0.6, 0.3, 0.1), 152),
    (8192, 28672, (0.95, 0.04, 0.01), 152),
    (4096, 4096, (0.85, 0.1, 0.05), 148),
    (4096, 14336, (0, 0, 1), 152),
    (4096, 14336, (1, 0, 0), 152),
    (32, 5, (1, 0, 0), 152),
    (96, 300, (0, 1, 0), 152),
    (65536, 129, (0.5, 0.3, 0.2), 152),
    (1056, 700, (0.5, 0.3, 0.2), 152),      # odd runs: 4-bit and 6/8-bit ends off a plane stage
])
def test_dtc_split_single(K, N, p, sms):
    """The tensor-core decode split: plane-stage cuts, shares of equal weight,
    as many CTAs as the SMs unless a share would drop below 64 KB."""
    bits = I.width_map(K // 32, *p, I.rng(402, K, N))
    ncta, spans = _split([(K, bits, N)], sms, "mxs_test_dtc_split")
    _check_problem(K, bits, N, spans, w8=_weights()[1], stage=True)
    nb = K // 32
    n4 = int(np.sum(bits == 4))
    W = ((N + 127) // 128) * (2176 * n4 + 4224 * (nb - n4))
    assert ncta[0] == min(sms, 256, max(1, min(W // 8705, W // 65536)))


def test_split_rejects_bad_arguments():
    L = mxs.lib()
    bits = np.full(4, 4, np.uint8)
    K = (ctypes.c_int64 * 1)(100)  # not a multiple of 32
    N = (ctypes.c_int64 * 1)(16)
    bp = (ctypes.c_void_p * 1)(bits.ctypes.data)
    out = np.zeros(4 * 256, np.int32)
    n = np.zeros(1, np.int32)
    assert L.mxs_test_gemv_split(K, bp, N, 1, 152, n.ctypes.data, out.ctypes.data) == -2
    K[0] = 128
    assert L.mxs_test_gemv_split(K, bp, N, 0, 152, n.ctypes.data, out.ctypes.data) == -1
    assert L.mxs_test_gemv_split(K, bp, N, 1, 0, n.ctypes.data, out.ctypes.data) == -1
