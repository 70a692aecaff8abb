"""Pure-numpy decoder of the library's storage format (test helper).

Written from the format description only; it turns packed activation streams,
packed weight buffers and MMA planes back into natural-order codes and scales
so that tests can compare them with the oracle and check the layouts by eye.
"""
import numpy as np


def slot_blocks(bits):
    bits = np.asarray(bits)
    order = [np.flatnonzero(bits == w) for w in (4, 6, 8)]
    return np.concatenate(order).astype(np.int64), tuple(int(o.size) for o in order)


def align256(v):
    return (v + 255) // 256 * 256


def signmag4(n):
    n = n.astype(np.int16)
    return np.where(n & 8, -(n & 7), n & 7).astype(np.int8)


def signmag8(n):
    n = n.astype(np.int16)
    return np.where(n & 0x80, -(n & 0x7F), n & 0x7F).astype(np.int8)


def sext4(n):
    n = n.astype(np.int16)
    return np.where(n >= 8, n - 16, n).astype(np.int8)


def decode_act(bits, pcodes, pscales):
    """row-major grouped stream -> (scales [R,nb], codes [R,K]) in natural order."""
    sb, (n4, n6, n8) = slot_blocks(bits)
    R = pcodes.shape[0]
    nb = len(bits)
    K = 32 * nb
    codes = np.zeros((R, K), np.int8)
    scales = np.zeros((R, nb), np.uint8)
    for s, kb in enumerate(sb):
        scales[:, kb] = pscales[:, s]
        if s < n4:
            byts = pcodes[:, 16 * s:16 * s + 16]
            codes[:, 32 * kb + 0:32 * kb + 32:2] = sext4(byts & 0xF)
            codes[:, 32 * kb + 1:32 * kb + 32:2] = sext4(byts >> 4)
        else:
            off = 16 * n4 + 32 * (s - n4)
            codes[:, 32 * kb:32 * kb + 32] = pcodes[:, off:off + 32].view(np.int8)
    return scales, codes


def weight_compact(N, bits):
    sb, (n4, n6, n8) = slot_blocks(bits)
    G = (N + 127) // 128
    return align256(G * (2176 * n4 + 4224 * (n6 + n8)))


def decode_weight(N, bits, buf):
    """compact weight buffer -> (scales [N,nb], codes [N,K]) in natural order."""
    sb, (n4, n6, n8) = slot_blocks(bits)
    n68 = n6 + n8
    nb = len(bits)
    K = 32 * nb
    G = (N + 127) // 128
    GB = 2176 * n4 + 4224 * n68
    codes = np.zeros((128 * G, K), np.int8)
    scales = np.zeros((128 * G, nb), np.uint8)
    # element e of a 4-bit row: word e//8, byte (e%8)%4, low nibble if e%8 < 4
    e = np.arange(32)
    byte_of = 4 * (e // 8) + (e % 8) % 4
    high = (e % 8) >= 4
    for s, kb in enumerate(sb):
        for grp in range(G):
            rows = slice(128 * grp, 128 * grp + 128)
            if s < n4:
                base = grp * GB + 2176 * s
                blk = buf[base:base + 2048].reshape(128, 16)
                nib = np.where(high[None, :], blk[:, byte_of] >> 4, blk[:, byte_of] & 0xF)
                codes[rows, 32 * kb:32 * kb + 32] = signmag4(nib)
                scales[rows, kb] = buf[base + 2048:base + 2176]
            else:
                base = grp * GB + 2176 * n4 + 4224 * (s - n4)
                codes[rows, 32 * kb:32 * kb + 32] = signmag8(buf[base:base + 4096].reshape(128, 32))
                scales[rows, kb] = buf[base + 4096:base + 4224]
    return scales[:N], codes[:N]


def e4m3_value(code):
    code = int(code)
    s = -1.0 if code & 0x80 else 1.0
    e = (code >> 3) & 0xF
    f = code & 7
    if e == 0xF and f == 7:
        return float("nan")
    if e == 0:
        return s * f / 8.0 * 2.0 ** -6
    return s * (1 + f / 8.0) * 2.0 ** (e - 7)


E4M3_TABLE = np.array([e4m3_value(c) for c in range(256)])


def decode_planes(bits, planes, sf, bf16_68=False):
    """planes [R,Kp] + scale tiles -> (scales [R,nb], codes [R,K]) natural order.
    6/8-bit blocks as high/low e4m3 digits, or (bf16_68) as bf16 values
    m * 2^(S-127-(b-2))."""
    sb, (n4, n6, n8) = slot_blocks(bits)
    n68 = n6 + n8
    st4 = (n4 + 3) // 4
    nst = st4 + (n68 + 1) // 2
    R = planes.shape[0]
    nb = len(bits)
    # scale tiles: [tau][st][i][w][q] -> row 128 tau + 32 w + i
    tiles = sf.reshape(-1, nst, 32, 4, 4)
    scales = np.zeros((R, nb), np.uint8)
    for s, kb in enumerate(sb):
        if s < n4:
            st, qq = s // 4, s % 4
        else:
            st, qq = st4 + (s - n4) // 2, (s - n4) % 2
        col = tiles[:, st, :, :, qq]            # [tau, i, w]
        rows = col.transpose(0, 2, 1).reshape(-1)  # row = 128 tau + 32 w + i
        scales[:, kb] = rows[:R]
    codes = np.zeros((R, 32 * nb), np.int8)
    vals = E4M3_TABLE[planes]
    for s, kb in enumerate(sb):
        b = int(bits[kb])
        if s < n4:
            v = vals[:, 32 * s:32 * s + 32]
        elif bf16_68:
            off = 128 * st4 + 64 * (s - n4)
            h = planes[:, off:off + 64].copy().view(np.uint16).astype(np.uint32) << 16
            f = h.view(np.float32).astype(np.float64)
            e = scales[:, kb].astype(np.float64) - 127.0
            v = f * np.exp2(-e)[:, None]
            v = np.where(scales[:, kb][:, None] == 255, 0.0, v)  # NaN blocks hold zero codes
        else:
            off = 128 * st4 + 64 * (s - n4)
            v = vals[:, off:off + 32] + vals[:, off + 32:off + 64]
        codes[:, 32 * kb:32 * kb + 32] = np.rint(v * 2.0 ** (b - 2)).astype(np.int8)
    return scales, codes
