/*
 * mxo.c -- CPU oracle for the MXINT mixed-precision linear layer of MXSens.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may link, load or
 * call this file: only tests/, __graft_entry__.smoke() and the cpu_baseline /
 * reference legs of bench.py use it.  It shares no code, header, table or
 * constant with the CUDA library under paper_2607_17733_gb300/csrc.
 *
 * It is deliberately plain and slow: fp64 for every real number, int64 for
 * every integer dot product, no blocking, no fusion, no reordering beyond what
 * the definitions below state.
 *
 * What the paper fixes (arxiv 2607.17733):
 *   - MXINT: blocks of 32 consecutive values share one power-of-two scale, the
 *     elements are fixed-point integers processed by integer MACs (Sec. 2).
 *   - One mantissa width per block, widths {4, 6, 8}; 6/8-bit columns come in
 *     whole blocks (Sec. 4.1).
 *   - The shared scale is an 8-bit exponent per 32 elements, i.e. +0.25
 *     bit per element (Sec. 5.1).
 *   - Weights and activations of every linear layer are quantized
 *     (Appendix A.2).
 * What the paper leaves open and this oracle reads (the OCP MX v1.0 MXINT
 * definition the paper cites in Sec. 2 and Sec. 6):
 *   R1 shared exponent E = floor(log2(max_i |x_i|)), clamped to [-127, 127];
 *      stored as the E8M0 byte S = E + 127.  All-zero block: S = 0.
 *   R2 an element of a b-bit block is a two's-complement fixed-point number
 *      with b-2 fraction bits: value = m * 2^(E - (b-2)).
 *   R3 m = round(x * 2^((b-2) - E)); ties to even (MXO_RNE, default) or away
 *      from zero (MXO_RHAZ).
 *   R4 m is clamped to the symmetric range [-(2^(b-1)-1), 2^(b-1)-1].
 *   R5 a block holding a NaN or an infinity gets S = 255 (the E8M0 NaN) and
 *      all-zero codes; any dot product that touches it is NaN.
 * GEMM: y[m,n] = sum_kb 2^(Ea'+Ew') * sum_{i<32} a_i * w_i with E' = E-(b-2);
 * every block dot product is an exact int64, every term is exact in fp64, and
 * the terms are added with an exactly rounded summation (Shewchuk's
 * non-overlapping partials), so y is the correctly rounded real result.
 *
 * The packed layouts produced by mxo_pack_* and mxo_planes_* follow the
 * library's documented storage format (written independently from that
 * description, not from the library's code).
 */
#include <fenv.h>
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define MXO_RNE 0
#define MXO_RHAZ 1
#define MXO_BLOCK 32

/* ------------------------------------------------------------------ */
/* bf16 -> fp64 (exact: bf16 is the top half of an IEEE binary32)       */
/* ------------------------------------------------------------------ */
static double bf16_value(uint16_t bits)
{
    uint32_t u = (uint32_t)bits << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* ------------------------------------------------------------------ */
/* R1-R5: quantize one block of 32 values to width b (2..8).            */
/* ------------------------------------------------------------------ */
int mxo_quantize_block(const double *x, int b, int rounding, uint8_t *scale, int8_t *m)
{
    if (b < 2 || b > 8) return -1;
    if (rounding != MXO_RNE && rounding != MXO_RHAZ) return -1;
    if (fegetround() != FE_TONEAREST) return -2; /* nearbyint must be ties-to-even */

    int finite = 1;
    double amax = 0.0;
    for (int i = 0; i < MXO_BLOCK; ++i) {
        if (!isfinite(x[i])) finite = 0;
        else if (fabs(x[i]) > amax) amax = fabs(x[i]);
    }
    if (!finite) { /* R5 */
        *scale = 255;
        for (int i = 0; i < MXO_BLOCK; ++i) m[i] = 0;
        return 0;
    }

    /* R1: floor(log2(amax)); frexp gives amax = f * 2^e with f in [0.5, 1). */
    int E;
    if (amax == 0.0) {
        E = -127;
    } else {
        int e;
        frexp(amax, &e);
        E = e - 1;
        if (E < -127) E = -127;
        if (E > 127) E = 127;
    }
    *scale = (uint8_t)(E + 127);

    const int Q = (1 << (b - 1)) - 1; /* R4 */
    for (int i = 0; i < MXO_BLOCK; ++i) {
        double v = ldexp(x[i], (b - 2) - E); /* exact: a power-of-two scaling */
        double r = (rounding == MXO_RHAZ) ? round(v) : nearbyint(v); /* R3 */
        if (r > Q) r = Q;
        if (r < -Q) r = -Q;
        m[i] = (int8_t)r;
    }
    return 0;
}

/* value of one element: m * 2^(S - 127 - (b-2)); NaN for S = 255 (R2, R5) */
double mxo_element_value(int8_t m, uint8_t scale, int b)
{
    if (scale == 255) return NAN;
    return ldexp((double)m, (int)scale - 127 - (b - 2));
}

/* ------------------------------------------------------------------ */
/* Row quantization: R rows of K bf16 values (row stride ld elements),  */
/* block kb of every row has width bits[kb].  Outputs in natural order: */
/* scales[R, K/32], codes[R, K] (one int8 per element).                 */
/* ------------------------------------------------------------------ */
int mxo_quantize_bf16(const uint16_t *x, int64_t R, int64_t K, int64_t ld,
                      const uint8_t *bits, int rounding, uint8_t *scales, int8_t *codes)
{
    if (K % MXO_BLOCK != 0 || R < 0 || ld < K) return -1;
    const int64_t nb = K / MXO_BLOCK;
    int err = 0;
#pragma omp parallel for schedule(static) reduction(| : err)
    for (int64_t r = 0; r < R; ++r) {
        double blk[MXO_BLOCK];
        for (int64_t kb = 0; kb < nb; ++kb) {
            for (int i = 0; i < MXO_BLOCK; ++i)
                blk[i] = bf16_value(x[r * ld + kb * MXO_BLOCK + i]);
            err |= mxo_quantize_block(blk, bits[kb], rounding, &scales[r * nb + kb],
                                      &codes[r * K + kb * MXO_BLOCK]) != 0;
        }
    }
    return err ? -1 : 0;
}

/* ------------------------------------------------------------------ */
/* Exactly rounded summation of doubles (Shewchuk 1997, "Adaptive      */
/* precision floating-point arithmetic"): keep a list of non-overlapping */
/* partials whose exact sum is the exact running total, then round the  */
/* top of the list once, with a half-way correction.                    */
/* ------------------------------------------------------------------ */
#define MXO_MAX_PARTIALS 2200
double mxo_fsum(const double *v, int64_t n)
{
    double p[MXO_MAX_PARTIALS];
    int np = 0;
    for (int64_t k = 0; k < n; ++k) {
        double x = v[k];
        if (!isfinite(x)) { /* NaN/inf: plain IEEE sum of the special terms */
            double special = 0.0;
            for (int64_t j = k; j < n; ++j) if (!isfinite(v[j])) special += v[j];
            return special;
        }
        int keep = 0;
        for (int j = 0; j < np; ++j) {
            double y = p[j];
            if (fabs(x) < fabs(y)) { double t = x; x = y; y = t; }
            double hi = x + y;            /* two-sum with |x| >= |y| */
            double lo = y - (hi - x);
            if (lo != 0.0) p[keep++] = lo;
            x = hi;
        }
        np = keep;
        if (np >= MXO_MAX_PARTIALS) return NAN; /* cannot happen for finite doubles */
        p[np++] = x;
    }
    if (np == 0) return 0.0;
    /* add partials from the largest down until the sum stops being exact */
    int j = np - 1;
    double hi = p[j], lo = 0.0;
    while (j > 0) {
        double x = hi, y = p[--j];
        hi = x + y;
        lo = y - (hi - x);
        if (lo != 0.0) break;
    }
    /* round-half-even fix: the rest of the partials decide a tie in lo */
    if (j > 0 && ((lo < 0.0 && p[j - 1] < 0.0) || (lo > 0.0 && p[j - 1] > 0.0))) {
        double y = lo * 2.0;
        double x = hi + y;
        if (y == x - hi) hi = x;
    }
    return hi;
}

/* ------------------------------------------------------------------ */
/* GEMM: y[m,n] = sum over blocks of 2^(Ea'+Ew') * (exact int dot).     */
/* Operands in natural order: a_codes[M,K], a_scales[M,nb],            */
/* w_codes[N,K], w_scales[N,nb]; one width map for both (Alg. 3 gives  */
/* one column allocation per linear layer, applied to W and A alike).  */
/* ------------------------------------------------------------------ */
static void gemm_one(int64_t K, const uint8_t *bits, const int8_t *ac, const uint8_t *as,
                     const int8_t *wc, const uint8_t *ws, double *terms, double *y, double *abssum)
{
    const int64_t nb = K / MXO_BLOCK;
    int nan = 0;
    for (int64_t kb = 0; kb < nb; ++kb) {
        if (as[kb] == 255 || ws[kb] == 255) nan = 1;
        int64_t d = 0;
        for (int i = 0; i < MXO_BLOCK; ++i)
            d += (int64_t)ac[kb * MXO_BLOCK + i] * (int64_t)wc[kb * MXO_BLOCK + i];
        int b = bits[kb];
        int ea = (int)as[kb] - 127 - (b - 2);
        int ew = (int)ws[kb] - 127 - (b - 2);
        terms[kb] = ldexp((double)d, ea + ew); /* exact: |d| < 2^20, exponent in fp64 range */
    }
    if (nan) { *y = NAN; *abssum = NAN; return; }
    *y = mxo_fsum(terms, nb);
    for (int64_t kb = 0; kb < nb; ++kb) terms[kb] = fabs(terms[kb]);
    *abssum = mxo_fsum(terms, nb);
}

int mxo_gemm(int64_t M, int64_t N, int64_t K, const uint8_t *bits,
             const int8_t *a_codes, const uint8_t *a_scales,
             const int8_t *w_codes, const uint8_t *w_scales,
             double *y, double *abssum)
{
    if (K % MXO_BLOCK != 0) return -1;
    const int64_t nb = K / MXO_BLOCK;
    int err = 0;
#pragma omp parallel reduction(| : err)
    {
        double *terms = (double *)malloc(sizeof(double) * (size_t)(nb > 0 ? nb : 1));
        if (!terms) err = 1;
#pragma omp for schedule(dynamic, 1)
        for (int64_t m = 0; m < M; ++m) {
            if (!terms) continue;
            for (int64_t n = 0; n < N; ++n)
                gemm_one(K, bits, a_codes + m * K, a_scales + m * nb, w_codes + n * K,
                         w_scales + n * nb, terms, &y[m * N + n], &abssum[m * N + n]);
        }
        free(terms);
    }
    return err ? -1 : 0;
}

/* Selected entries only (rows[i], cols[i]) -- for spot checks at full size. */
int mxo_gemm_entries(int64_t K, const uint8_t *bits,
                     const int8_t *a_codes, const uint8_t *a_scales, /* [*, K] / [*, nb] */
                     const int8_t *w_codes, const uint8_t *w_scales,
                     int64_t count, const int64_t *rows, const int64_t *cols,
                     double *y, double *abssum)
{
    if (K % MXO_BLOCK != 0) return -1;
    const int64_t nb = K / MXO_BLOCK;
    int err = 0;
#pragma omp parallel reduction(| : err)
    {
        double *terms = (double *)malloc(sizeof(double) * (size_t)(nb > 0 ? nb : 1));
        if (!terms) err = 1;
#pragma omp for schedule(static)
        for (int64_t i = 0; i < count; ++i) {
            if (!terms) continue;
            gemm_one(K, bits, a_codes + rows[i] * K, a_scales + rows[i] * nb,
                     w_codes + cols[i] * K, w_scales + cols[i] * nb, terms, &y[i], &abssum[i]);
        }
        free(terms);
    }
    return err ? -1 : 0;
}

/* ================================================================== */
/* Storage format (library layout), restated from its description.    */
/* ================================================================== */

/* Stable partition of block indices by width: slot s < n4 holds the s-th
 * 4-bit block, then the 6-bit blocks, then the 8-bit blocks, each group in
 * increasing block order.  slot_block[s] = original block index. */
int mxo_slots(const uint8_t *bits, int64_t nb, int32_t *slot_block, int64_t *counts /*[3]*/)
{
    int64_t s = 0;
    const int widths[3] = {4, 6, 8};
    for (int g = 0; g < 3; ++g) {
        counts[g] = 0;
        for (int64_t kb = 0; kb < nb; ++kb)
            if (bits[kb] == widths[g]) { slot_block[s++] = (int32_t)kb; counts[g]++; }
    }
    return s == nb ? 0 : -1; /* a width outside {4,6,8} */
}

static int64_t align256(int64_t v) { return (v + 255) / 256 * 256; }

/* Activation stream: per row, row_bytes = 16*n4 + 32*(n6+n8).
 * 4-bit slot s: bytes [16s, 16s+16); element i in byte i/2, low nibble for
 * even i, high nibble for odd i, two's complement.  6/8-bit slot s: bytes
 * [16*n4 + 32(s-n4), +32), one int8 per element.  Scales: [R, nb] per slot. */
int mxo_pack_act(int64_t R, int64_t K, const uint8_t *bits, const uint8_t *scales,
                 const int8_t *codes, uint8_t *pcodes, uint8_t *pscales)
{
    const int64_t nb = K / MXO_BLOCK;
    int32_t *sb = (int32_t *)malloc(sizeof(int32_t) * (size_t)(nb > 0 ? nb : 1));
    int64_t cnt[3];
    if (!sb || mxo_slots(bits, nb, sb, cnt) != 0) { free(sb); return -1; }
    const int64_t n4 = cnt[0], row_bytes = 16 * n4 + 32 * (cnt[1] + cnt[2]);
    for (int64_t r = 0; r < R; ++r) {
        uint8_t *row = pcodes + r * row_bytes;
        memset(row, 0, (size_t)row_bytes);
        for (int64_t s = 0; s < nb; ++s) {
            int64_t kb = sb[s];
            const int8_t *c = codes + r * K + kb * MXO_BLOCK;
            pscales[r * nb + s] = scales[r * nb + kb];
            if (s < n4) {
                for (int i = 0; i < MXO_BLOCK; ++i) {
                    uint8_t nib = (uint8_t)c[i] & 0x0F;
                    row[16 * s + i / 2] |= (uint8_t)((i % 2) ? (nib << 4) : nib);
                }
            } else {
                for (int i = 0; i < MXO_BLOCK; ++i)
                    row[16 * n4 + 32 * (s - n4) + i] = (uint8_t)c[i];
            }
        }
    }
    free(sb);
    return 0;
}

/* Weight stream.  Codes are stored sign-magnitude: a 4-bit code as
 * (sign << 3) | |m| and a 6/8-bit code as (sign << 7) | |m| (the symmetric
 * clamp R4 never produces -2^(b-1), so nothing is lost).  Rows are padded to
 * a multiple of 128 and cut into groups of 128 rows; group g occupies
 * GB = 2176*n4 + 4224*(n6+n8) contiguous bytes at g*GB:
 *   4-bit slot s at 2176*s: 128 rows x 16 code bytes (row r at 16r), then
 *     128 scale bytes (row r at 2048 + r).  In a row, byte 4i+j holds
 *     element 8i+j in its low nibble and element 8i+4+j in its high nibble;
 *   6/8-bit slot n4+j at 2176*n4 + 4224*j: 128 rows x 32 code bytes (row r
 *     at 32r, byte e = element e), then 128 scale bytes (row r at 4096 + r).
 *   Scale bytes of padding rows are zero.  Compact size = align256(G*GB).
 *   With planes: section P (offset compact size): [N, Kp] e4m3 planes and
 *   section SF (offset align256(P + N*Kp)): tcgen05 scale tiles, see below. */
static int64_t group_bytes(int64_t n4, int64_t n68) { return 2176 * n4 + 4224 * n68; }
static int64_t weight_compact(int64_t N, int64_t n4, int64_t n68)
{
    return align256((N + 127) / 128 * group_bytes(n4, n68));
}

/* Planes: for every row, Kp = 128*(ceil(n4/4) + ceil(n68/2)) bytes.
 * 4-bit slot s: bytes [32s, 32s+32) = e4m3(m/4).  Slots n4..4*ceil(n4/4)-1
 * are zero padding.  6/8-bit slot j at P68 = 128*ceil(n4/4), bytes
 * [P68+64j, +64), in one of two forms:
 *  - digit form: [P68+64j, +32) = high digit, [P68+64j+32, +32) = low digit
 *    (e4m3), with
 *      b=6: m = 8h + l (l in 0..7),  high = h/2, low = l/16;
 *      b=8: m = 16h + l (l in 0..15), high = h/4, low = l/64.
 *    so that high + low = m * 2^-(b-2) and the E8M0 scale S applies to both;
 *  - bf16 form: element i is the bf16 value m * 2^(S-127-(b-2)) (exact: |m|
 *    has at most 7 significant bits and bf16 keeps 8, with fp32's exponent
 *    range and subnormals), little-endian at P68+64j+2i; a block with S = 255
 *    (NaN/Inf) holds the bf16 NaN 0x7FC0.
 * Scale tiles SF: for row tile tau (128 rows) and stage st (one 128-byte
 * K' step: 4 slots of 4-bit or 2 slots of 6/8-bit), 512 bytes ordered
 * [i in 0..31][w in 0..3][q in 0..3]: the byte is S of row 128tau+32w+i,
 * slot 4st+q (4-bit stages) or 2(st-ceil(n4/4))+q for q<2 (6/8-bit stages);
 * zero for padding rows, padding slots and q>=2 in 6/8-bit stages. */
static int64_t kp_bytes(int64_t n4, int64_t n68) { return 128 * ((n4 + 3) / 4 + (n68 + 1) / 2); }
static int64_t n_stages(int64_t n4, int64_t n68) { return (n4 + 3) / 4 + (n68 + 1) / 2; }

int64_t mxo_weight_bytes(int64_t N, int64_t K, const uint8_t *bits, int with_planes)
{
    const int64_t nb = K / MXO_BLOCK;
    int32_t *sb = (int32_t *)malloc(sizeof(int32_t) * (size_t)(nb > 0 ? nb : 1));
    int64_t cnt[3];
    if (!sb || mxo_slots(bits, nb, sb, cnt) != 0) { free(sb); return -1; }
    free(sb);
    const int64_t compact = weight_compact(N, cnt[0], cnt[1] + cnt[2]);
    if (!with_planes) return compact;
    const int64_t kp = kp_bytes(cnt[0], cnt[1] + cnt[2]);
    const int64_t sf = align256(compact + N * kp);
    return align256(sf + (N + 127) / 128 * n_stages(cnt[0], cnt[1] + cnt[2]) * 512);
}

/* e4m3 (1 sign, 4 exponent bits with bias 7, 3 fraction bits) encoding of a
 * value that is exactly representable; returns -1 otherwise. */
int mxo_e4m3_encode(double v)
{
    if (v == 0.0) return signbit(v) ? 0x80 : 0x00;
    int sign = v < 0.0;
    double a = fabs(v);
    int e;
    double f = frexp(a, &e); /* a = f * 2^e, f in [0.5,1) -> a = (2f) * 2^(e-1) */
    int E = e - 1;           /* unbiased exponent of a normal number */
    int code;
    if (E >= -6) { /* normal: a = (1 + k/8) * 2^E, biased exponent E+7 in 1..15 */
        double k = (2.0 * f - 1.0) * 8.0;
        if (k != floor(k) || E + 7 > 15) return -1;
        code = ((E + 7) << 3) | (int)k;
        if (code == 0x7F) return -1; /* the NaN code */
    } else { /* subnormal: a = k/8 * 2^-6 */
        double k = ldexp(a, 9);
        if (k != floor(k) || k < 1.0 || k > 7.0) return -1;
        code = (int)k;
    }
    return (sign ? 0x80 : 0) | code;
}

/* bf16 (1 sign, 8 exponent bits with bias 127, 7 fraction bits) encoding of a
 * value that is exactly representable; returns -1 otherwise. */
int mxo_bf16_encode(double v)
{
    if (v == 0.0) return signbit(v) ? 0x8000 : 0x0000;
    int sign = v < 0.0;
    double a = fabs(v);
    int e;
    double f = frexp(a, &e);
    int E = e - 1;
    int code;
    if (E >= -126) { /* normal: a = (1 + k/128) * 2^E */
        double k = (2.0 * f - 1.0) * 128.0;
        if (k != floor(k) || E + 127 > 254) return -1;
        code = ((E + 127) << 7) | (int)k;
    } else { /* subnormal: a = k/128 * 2^-126 */
        double k = ldexp(a, 133);
        if (k != floor(k) || k < 1.0 || k > 127.0) return -1;
        code = (int)k;
    }
    return (sign ? 0x8000 : 0) | code;
}

static int plane_digits(int b, int m, double *hi, double *lo)
{
    if (b == 4) { *hi = m / 4.0; *lo = 0.0; return 1; }
    int s = (b == 6) ? 3 : 4;              /* m = 2^s * h + l with 0 <= l < 2^s */
    int h = (int)floor((double)m / (double)(1 << s));
    int l = m - h * (1 << s);
    *hi = ldexp((double)h * (double)(1 << s), -(b - 2));
    *lo = ldexp((double)l, -(b - 2));
    return 2;
}

/* Planes [R, Kp] and scale tiles for R rows quantized with map bits; 6/8-bit
 * blocks in digit form (bf16_68 = 0) or bf16 form (bf16_68 = 1). */
int mxo_planes(int64_t R, int64_t K, const uint8_t *bits, const uint8_t *scales,
               const int8_t *codes, uint8_t *planes, uint8_t *sf, int bf16_68)
{
    const int64_t nb = K / MXO_BLOCK;
    int32_t *sb = (int32_t *)malloc(sizeof(int32_t) * (size_t)(nb > 0 ? nb : 1));
    int64_t cnt[3];
    if (!sb || mxo_slots(bits, nb, sb, cnt) != 0) { free(sb); return -1; }
    const int64_t n4 = cnt[0], n68 = cnt[1] + cnt[2];
    const int64_t kp = kp_bytes(n4, n68), st4 = (n4 + 3) / 4, nst = n_stages(n4, n68);
    const int64_t p68 = 128 * st4;
    int err = 0;
    memset(planes, 0, (size_t)(R * kp));
    for (int64_t r = 0; r < R; ++r) {
        for (int64_t s = 0; s < nb; ++s) {
            const int64_t kb = sb[s];
            const int b = bits[kb];
            if (s >= n4 && bf16_68) {
                const int S = scales[r * nb + kb];
                for (int i = 0; i < MXO_BLOCK; ++i) {
                    const int m = codes[r * K + kb * MXO_BLOCK + i];
                    const int v = S == 255 ? 0x7FC0 : mxo_bf16_encode(ldexp((double)m, S - 127 - (b - 2)));
                    if (v < 0) err = 1;
                    planes[r * kp + p68 + 64 * (s - n4) + 2 * i] = (uint8_t)(v & 0xFF);
                    planes[r * kp + p68 + 64 * (s - n4) + 2 * i + 1] = (uint8_t)((v >> 8) & 0xFF);
                }
                continue;
            }
            for (int i = 0; i < MXO_BLOCK; ++i) {
                double hi, lo;
                plane_digits(b, codes[r * K + kb * MXO_BLOCK + i], &hi, &lo);
                int ch = mxo_e4m3_encode(hi), cl = mxo_e4m3_encode(lo);
                if (ch < 0 || cl < 0) err = 1;
                if (s < n4) {
                    planes[r * kp + 32 * s + i] = (uint8_t)ch;
                } else {
                    planes[r * kp + p68 + 64 * (s - n4) + i] = (uint8_t)ch;
                    planes[r * kp + p68 + 64 * (s - n4) + 32 + i] = (uint8_t)cl;
                }
            }
        }
    }
    const int64_t tiles = (R + 127) / 128;
    memset(sf, 0, (size_t)(tiles * nst * 512));
    for (int64_t tau = 0; tau < tiles; ++tau)
        for (int64_t st = 0; st < nst; ++st)
            for (int i = 0; i < 32; ++i)
                for (int w = 0; w < 4; ++w)
                    for (int q = 0; q < 4; ++q) {
                        int64_t r = 128 * tau + 32 * w + i, s;
                        if (r >= R) continue;
                        if (st < st4) {
                            s = 4 * st + q;
                            if (s >= n4) continue;
                        } else {
                            if (q >= 2) continue;
                            int64_t j = 2 * (st - st4) + q;
                            if (j >= n68) continue;
                            s = n4 + j;
                        }
                        sf[((tau * nst + st) * 32 + i) * 16 + w * 4 + q] = scales[r * nb + sb[s]];
                    }
    free(sb);
    return err ? -1 : 0;
}

int mxo_pack_weight(int64_t N, int64_t K, const uint8_t *bits, const uint8_t *scales,
                    const int8_t *codes, int with_planes, uint8_t *out)
{
    const int64_t nb = K / MXO_BLOCK;
    int32_t *sb = (int32_t *)malloc(sizeof(int32_t) * (size_t)(nb > 0 ? nb : 1));
    int64_t cnt[3];
    if (!sb || mxo_slots(bits, nb, sb, cnt) != 0) { free(sb); return -1; }
    const int64_t n4 = cnt[0], n68 = cnt[1] + cnt[2];
    const int64_t GB = group_bytes(n4, n68), compact = weight_compact(N, n4, n68);
    const int64_t total = mxo_weight_bytes(N, K, bits, with_planes);
    memset(out, 0, (size_t)total);
    for (int64_t r = 0; r < N; ++r) {
        const int64_t grp = r / 128, rr = r % 128;
        for (int64_t s = 0; s < nb; ++s) {
            const int64_t kb = sb[s];
            const int8_t *c = codes + r * K + kb * MXO_BLOCK;
            uint8_t *slot = out + grp * GB + (s < n4 ? 2176 * s : 2176 * n4 + 4224 * (s - n4));
            if (s < n4) {
                slot[2048 + rr] = scales[r * nb + kb];
                for (int e = 0; e < MXO_BLOCK; ++e) {
                    const int mag = c[e] < 0 ? -c[e] : c[e];
                    const uint8_t nib = (uint8_t)(((c[e] < 0) << 3) | mag);
                    const int i = e / 8, within = e % 8;       /* word i of the row */
                    uint8_t *byte = slot + 16 * rr + 4 * i + (within % 4);
                    *byte |= (uint8_t)(within < 4 ? nib : (nib << 4));
                }
            } else {
                slot[4096 + rr] = scales[r * nb + kb];
                for (int e = 0; e < MXO_BLOCK; ++e) {
                    const int mag = c[e] < 0 ? -c[e] : c[e];
                    slot[32 * rr + e] = (uint8_t)(((c[e] < 0) << 7) | mag);
                }
            }
        }
    }
    int err = 0;
    if (with_planes) {
        const int64_t kp = kp_bytes(n4, n68);
        const int64_t psf = align256(compact + N * kp);
        err = mxo_planes(N, K, bits, scales, codes, out + compact, out + psf, 1) != 0;  /* prefill operand */
    }
    free(sb);
    return err ? -1 : 0;
}
