/*
 * laq_oracle.c -- plain, slow CPU oracle for the WbG128 weight-only quantized linear layer.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path links, loads or calls this file; only
 * the tests, the package's smoke check and the CPU-baseline leg of the benchmark use it.  It
 * shares no code, header, table or constant generator with the CUDA library.
 *
 * What it computes, each function citing the passage it follows (LAQuant, arXiv 2605.08755):
 *
 *   laqo_quantize_rtn   Eq. (1): q = clip(round(w / s) + z, 0, 2^b - 1) with scale s and zero z
 *                       per group of g = 128 consecutive elements of a weight row (Sec. 2,
 *                       "Grouped quantization", W3G128).  The paper learns s and z by QAT; this
 *                       oracle initialises them by min-max round-to-nearest (RTN), the quantizer
 *                       the deployment kernel is agnostic to.  Readings where the paper is silent:
 *                         - the range is widened to include 0, so z lies in [0, 2^b - 1];
 *                         - s is the fp64 quotient (hi - lo) / (2^b - 1) rounded UP to fp16, then
 *                           floored at the smallest normal fp16 (2^-14);
 *                         - round() is round-half-to-even; Eq. (1) rounds w/s first, then adds z;
 *                         - w / s and -lo / s are fp64 quotients;
 *                         - a constant group c quantizes exactly: s = |c| (1 if c == 0),
 *                           z = 1 if c < 0 else 0.
 *   laqo_dequant        Eq. (1): w_hat = s * (q - z), exact in fp64.
 *   laqo_pack/unpack    The bit layout of packed codes (the library's own layout, App. H only
 *                       fixes that the INT3 kernel packs codes into 32-bit words).  Written here
 *                       from the layout's definition, bit by bit.
 *   laqo_gemm           Y = X * W_hat in fp64: the linear layer y = W x of the decode step
 *                       (Sec. 5.2 "Inference", Table 3), a naive sum over k in increasing order.
 *
 * Storage: W[K][N] fp16 (bit patterns), codes[K][N] u8, s[K/128][N] fp16 bits,
 * z[K/128][N] u8 -- the (num_groups, outfeatures) scale/zero tensors of App. H.
 * Every function returns 0 on success, a positive status otherwise.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define LAQO_GROUP 128

/* ---------- IEEE 754 binary16, written out from its definition ---------- */

/* Exact value of an fp16 bit pattern: (-1)^s * 2^(e-15) * (1 + m/1024), subnormal m * 2^-24. */
double laqo_half_to_double(uint16_t h)
{
    int sign = (h >> 15) & 1;
    int e = (h >> 10) & 0x1f;
    int m = h & 0x3ff;
    double v;
    if (e == 0)
        v = ldexp((double)m, -24);
    else if (e == 31)
        v = m ? NAN : INFINITY;
    else
        v = ldexp((double)(m + 1024), e - 25);
    return sign ? -v : v;
}

/* Smallest positive finite fp16 whose value is >= v (0 < v <= 65504).  The positive fp16 bit
 * patterns 0x0001..0x7bff are ordered like their values, so a bisection over them is exact. */
static uint16_t half_round_up_positive(double v)
{
    uint16_t lo = 0x0001, hi = 0x7bff;
    if (laqo_half_to_double(lo) >= v) return lo;
    while (hi - lo > 1) {
        uint16_t mid = (uint16_t)((lo + hi) / 2);
        if (laqo_half_to_double(mid) >= v) hi = mid; else lo = mid;
    }
    return hi;
}

/* ---------- Eq. (1): RTN group quantizer ---------- */

/* Group g of column n (rows 128g .. 128g + 127): its scale, zero and codes. */
static void quantize_group(const uint16_t *W, int64_t N, int64_t g, int64_t n, int qmax,
                           uint8_t *codes, uint16_t *s, uint8_t *z)
{
    double lo = INFINITY, hi = -INFINITY;
    for (int64_t k = g * LAQO_GROUP; k < (g + 1) * LAQO_GROUP; ++k) {
        double w = laqo_half_to_double(W[k * N + n]);
        if (w < lo) lo = w;
        if (w > hi) hi = w;
    }
    uint16_t sh;
    int zz;
    if (lo == hi) {                       /* constant group: exact by construction */
        if (lo != 0.0) {
            sh = (uint16_t)(W[g * LAQO_GROUP * N + n] & 0x7fff);   /* |c| */
            zz = lo < 0.0 ? 1 : 0;
        } else {
            sh = 0x3c00;                                           /* 1.0 */
            zz = 0;
        }
    } else {
        double lo0 = lo < 0.0 ? lo : 0.0;  /* zero-inclusive range */
        double hi0 = hi > 0.0 ? hi : 0.0;
        double sd = (hi0 - lo0) / (double)qmax;
        sh = half_round_up_positive(sd);
        if (sh < 0x0400) sh = 0x0400;       /* floor: smallest normal fp16 */
        zz = (int)rint(-lo0 / laqo_half_to_double(sh));
    }
    double sv = laqo_half_to_double(sh);
    s[g * N + n] = sh;
    z[g * N + n] = (uint8_t)zz;
    for (int64_t k = g * LAQO_GROUP; k < (g + 1) * LAQO_GROUP; ++k) {
        double w = laqo_half_to_double(W[k * N + n]);
        int q = (int)rint(w / sv) + zz;    /* round first, then add z (Eq. 1) */
        if (q < 0) q = 0;
        if (q > qmax) q = qmax;
        codes[k * N + n] = (uint8_t)q;
    }
}

int laqo_quantize_rtn(const uint16_t *W, int64_t K, int64_t N, int bits, int group,
                      uint8_t *codes, uint16_t *s, uint8_t *z)
{
    if (bits != 3 && bits != 4) return 2;
    if (group != LAQO_GROUP) return 3;
    if (K < 0 || N < 0 || K % LAQO_GROUP) return 4;
    const int qmax = (1 << bits) - 1;
    const int64_t G = K / LAQO_GROUP;
    for (int64_t g = 0; g < G; ++g)
        for (int64_t n = 0; n < N; ++n) quantize_group(W, N, g, n, qmax, codes, s, z);
    return 0;
}

/* laqo_quantize_rtn with the columns split over the host's threads (OpenMP, when the oracle is
 * built with it): every (group, column) is quantized by the same quantize_group, so the codes,
 * scales and zeros are laqo_quantize_rtn's bit for bit.  Used to check whole passes. */
int laqo_quantize_rtn_threads(const uint16_t *W, int64_t K, int64_t N, int bits, int group,
                              uint8_t *codes, uint16_t *s, uint8_t *z)
{
    if (bits != 3 && bits != 4) return 2;
    if (group != LAQO_GROUP) return 3;
    if (K < 0 || N < 0 || K % LAQO_GROUP) return 4;
    const int qmax = (1 << bits) - 1;
    const int64_t G = K / LAQO_GROUP;
    const int64_t cb = 64; /* columns per task */
    const int64_t ntask = (N + cb - 1) / cb;
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t t = 0; t < ntask; ++t) {
        const int64_t n1 = (t + 1) * cb < N ? (t + 1) * cb : N;
        for (int64_t g = 0; g < G; ++g)
            for (int64_t n = t * cb; n < n1; ++n) quantize_group(W, N, g, n, qmax, codes, s, z);
    }
    return 0;
}

/* Eq. (1): w_hat[k][n] = s[g][n] * (q[k][n] - z[g][n]), g = k / 128. */
int laqo_dequant(const uint8_t *codes, const uint16_t *s, const uint8_t *z, int64_t K, int64_t N,
                 double *What)
{
    if (K < 0 || N < 0 || K % LAQO_GROUP) return 4;
    for (int64_t k = 0; k < K; ++k)
        for (int64_t n = 0; n < N; ++n) {
            int64_t g = k / LAQO_GROUP;
            What[k * N + n] = laqo_half_to_double(s[g * N + n]) *
                              (double)((int)codes[k * N + n] - (int)z[g * N + n]);
        }
    return 0;
}

/* Y[m][n] = sum_k X[m][k] * w_hat[k][n], fp64, k ascending, w_hat formed on the fly. */
int laqo_gemm(const uint16_t *X, int64_t M, int64_t K, int64_t N, const uint8_t *codes,
              const uint16_t *s, const uint8_t *z, double *Y)
{
    if (M < 0 || K < 0 || N < 0 || K % LAQO_GROUP) return 4;
    for (int64_t m = 0; m < M; ++m) {
        double *y = Y + m * N;
        for (int64_t n = 0; n < N; ++n) y[n] = 0.0;
        for (int64_t k = 0; k < K; ++k) {
            double x = laqo_half_to_double(X[m * K + k]);
            int64_t g = k / LAQO_GROUP;
            for (int64_t n = 0; n < N; ++n) {
                double w = laqo_half_to_double(s[g * N + n]) *
                           (double)((int)codes[k * N + n] - (int)z[g * N + n]);
                y[n] += x * w;
            }
        }
    }
    return 0;
}

/* laqo_gemm with the output columns split over the host's threads (OpenMP, when the oracle is
 * built with it): every column is still its own k-ascending fp64 sum, so the result is
 * laqo_gemm's bit for bit.  Used to time the oracle on all host cores. */
int laqo_gemm_threads(const uint16_t *X, int64_t M, int64_t K, int64_t N, const uint8_t *codes,
                      const uint16_t *s, const uint8_t *z, double *Y)
{
    if (M < 0 || K < 0 || N < 0 || K % LAQO_GROUP) return 4;
    const int64_t cb = 64; /* columns per task */
    const int64_t ntask = (N + cb - 1) / cb;
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t t = 0; t < ntask; ++t) {
        const int64_t n0 = t * cb, n1 = n0 + cb < N ? n0 + cb : N;
        for (int64_t m = 0; m < M; ++m) {
            double *y = Y + m * N;
            for (int64_t n = n0; n < n1; ++n) y[n] = 0.0;
            for (int64_t k = 0; k < K; ++k) {
                double x = laqo_half_to_double(X[m * K + k]);
                int64_t g = k / LAQO_GROUP;
                for (int64_t n = n0; n < n1; ++n) {
                    double w = laqo_half_to_double(s[g * N + n]) *
                               (double)((int)codes[k * N + n] - (int)z[g * N + n]);
                    y[n] += x * w;
                }
            }
        }
    }
    return 0;
}

/* Threads the oracle runs laqo_gemm_threads with (1 without OpenMP). */
int laqo_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* Same sum restricted to the listed output columns (for sampled checks of large layers). */
int laqo_gemm_columns(const uint16_t *X, int64_t M, int64_t K, int64_t N, const uint8_t *codes,
                      const uint16_t *s, const uint8_t *z, const int64_t *cols, int64_t ncols,
                      double *Y)
{
    if (M < 0 || K < 0 || N < 0 || K % LAQO_GROUP) return 4;
    for (int64_t m = 0; m < M; ++m)
        for (int64_t i = 0; i < ncols; ++i) {
            int64_t n = cols[i];
            double acc = 0.0;
            for (int64_t k = 0; k < K; ++k) {
                int64_t g = k / LAQO_GROUP;
                double w = laqo_half_to_double(s[g * N + n]) *
                           (double)((int)codes[k * N + n] - (int)z[g * N + n]);
                acc += laqo_half_to_double(X[m * K + k]) * w;
            }
            Y[m * ncols + i] = acc;
        }
    return 0;
}

/* ---------- packed layout ----------
 *
 * Codes are packed in records of 16 output columns x 128 rows of K (one group of one 16-column
 * tile).  Record (t, g) covers columns n = 16t .. 16t+15 and rows k = 128g .. 128g+127; records
 * are stored tile-major: record index t * (K/128) + g.  A record holds 32 lanes; lane l has
 * c = l % 4 and r = l / 4 and owns the 64 codes at columns r and r + 8 of the tile and rows
 *     k = 32c + 4j + 2h + e    (j = 0..7, h = 0..1, e = 0..1) of the group.
 * A "pair" (j, h, row) is the two codes e = 0 (bits 0..15 of a word) and e = 1 (bits 16..31,
 * same position + 16).  Within each 16-bit half:
 *
 * b = 4: 8 words per lane, word j holds step j.  Half-bits 0-3: (j, h=0, row r), 4-7: (j, h=1,
 *        row r), 8-11: (j, h=0, row r+8), 12-15: (j, h=1, row r+8).  Word w of lane l sits at
 *        word offset (w / 4) * 128 + 4 l + (w % 4) of the 256-word record.
 * b = 3: 6 words per lane.  Let pair index i = 2j + h (0..15).  In word w, half-bits
 *        0: bit (w % 3) of pair i = 15, row r for w < 3 else r + 8;
 *        1-3: pair i = w, row r;      4-6: pair i = 6 + w, row r;
 *        7-9: pair i = 12 + w/2, row r if w is even else r + 8;
 *        10-12: pair i = w, row r+8;  13-15: pair i = 6 + w, row r+8.
 *        Word w of lane l sits at word offset 4 l + w (w < 4) or 128 + 2 l + (w - 4) (w >= 4)
 *        of the 192-word record.
 * Bit 0 of a field is the code's least significant bit.  Words are little-endian uint32.
 */

/* For bit `b` (0..31) of word `w` of lane `l`: the row-in-group kk, the column-in-tile nn and the
 * bit of the code it carries. */
static void layout_bit(int bits, int l, int w, int b, int *kk, int *nn, int *cb)
{
    int c = l % 4, r = l / 4;
    int e = b / 16, hb = b % 16;
    int j, h, row;
    if (bits == 4) {
        int f = hb / 4;
        *cb = hb % 4;
        j = w;
        h = f % 2;
        row = f / 2;
    } else {
        int i;
        if (hb == 0)      { i = 15;         row = w >= 3;  *cb = w % 3; }
        else if (hb < 4)  { i = w;          row = 0;       *cb = hb - 1; }
        else if (hb < 7)  { i = 6 + w;      row = 0;       *cb = hb - 4; }
        else if (hb < 10) { i = 12 + w / 2; row = w % 2;   *cb = hb - 7; }
        else if (hb < 13) { i = w;          row = 1;       *cb = hb - 10; }
        else              { i = 6 + w;      row = 1;       *cb = hb - 13; }
        j = i / 2;
        h = i % 2;
    }
    *kk = 32 * c + 4 * j + 2 * h + e;
    *nn = r + 8 * row;
}

static int words_per_lane(int bits) { return bits == 4 ? 8 : 6; }

static int64_t word_offset(int bits, int l, int w)
{
    if (bits == 4) return (w / 4) * 128 + 4 * l + (w % 4);
    return w < 4 ? 4 * l + w : 128 + 2 * l + (w - 4);
}

int64_t laqo_packed_words(int64_t K, int64_t N, int bits) { return K * N * bits / 32; }

int laqo_pack(const uint8_t *codes, int64_t K, int64_t N, int bits, uint32_t *packed)
{
    if (bits != 3 && bits != 4) return 2;
    if (K < 0 || N < 0 || K % LAQO_GROUP || N % 16) return 4;
    const int64_t G = K / LAQO_GROUP, T = N / 16;
    const int wpl = words_per_lane(bits);
    const int64_t rec_words = 32 * wpl;
    memset(packed, 0, (size_t)(T * G * rec_words) * sizeof(uint32_t));
    for (int64_t t = 0; t < T; ++t)
        for (int64_t g = 0; g < G; ++g) {
            uint32_t *rec = packed + (t * G + g) * rec_words;
            for (int l = 0; l < 32; ++l)
                for (int w = 0; w < wpl; ++w) {
                    uint32_t word = 0;
                    for (int b = 0; b < 32; ++b) {
                        int kk, nn, cb;
                        layout_bit(bits, l, w, b, &kk, &nn, &cb);
                        int64_t k = g * LAQO_GROUP + kk, n = t * 16 + nn;
                        uint32_t bit = (codes[k * N + n] >> cb) & 1u;
                        word |= bit << b;
                    }
                    rec[word_offset(bits, l, w)] = word;
                }
        }
    return 0;
}

int laqo_unpack(const uint32_t *packed, int64_t K, int64_t N, int bits, uint8_t *codes)
{
    if (bits != 3 && bits != 4) return 2;
    if (K < 0 || N < 0 || K % LAQO_GROUP || N % 16) return 4;
    const int64_t G = K / LAQO_GROUP, T = N / 16;
    const int wpl = words_per_lane(bits);
    const int64_t rec_words = 32 * wpl;
    memset(codes, 0, (size_t)(K * N));
    for (int64_t t = 0; t < T; ++t)
        for (int64_t g = 0; g < G; ++g) {
            const uint32_t *rec = packed + (t * G + g) * rec_words;
            for (int l = 0; l < 32; ++l)
                for (int w = 0; w < wpl; ++w) {
                    uint32_t word = rec[word_offset(bits, l, w)];
                    for (int b = 0; b < 32; ++b) {
                        int kk, nn, cb;
                        layout_bit(bits, l, w, b, &kk, &nn, &cb);
                        int64_t k = g * LAQO_GROUP + kk, n = t * 16 + nn;
                        codes[k * N + n] |= (uint8_t)(((word >> b) & 1u) << cb);
                    }
                }
        }
    return 0;
}

/* The (row-in-group, column-in-tile, code bit) carried by bit b of word w of lane l; used by the
 * tests to check that the layout is a bijection. */
int laqo_layout_bit(int bits, int l, int w, int b, int *kk, int *nn, int *cb)
{
    if (bits != 3 && bits != 4) return 2;
    if (l < 0 || l >= 32 || w < 0 || w >= words_per_lane(bits) || b < 0 || b >= 32) return 4;
    layout_bit(bits, l, w, b, kk, nn, cb);
    return 0;
}

int64_t laqo_word_offset(int bits, int l, int w) { return word_offset(bits, l, w); }
