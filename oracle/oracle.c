/*
 * Oracle for the quantized HWC convolution path of PULP-NN (arXiv 1908.11263).
 *
 * TEST INFRASTRUCTURE ONLY.  This file is a plain, slow, obviously correct CPU
 * statement of what the GPU library computes.  Only the test-suite, the smoke
 * check and the CPU-baseline leg of bench.py may load it.  It shares no code,
 * header, table or constant with the CUDA library, and the library never loads it.
 *
 * Every value is an integer; every intermediate is held in int64, so the only
 * way this code can differ from the mathematics is a logic error, which the
 * pins in tests/test_oracle_pins.py are written to catch.
 *
 * Readings of the paper that this file fixes:
 *  - Activations are unsigned Q-bit integers, weights signed two's-complement
 *    Q-bit integers (the paper's INT-Q representation, Sec. III-A, Eq. 1).
 *  - The accumulator is the integer sum of products Phi(W,X) (Sec. III-A, Eq. 2),
 *    held here in int64 and required to fit int32 (the paper's INT-32
 *    accumulator); a call whose accumulator would leave int32 is rejected.
 *  - Compression back to Q bits ("scaling and clamp", Sec. III-A) is
 *    y = clip( floor( ((acc + bias) * kappa + lambda) / 2^shift ), 0, 2^Q - 1 ):
 *    bias is added to the accumulator before the per-channel scale kappa (the
 *    batch-norm form in the footnote to Eq. 3), the shift rounds toward minus
 *    infinity, and the clip to [0, 2^Q-1] doubles as the ReLU of Sec. IV-A.
 *  - Zero padding (activation value 0) outside the input image.
 *  - Filters are [M][KH][KW][C] with C innermost, i.e. each filter bank W(m) is
 *    stored in im2col order (Sec. III-B, Eq. 6).
 *  - Sub-byte storage (Sec. IV-A, "Sub-byte Extensions"): element e of a packed
 *    Q-bit stream sits in byte e / (8/Q) at bits [(e mod (8/Q)) * Q, +Q); the
 *    first element takes the least significant bits.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_OK 0
#define ORACLE_EINVAL 1
#define ORACLE_EOVERFLOW 2

static int valid_bits(int bits) { return bits == 8 || bits == 4 || bits == 2; }

/* ---- sub-byte storage (Sec. IV-A: two INT-4 values per byte, INT-2 likewise four) ---- */

/* Reads element e of a packed stream as an unsigned Q-bit field. */
static uint32_t field_at(const uint8_t *src, int64_t e, int bits)
{
    int per_byte = 8 / bits;
    uint8_t byte = src[e / per_byte];
    int pos = (int)(e % per_byte) * bits;
    return (uint32_t)(byte >> pos) & ((1u << bits) - 1u);
}

int oracle_unpack(const uint8_t *src, int64_t count, int bits, int is_signed, int32_t *dst)
{
    if (!valid_bits(bits) || count < 0) return ORACLE_EINVAL;
    for (int64_t e = 0; e < count; ++e) {
        int32_t v = (int32_t)field_at(src, e, bits);
        if (is_signed && v >= (1 << (bits - 1))) v -= (1 << bits); /* two's complement */
        dst[e] = v;
    }
    return ORACLE_OK;
}

/* Stores the low Q bits of each value; count must fill whole bytes. */
int oracle_pack(const int32_t *src, int64_t count, int bits, uint8_t *dst)
{
    if (!valid_bits(bits) || count < 0 || count % (8 / bits) != 0) return ORACLE_EINVAL;
    int per_byte = 8 / bits;
    int64_t nbytes = count / per_byte;
    memset(dst, 0, (size_t)nbytes);
    for (int64_t e = 0; e < count; ++e) {
        uint32_t field = (uint32_t)src[e] & ((1u << bits) - 1u);
        dst[e / per_byte] |= (uint8_t)(field << ((e % per_byte) * bits));
    }
    return ORACLE_OK;
}

/* ---- convolution, Sec. III-B Eq. 6: O(m,x,y) = dot(W(m), im2col(x,y)) written as the direct sum ---- */

static int conv_shape_ok(int n, int h, int w, int c, int m, int kh, int kw, int sh, int sw, int ph, int pw,
                         int *oh, int *ow)
{
    if (n < 0 || h <= 0 || w <= 0 || c <= 0 || m <= 0 || kh <= 0 || kw <= 0) return 0;
    if (sh <= 0 || sw <= 0 || ph < 0 || pw < 0) return 0;
    *oh = (h + 2 * ph - kh) / sh + 1;
    *ow = (w + 2 * pw - kw) / sw + 1;
    return (h + 2 * ph - kh) >= 0 && (w + 2 * pw - kw) >= 0;
}

/* One output accumulator: the sum over the receptive field, zero outside the image. */
static int64_t conv_sum(int h, int w, int c, int kh, int kw, int sh, int sw, int ph, int pw,
                        const int32_t *x_img, const int32_t *w_bank, int oy, int ox)
{
    int64_t acc = 0;
    for (int i = 0; i < kh; ++i) {
        int iy = oy * sh - ph + i;
        for (int j = 0; j < kw; ++j) {
            int ix = ox * sw - pw + j;
            for (int ch = 0; ch < c; ++ch) {
                int64_t xv = 0;
                if (iy >= 0 && iy < h && ix >= 0 && ix < w)
                    xv = x_img[((int64_t)iy * w + ix) * c + ch];
                int64_t wv = w_bank[((int64_t)i * kw + j) * c + ch];
                acc += xv * wv;
            }
        }
    }
    return acc;
}

/* Accumulators of every output, before compression (int64, no range check). */
int oracle_conv_acc(int n, int h, int w, int c, int m, int kh, int kw, int sh, int sw, int ph, int pw,
                    const int32_t *x, const int32_t *wt, int64_t *acc)
{
    int oh, ow;
    if (!conv_shape_ok(n, h, w, c, m, kh, kw, sh, sw, ph, pw, &oh, &ow)) return ORACLE_EINVAL;
    for (int b = 0; b < n; ++b) {
        const int32_t *x_img = x + (int64_t)b * h * w * c;
        for (int oy = 0; oy < oh; ++oy)
            for (int ox = 0; ox < ow; ++ox)
                for (int o = 0; o < m; ++o)
                    acc[(((int64_t)b * oh + oy) * ow + ox) * m + o] =
                        conv_sum(h, w, c, kh, kw, sh, sw, ph, pw, x_img, wt + (int64_t)o * kh * kw * c, oy, ox);
    }
    return ORACLE_OK;
}

/* floor(t / 2^s) for 0 <= s <= 62, written as a division so it does not rely on
 * the compiler's treatment of right shifts of negative numbers. */
int64_t oracle_floor_shift(int64_t t, int s)
{
    int64_t d = (int64_t)1 << s;
    int64_t q = t / d;             /* C division truncates toward zero */
    if ((t % d != 0) && (t < 0)) q -= 1;
    return q;
}

/* Compression of one accumulator to a Q-bit unsigned output (reading of Sec. III-A). */
int32_t oracle_requant(int64_t acc, int32_t bias, int32_t kappa, int32_t lambda, int shift, int bits)
{
    int64_t t = (acc + (int64_t)bias) * (int64_t)kappa + (int64_t)lambda;
    int64_t y = oracle_floor_shift(t, shift);
    int64_t top = ((int64_t)1 << bits) - 1;
    if (y < 0) y = 0;
    if (y > top) y = top;
    return (int32_t)y;
}

static int fits_i32(int64_t v) { return v >= INT32_MIN && v <= INT32_MAX; }

/* Full layer on packed buffers: unpack, direct convolution, compression, pack.
 * shifts may be NULL (then every channel uses `shift`); bias may be NULL (zero).
 * nthreads > 1 splits the batch across OpenMP threads; the arithmetic per output
 * is unchanged. */
int oracle_conv_hwc(int n, int h, int w, int c, int m, int kh, int kw, int sh, int sw, int ph, int pw, int bits,
                    const uint8_t *x_packed, const uint8_t *w_packed, const int32_t *bias, const int16_t *kappa,
                    const int32_t *lambda, const uint8_t *shifts, int shift, uint8_t *y_packed, int nthreads)
{
    int oh, ow;
    if (!valid_bits(bits)) return ORACLE_EINVAL;
    if (!conv_shape_ok(n, h, w, c, m, kh, kw, sh, sw, ph, pw, &oh, &ow)) return ORACLE_EINVAL;
    int64_t nx = (int64_t)n * h * w * c, nw = (int64_t)m * kh * kw * c, ny = (int64_t)n * oh * ow * m;
    if (nx % (8 / bits) || nw % (8 / bits) || ny % (8 / bits)) return ORACLE_EINVAL;
    int32_t *x = (int32_t *)malloc(sizeof(int32_t) * (size_t)(nx ? nx : 1));
    int32_t *wt = (int32_t *)malloc(sizeof(int32_t) * (size_t)nw);
    int32_t *y = (int32_t *)malloc(sizeof(int32_t) * (size_t)(ny ? ny : 1));
    if (!x || !wt || !y) { free(x); free(wt); free(y); return ORACLE_EINVAL; }
    oracle_unpack(x_packed, nx, bits, 0, x);
    oracle_unpack(w_packed, nw, bits, 1, wt);
    int status = ORACLE_OK;
    if (nthreads < 1) nthreads = 1;
#pragma omp parallel for num_threads(nthreads) schedule(dynamic, 1)
    for (int b = 0; b < n; ++b) {
        const int32_t *x_img = x + (int64_t)b * h * w * c;
        for (int oy = 0; oy < oh; ++oy)
            for (int ox = 0; ox < ow; ++ox)
                for (int o = 0; o < m; ++o) {
                    int64_t acc = conv_sum(h, w, c, kh, kw, sh, sw, ph, pw, x_img, wt + (int64_t)o * kh * kw * c,
                                           oy, ox);
                    int32_t bo = bias ? bias[o] : 0;
                    if (!fits_i32(acc) || !fits_i32(acc + bo)) status = ORACLE_EOVERFLOW;
                    int s = shifts ? shifts[o] : shift;
                    y[(((int64_t)b * oh + oy) * ow + ox) * m + o] = oracle_requant(acc, bo, kappa[o], lambda[o], s, bits);
                }
    }
    if (status == ORACLE_OK) oracle_pack(y, ny, bits, y_packed);
    free(x); free(wt); free(y);
    return status;
}

/* Staircase compression (Sec. III-A, Eq. 4): the output is the number of the
 * channel's 2^Q - 1 thresholds that do not exceed the accumulator.  For sorted
 * thresholds this is the index p of the interval [tau_p, tau_p+1) holding the
 * accumulator, counted from 0 for the lowest interval (unsigned outputs; the
 * thresholds absorb bias and batch normalisation, per the footnote to Eq. 3). */
int32_t oracle_staircase(int64_t acc, const int32_t *tau, int bits)
{
    int32_t y = 0;
    for (int k = 0; k < (1 << bits) - 1; ++k)
        if ((int64_t)tau[k] <= acc) ++y;
    return y;
}

/* Full layer with staircase compression: thresholds are [m][2^Q - 1] (int32). */
int oracle_conv_hwc_thresholds(int n, int h, int w, int c, int m, int kh, int kw, int sh, int sw, int ph, int pw,
                               int bits, const uint8_t *x_packed, const uint8_t *w_packed, const int32_t *thresholds,
                               uint8_t *y_packed, int nthreads)
{
    int oh, ow;
    if (!valid_bits(bits)) return ORACLE_EINVAL;
    if (!conv_shape_ok(n, h, w, c, m, kh, kw, sh, sw, ph, pw, &oh, &ow)) return ORACLE_EINVAL;
    int64_t nx = (int64_t)n * h * w * c, nw = (int64_t)m * kh * kw * c, ny = (int64_t)n * oh * ow * m;
    if (nx % (8 / bits) || nw % (8 / bits) || ny % (8 / bits)) return ORACLE_EINVAL;
    const int nt = (1 << bits) - 1;
    int32_t *x = (int32_t *)malloc(sizeof(int32_t) * (size_t)(nx ? nx : 1));
    int32_t *wt = (int32_t *)malloc(sizeof(int32_t) * (size_t)nw);
    int32_t *y = (int32_t *)malloc(sizeof(int32_t) * (size_t)(ny ? ny : 1));
    if (!x || !wt || !y) { free(x); free(wt); free(y); return ORACLE_EINVAL; }
    oracle_unpack(x_packed, nx, bits, 0, x);
    oracle_unpack(w_packed, nw, bits, 1, wt);
    int status = ORACLE_OK;
    if (nthreads < 1) nthreads = 1;
#pragma omp parallel for num_threads(nthreads) schedule(dynamic, 1)
    for (int b = 0; b < n; ++b) {
        const int32_t *x_img = x + (int64_t)b * h * w * c;
        for (int oy = 0; oy < oh; ++oy)
            for (int ox = 0; ox < ow; ++ox)
                for (int o = 0; o < m; ++o) {
                    int64_t acc = conv_sum(h, w, c, kh, kw, sh, sw, ph, pw, x_img, wt + (int64_t)o * kh * kw * c,
                                           oy, ox);
                    if (!fits_i32(acc)) status = ORACLE_EOVERFLOW;
                    y[(((int64_t)b * oh + oy) * ow + ox) * m + o] = oracle_staircase(acc, thresholds + (int64_t)o * nt, bits);
                }
    }
    if (status == ORACLE_OK) oracle_pack(y, ny, bits, y_packed);
    free(x); free(wt); free(y);
    return status;
}

/* INT-1 (Sec. III-A, Eq. 5; binary kernel of Sec. IV-A).  Values +1 / -1 are
 * bits 1 / 0, eight per byte, element e at bit e mod 8 of byte e / 8.  The
 * accumulator counts the ones of W xnor X over the window positions that lie
 * inside the image (a padded position contributes neither a match nor a
 * mismatch: zero padding of the +-1 values); the output bit is 1 when the
 * channel's threshold does not exceed that count. */
static int bit_at(const uint8_t *src, int64_t e) { return (src[e >> 3] >> (e & 7)) & 1; }

int oracle_conv_binary(int n, int h, int w, int c, int m, int kh, int kw, int sh, int sw, int ph, int pw,
                       const uint8_t *x_bits, const uint8_t *w_bits, const int32_t *thresholds, uint8_t *y_bits,
                       int32_t *acc_out)
{
    int oh, ow;
    if (!conv_shape_ok(n, h, w, c, m, kh, kw, sh, sw, ph, pw, &oh, &ow)) return ORACLE_EINVAL;
    if (c % 8 || m % 8) return ORACLE_EINVAL;
    int64_t ny = (int64_t)n * oh * ow * m;
    memset(y_bits, 0, (size_t)(ny / 8));
    for (int b = 0; b < n; ++b)
        for (int oy = 0; oy < oh; ++oy)
            for (int ox = 0; ox < ow; ++ox)
                for (int o = 0; o < m; ++o) {
                    int32_t ones = 0;
                    for (int i = 0; i < kh; ++i)
                        for (int j = 0; j < kw; ++j) {
                            int iy = oy * sh - ph + i, ix = ox * sw - pw + j;
                            if (iy < 0 || iy >= h || ix < 0 || ix >= w) continue;
                            for (int ch = 0; ch < c; ++ch) {
                                int xb = bit_at(x_bits, (((int64_t)b * h + iy) * w + ix) * c + ch);
                                int wb = bit_at(w_bits, (((int64_t)o * kh + i) * kw + j) * c + ch);
                                ones += (xb == wb);  /* xnor */
                            }
                        }
                    int64_t e = (((int64_t)b * oh + oy) * ow + ox) * m + o;
                    if (acc_out) acc_out[e] = ones;
                    if (thresholds[o] <= ones) y_bits[e >> 3] |= (uint8_t)(1u << (e & 7));
                }
    return ORACLE_OK;
}

/* Same layer, evaluated only at listed output pixels (triples n, oy, ox); writes
 * the unpacked outputs [npix][m].  Used to check very large layers one output
 * pixel at a time. */
int oracle_conv_hwc_pixels(int n, int h, int w, int c, int m, int kh, int kw, int sh, int sw, int ph, int pw,
                           int bits, const uint8_t *x_packed, const uint8_t *w_packed, const int32_t *bias,
                           const int16_t *kappa, const int32_t *lambda, const uint8_t *shifts, int shift,
                           const int32_t *pix, int npix, int32_t *y_out)
{
    int oh, ow;
    if (!valid_bits(bits)) return ORACLE_EINVAL;
    if (!conv_shape_ok(n, h, w, c, m, kh, kw, sh, sw, ph, pw, &oh, &ow)) return ORACLE_EINVAL;
    int64_t img = (int64_t)h * w * c, nw = (int64_t)m * kh * kw * c;
    int32_t *x = (int32_t *)malloc(sizeof(int32_t) * (size_t)img);
    int32_t *wt = (int32_t *)malloc(sizeof(int32_t) * (size_t)nw);
    if (!x || !wt) { free(x); free(wt); return ORACLE_EINVAL; }
    oracle_unpack(w_packed, nw, bits, 1, wt);
    int status = ORACLE_OK;
    for (int p = 0; p < npix; ++p) {
        int b = pix[3 * p], oy = pix[3 * p + 1], ox = pix[3 * p + 2];
        if (b < 0 || b >= n || oy < 0 || oy >= oh || ox < 0 || ox >= ow) { status = ORACLE_EINVAL; break; }
        /* unpack image b element by element (activations are unsigned) */
        for (int64_t e = 0; e < img; ++e) x[e] = (int32_t)field_at(x_packed, (int64_t)b * img + e, bits);
        for (int o = 0; o < m; ++o) {
            int64_t acc = conv_sum(h, w, c, kh, kw, sh, sw, ph, pw, x, wt + (int64_t)o * kh * kw * c, oy, ox);
            int32_t bo = bias ? bias[o] : 0;
            if (!fits_i32(acc) || !fits_i32(acc + bo)) status = ORACLE_EOVERFLOW;
            int s = shifts ? shifts[o] : shift;
            y_out[(int64_t)p * m + o] = oracle_requant(acc, bo, kappa[o], lambda[o], s, bits);
        }
    }
    free(x); free(wt);
    return status;
}

/* ---- max-pooling (Sec. IV-A): max over each k x k window, stride s, no padding, floor size ---- */
int oracle_maxpool(int n, int h, int w, int c, int k, int s, int bits, const uint8_t *x_packed, uint8_t *y_packed)
{
    if (!valid_bits(bits) || n < 0 || h <= 0 || w <= 0 || c <= 0 || k <= 0 || s <= 0 || k > h || k > w)
        return ORACLE_EINVAL;
    int oh = (h - k) / s + 1, ow = (w - k) / s + 1;
    int64_t nx = (int64_t)n * h * w * c, ny = (int64_t)n * oh * ow * c;
    if (nx % (8 / bits) || ny % (8 / bits)) return ORACLE_EINVAL;
    int32_t *x = (int32_t *)malloc(sizeof(int32_t) * (size_t)(nx ? nx : 1));
    int32_t *y = (int32_t *)malloc(sizeof(int32_t) * (size_t)(ny ? ny : 1));
    if (!x || !y) { free(x); free(y); return ORACLE_EINVAL; }
    oracle_unpack(x_packed, nx, bits, 0, x);
    for (int b = 0; b < n; ++b)
        for (int oy = 0; oy < oh; ++oy)
            for (int ox = 0; ox < ow; ++ox)
                for (int ch = 0; ch < c; ++ch) {
                    int32_t best = 0; /* activations are unsigned, so 0 is below every value */
                    for (int i = 0; i < k; ++i)
                        for (int j = 0; j < k; ++j) {
                            int32_t v = x[(((int64_t)b * h + oy * s + i) * w + ox * s + j) * c + ch];
                            if (v > best) best = v;
                        }
                    y[(((int64_t)b * oh + oy) * ow + ox) * c + ch] = best;
                }
    oracle_pack(y, ny, bits, y_packed);
    free(x); free(y);
    return ORACLE_OK;
}

/* ---- fully connected (Sec. IV-A): y[b][o] = sum_k x[b][k] * W[o][k] + bias[o], int32 output ---- */
int oracle_linear(int n, int k, int m, const uint8_t *x, const int8_t *wt, const int32_t *bias, int32_t *y)
{
    if (n < 0 || k <= 0 || m <= 0) return ORACLE_EINVAL;
    int status = ORACLE_OK;
    for (int b = 0; b < n; ++b)
        for (int o = 0; o < m; ++o) {
            int64_t acc = bias ? bias[o] : 0;
            for (int i = 0; i < k; ++i) acc += (int64_t)x[(int64_t)b * k + i] * (int64_t)wt[(int64_t)o * k + i];
            if (!fits_i32(acc)) status = ORACLE_EOVERFLOW;
            y[(int64_t)b * m + o] = (int32_t)acc;
        }
    return status;
}
