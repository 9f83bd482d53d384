/*
 * tbn_oracle.c -- plain double-precision CPU reference for Two-Bit Networks
 * (arXiv:1701.00485).  TEST INFRASTRUCTURE ONLY: loaded by the test suite,
 * the smoke check and the benchmark's CPU-baseline leg, never by the product.
 *
 * Written from the paper's definitions, one function per step, with no
 * blocking, fusion or reordering: a reader should be able to hold each loop
 * next to the equation it cites.  Shares no code with the CUDA library.
 */
#include "tbn_oracle.h"

#include <math.h>
#include <stddef.h>

#ifdef _OPENMP
#include <omp.h>
#endif

/* ---- Eq. 3 (Section 2): deterministic discretization -------------------- */
int orc_discretize_one(double w)
{
    if (w < -1.0)
        return -2;
    if (-1.0 <= w && w <= 0.0)
        return -1;
    if (0.0 < w && w <= 1.0)
        return 1;
    return 2; /* w > 1 */
}

void orc_discretize(const float *W, int64_t n, int8_t *wt)
{
    for (int64_t i = 0; i < n; ++i)
        wt[i] = (int8_t)orc_discretize_one((double)W[i]);
}

/* ---- Eq. 5 (Section 2): optimal scaling factor ------------------------- */
double orc_alpha(const float *W, int64_t n)
{
    /* B1 = {i : |W_i| <= 1},  B2 = {i : |W_i| > 1}  (sets defined with Eq. 4) */
    double sum_b1 = 0.0, sum_b2 = 0.0;
    int64_t size_b1 = 0, size_b2 = 0;
    for (int64_t i = 0; i < n; ++i) {
        double a = fabs((double)W[i]);
        if (a <= 1.0) {
            sum_b1 += a;
            size_b1 += 1;
        } else {
            sum_b2 += a;
            size_b2 += 1;
        }
    }
    double numerator = sum_b1 + 2.0 * sum_b2;
    double denominator = (double)size_b1 + 4.0 * (double)size_b2;
    return numerator / denominator;
}

/* ---- Algorithm 1, quantization loop over the filters of one layer ------- */
void orc_quantize(const float *W, int64_t K, int64_t n, int8_t *wt, double *alpha)
{
    for (int64_t k = 0; k < K; ++k) {
        orc_discretize(W + k * n, n, wt + k * n); /* W~ by Eq. 3 */
        alpha[k] = orc_alpha(W + k * n, n);       /* alpha* by Eq. 5 */
    }
}

/* ---- two-bit storage ---------------------------------------------------- */
/* Layout (build-defined; the paper fixes only that a weight takes two bits):
 * code i of a filter lives in word i / 16 of that filter.  Inside the word,
 * with l = i % 16, pair p = l / 2 and half h = l % 2, the code's magnitude
 * bit m sits at bit 16 h + p and its sign bit s at bit 16 h + 8 + p.  So byte
 * 0 holds the magnitude bits of the even codes, byte 1 their sign bits,
 * byte 2 the magnitude bits of the odd codes and byte 3 their sign bits. */
int64_t orc_words_per_filter(int64_t n)
{
    return (n + 15) / 16;
}

static int magnitude_bit(int64_t i)
{
    int64_t l = i % 16;
    return (int)(16 * (l % 2) + l / 2);
}

static int sign_bit(int64_t i)
{
    return magnitude_bit(i) + 8;
}

/* field value for a code: m + 2 s  (s = negative, m = magnitude two) */
static int field_of(int v, uint32_t *field)
{
    switch (v) {
    case 1:  *field = 0u; return 0;
    case 2:  *field = 1u; return 0;
    case -1: *field = 2u; return 0;
    case -2: *field = 3u; return 0;
    default: return -1;
    }
}

static int value_of(uint32_t field)
{
    uint32_t m = field & 1u;
    uint32_t s = (field >> 1) & 1u;
    return (1 - 2 * (int)s) * (1 + (int)m);
}

static uint32_t field_at(const uint32_t *words, int64_t wpf, int64_t k, int64_t i)
{
    uint32_t w = words[k * wpf + i / 16];
    uint32_t m = (w >> magnitude_bit(i)) & 1u;
    uint32_t s = (w >> sign_bit(i)) & 1u;
    return m + 2u * s;
}

int orc_pack(const int8_t *wt, int64_t K, int64_t n, uint32_t *words)
{
    int64_t wpf = orc_words_per_filter(n);
    for (int64_t k = 0; k < K; ++k) {
        for (int64_t j = 0; j < wpf; ++j)
            words[k * wpf + j] = 0u;
        for (int64_t i = 0; i < n; ++i) {
            uint32_t f;
            if (field_of(wt[k * n + i], &f) != 0)
                return -1;
            uint32_t m = f & 1u, s = f >> 1;
            words[k * wpf + i / 16] |= (m << magnitude_bit(i)) | (s << sign_bit(i));
        }
    }
    return 0;
}

int orc_unpack(const uint32_t *words, int64_t K, int64_t n, int8_t *wt)
{
    int64_t wpf = orc_words_per_filter(n);
    int bad_padding = 0;
    for (int64_t k = 0; k < K; ++k) {
        for (int64_t i = 0; i < n; ++i)
            wt[k * n + i] = (int8_t)value_of(field_at(words, wpf, k, i));
        for (int64_t i = n; i < wpf * 16; ++i)
            if (field_at(words, wpf, k, i) != 0u)
                bad_padding = 1;
    }
    return bad_padding ? -1 : 0;
}

/* Canonical ("sequential") two-bit layout, the interchange format: the same
 * field f = m + 2 s per code, code i of a filter in word i / 16 at bits
 * 2 (i mod 16) (the bit m) and 2 (i mod 16) + 1 (the bit s), little-endian,
 * unused fields 0. */
static uint32_t canonical_field_at(const uint32_t *words, int64_t wpf, int64_t k, int64_t i)
{
    uint32_t w = words[k * wpf + i / 16];
    return (w >> (2 * (i % 16))) & 3u;
}

int orc_pack_canonical(const int8_t *wt, int64_t K, int64_t n, uint32_t *words)
{
    int64_t wpf = orc_words_per_filter(n);
    for (int64_t k = 0; k < K; ++k) {
        for (int64_t j = 0; j < wpf; ++j)
            words[k * wpf + j] = 0u;
        for (int64_t i = 0; i < n; ++i) {
            uint32_t f;
            if (field_of(wt[k * n + i], &f) != 0)
                return -1;
            words[k * wpf + i / 16] |= f << (2 * (i % 16));
        }
    }
    return 0;
}

int orc_unpack_canonical(const uint32_t *words, int64_t K, int64_t n, int8_t *wt)
{
    int64_t wpf = orc_words_per_filter(n);
    int bad_padding = 0;
    for (int64_t k = 0; k < K; ++k) {
        for (int64_t i = 0; i < n; ++i)
            wt[k * n + i] = (int8_t)value_of(canonical_field_at(words, wpf, k, i));
        for (int64_t i = n; i < wpf * 16; ++i)
            if (canonical_field_at(words, wpf, k, i) != 0u)
                bad_padding = 1;
    }
    return bad_padding ? -1 : 0;
}

/* ---- Eq. 2 (Section 2): quantization error ------------------------------ */
double orc_quant_error(const float *W, const int8_t *wt, int64_t n, double alpha)
{
    double j = 0.0;
    for (int64_t i = 0; i < n; ++i) {
        double d = (double)W[i] - alpha * (double)wt[i];
        j += d * d;
    }
    return j;
}

/* ---- Eq. 1 (Section 2): convolution with alpha W~ ----------------------- */
static void conv_one_site(const float *x, int64_t C, int64_t H, int64_t W,
                          const int8_t *wt, const double *alpha, int64_t R,
                          int64_t S, int64_t sh, int64_t sw, int64_t ph,
                          int64_t pw, int64_t b, int64_t k, int64_t p,
                          int64_t q, double *y_out, double *bound_out)
{
    double acc = 0.0, abs_sum = 0.0;
    for (int64_t c = 0; c < C; ++c)
        for (int64_t r = 0; r < R; ++r)
            for (int64_t s = 0; s < S; ++s) {
                int64_t h = p * sh - ph + r;
                int64_t w = q * sw - pw + s;
                if (h < 0 || h >= H || w < 0 || w >= W)
                    continue; /* zero padding */
                double xv = (double)x[((b * C + c) * H + h) * W + w];
                double wv = (double)wt[((k * C + c) * R + r) * S + s];
                acc += xv * wv;
                abs_sum += fabs(xv);
            }
    *y_out = alpha[k] * acc;
    if (bound_out)
        *bound_out = fabs(alpha[k]) * abs_sum;
}

static int64_t out_extent(int64_t in, int64_t k, int64_t stride, int64_t pad)
{
    return (in + 2 * pad - k) / stride + 1;
}

void orc_conv2d_nchw(const float *x, int64_t N, int64_t C, int64_t H, int64_t W,
                     const int8_t *wt, const double *alpha, int64_t K, int64_t R,
                     int64_t S, int64_t sh, int64_t sw, int64_t ph, int64_t pw,
                     double *y, double *bound)
{
    int64_t P = out_extent(H, R, sh, ph);
    int64_t Q = out_extent(W, S, sw, pw);
    int64_t NK = N * K;
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1)
#endif
    for (int64_t bk = 0; bk < NK; ++bk) {
        int64_t b = bk / K, k = bk % K;
        for (int64_t p = 0; p < P; ++p)
            for (int64_t q = 0; q < Q; ++q) {
                int64_t o = ((b * K + k) * P + p) * Q + q;
                conv_one_site(x, C, H, W, wt, alpha, R, S, sh, sw, ph, pw, b,
                              k, p, q, &y[o], bound ? &bound[o] : NULL);
            }
    }
}

/* ---- Algorithm 1, TwoBitBackward: gradients through Eq. 1 -------------- */
/* dx is the adjoint of the convolution with the approximate filters
 * alpha[k] wt[k]: every product that Eq. 1 adds into y[b,k,p,q] sends
 * dy[b,k,p,q] * alpha[k] * wt back to the input element it read. */
void orc_conv2d_bwd_data_nchw(const float *dy, int64_t N, int64_t K, int64_t P,
                              int64_t Q, const int8_t *wt, const double *alpha,
                              int64_t C, int64_t H, int64_t W, int64_t R, int64_t S,
                              int64_t sh, int64_t sw, int64_t ph, int64_t pw,
                              double *dx, double *bound)
{
    for (int64_t i = 0; i < N * C * H * W; ++i) {
        dx[i] = 0.0;
        if (bound)
            bound[i] = 0.0;
    }
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1)
#endif
    for (int64_t b = 0; b < N; ++b)
        for (int64_t k = 0; k < K; ++k)
            for (int64_t p = 0; p < P; ++p)
                for (int64_t q = 0; q < Q; ++q) {
                    double g = (double)dy[((b * K + k) * P + p) * Q + q];
                    for (int64_t c = 0; c < C; ++c)
                        for (int64_t r = 0; r < R; ++r)
                            for (int64_t s = 0; s < S; ++s) {
                                int64_t h = p * sh + r - ph;
                                int64_t w = q * sw + s - pw;
                                if (h < 0 || h >= H || w < 0 || w >= W)
                                    continue;
                                double wv = alpha[k] * (double)wt[((k * C + c) * R + r) * S + s];
                                int64_t o = ((b * C + c) * H + h) * W + w;
                                dx[o] += g * wv;
                                if (bound)
                                    bound[o] += fabs(g * wv);
                            }
                }
}

/* dW^[k,c,r,s] = sum over (b, p, q) of dy[b,k,p,q] times the input element
 * x[b, c, p sh - ph + r, q sw - pw + s] that Eq. 1 multiplies by
 * W^[k,c,r,s] (zero outside the image). */
void orc_conv2d_bwd_filter_nchw(const float *x, int64_t N, int64_t C, int64_t H,
                                int64_t W, const float *dy, int64_t K, int64_t P,
                                int64_t Q, int64_t R, int64_t S, int64_t sh, int64_t sw,
                                int64_t ph, int64_t pw, double *dw, double *bound)
{
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1)
#endif
    for (int64_t k = 0; k < K; ++k)
        for (int64_t c = 0; c < C; ++c)
            for (int64_t r = 0; r < R; ++r)
                for (int64_t s = 0; s < S; ++s) {
                    double acc = 0.0, mag = 0.0;
                    for (int64_t b = 0; b < N; ++b)
                        for (int64_t p = 0; p < P; ++p)
                            for (int64_t q = 0; q < Q; ++q) {
                                int64_t h = r + p * sh - ph;
                                int64_t w = s + q * sw - pw;
                                if (h < 0 || h >= H || w < 0 || w >= W)
                                    continue;
                                double t = (double)dy[((b * K + k) * P + p) * Q + q] *
                                           (double)x[((b * C + c) * H + h) * W + w];
                                acc += t;
                                mag += fabs(t);
                            }
                    int64_t o = ((k * C + c) * R + r) * S + s;
                    dw[o] = acc;
                    if (bound)
                        bound[o] = mag;
                }
}

void orc_conv2d_nchw_sites(const float *x, int64_t N, int64_t C, int64_t H,
                           int64_t W, const int8_t *wt, const double *alpha,
                           int64_t K, int64_t R, int64_t S, int64_t sh,
                           int64_t sw, int64_t ph, int64_t pw,
                           const int64_t *sites, int64_t npts, double *y,
                           double *bound)
{
    (void)N;
    (void)K;
#ifdef _OPENMP
#pragma omp parallel for schedule(static)
#endif
    for (int64_t j = 0; j < npts; ++j) {
        const int64_t *t = sites + 4 * j;
        conv_one_site(x, C, H, W, wt, alpha, R, S, sh, sw, ph, pw, t[0], t[1],
                      t[2], t[3], &y[j], bound ? &bound[j] : NULL);
    }
}

/* ---- Section 3: fully-connected layer as a convolution ------------------ */
void orc_linear(const float *x, int64_t B, int64_t Kin, const int8_t *wt,
                const double *alpha, int64_t Kout, double *y, double *bound)
{
#ifdef _OPENMP
#pragma omp parallel for schedule(static)
#endif
    for (int64_t bk = 0; bk < B * Kout; ++bk) {
        int64_t b = bk / Kout, k = bk % Kout;
        double acc = 0.0, abs_sum = 0.0;
        for (int64_t j = 0; j < Kin; ++j) {
            double xv = (double)x[b * Kin + j];
            acc += xv * (double)wt[k * Kin + j];
            abs_sum += fabs(xv);
        }
        y[bk] = alpha[k] * acc;
        if (bound)
            bound[bk] = fabs(alpha[k]) * abs_sum;
    }
}

/* ---- network glue ------------------------------------------------------- */
void orc_epilogue(double *y, const double *residual, int64_t count, int relu)
{
    for (int64_t i = 0; i < count; ++i) {
        double v = y[i];
        if (residual)
            v += residual[i];
        if (relu && v < 0.0)
            v = 0.0;
        y[i] = v;
    }
}

void orc_maxpool2d_nchw(const double *x, int64_t N, int64_t C, int64_t H,
                        int64_t W, int64_t kh, int64_t kw, int64_t sh,
                        int64_t sw, int64_t ph, int64_t pw, double *y)
{
    int64_t Ho = (H + 2 * ph - kh) / sh + 1, Wo = (W + 2 * pw - kw) / sw + 1;
    for (int64_t b = 0; b < N; ++b)
        for (int64_t c = 0; c < C; ++c)
            for (int64_t i = 0; i < Ho; ++i)
                for (int64_t j = 0; j < Wo; ++j) {
                    double m = -INFINITY;
                    for (int64_t u = 0; u < kh; ++u)
                        for (int64_t v = 0; v < kw; ++v) {
                            int64_t h = i * sh - ph + u, w = j * sw - pw + v;
                            if (h < 0 || h >= H || w < 0 || w >= W)
                                continue; /* padding never wins the max */
                            double t = x[((b * C + c) * H + h) * W + w];
                            if (t > m)
                                m = t;
                        }
                    y[((b * C + c) * Ho + i) * Wo + j] = m;
                }
}

/* ---- the full-precision layers around the two-bit ones ------------------ */
/* Networks keep their first convolution and last fully-connected layer in
 * full precision (the ResNet-18 workload); these are their definitions. */
void orc_dense_conv2d_nchw(const float *x, int64_t N, int64_t C, int64_t H, int64_t W,
                           const float *w, int64_t K, int64_t R, int64_t S, int64_t sh,
                           int64_t sw, int64_t ph, int64_t pw, double *y, double *bound)
{
    int64_t P = out_extent(H, R, sh, ph);
    int64_t Q = out_extent(W, S, sw, pw);
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1)
#endif
    for (int64_t bk = 0; bk < N * K; ++bk) {
        int64_t b = bk / K, k = bk % K;
        for (int64_t p = 0; p < P; ++p)
            for (int64_t q = 0; q < Q; ++q) {
                double acc = 0.0, mag = 0.0;
                for (int64_t c = 0; c < C; ++c)
                    for (int64_t r = 0; r < R; ++r)
                        for (int64_t s = 0; s < S; ++s) {
                            int64_t h_in = p * sh - ph + r;
                            int64_t w_in = q * sw - pw + s;
                            if (h_in < 0 || h_in >= H || w_in < 0 || w_in >= W)
                                continue; /* zero padding */
                            double xw = (double)x[((b * C + c) * H + h_in) * W + w_in] *
                                       (double)w[((k * C + c) * R + r) * S + s];
                            acc += xw;
                            mag += fabs(xw);
                        }
                int64_t o = ((b * K + k) * P + p) * Q + q;
                y[o] = acc;
                if (bound)
                    bound[o] = mag;
            }
    }
}

void orc_avgpool_global_nchw(const double *x, int64_t N, int64_t C, int64_t H, int64_t W,
                             double *y)
{
    for (int64_t b = 0; b < N; ++b)
        for (int64_t c = 0; c < C; ++c) {
            double acc = 0.0;
            for (int64_t h = 0; h < H; ++h)
                for (int64_t w = 0; w < W; ++w)
                    acc += x[((b * C + c) * H + h) * W + w];
            y[b * C + c] = acc / (double)(H * W);
        }
}

void orc_dense_linear(const float *x, int64_t B, int64_t Kin, const float *w, int64_t Kout,
                      double *y, double *bound)
{
#ifdef _OPENMP
#pragma omp parallel for schedule(static)
#endif
    for (int64_t bk = 0; bk < B * Kout; ++bk) {
        int64_t b = bk / Kout, k = bk % Kout;
        double acc = 0.0, mag = 0.0;
        for (int64_t j = 0; j < Kin; ++j) {
            double prod = (double)x[b * Kin + j] * (double)w[k * Kin + j];
            acc += prod;
            mag += fabs(prod);
        }
        y[bk] = acc;
        if (bound)
            bound[bk] = mag;
    }
}

int orc_num_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

void orc_set_num_threads(int n)
{
#ifdef _OPENMP
    if (n > 0)
        omp_set_num_threads(n);
#else
    (void)n;
#endif
}
