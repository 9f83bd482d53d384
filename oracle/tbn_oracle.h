/*
 * tbn_oracle.h -- CPU reference ("oracle") for Two-Bit Networks (Meng, Gu,
 * Zhang, Wu, arXiv:1701.00485).
 *
 * TEST INFRASTRUCTURE ONLY.  Only the test suite, the smoke check and the
 * CPU-baseline leg of the benchmark may load this library.  The product
 * (the CUDA library and its Python binding) never calls it, and it shares no
 * code, header, table or constant with the CUDA path.
 *
 * Everything is computed in IEEE double precision with plain loops in the
 * order the paper states the method:
 *   Eq. 3  (Section 2)  deterministic discretization W -> W~ in {-2,-1,1,2}
 *   Eq. 5  (Section 2)  optimal scaling factor alpha* given W~
 *   Eq. 2  (Section 2)  quantization error ||W - alpha W~||^2
 *   Eq. 1  (Section 2)  convolution with the approximated filter alpha W~
 *   Section 3           fully-connected layers treated as convolutions
 * plus the two-bit storage format (the paper fixes only that each of the four
 * values takes two bits, Section 1; the bit layout is this library's own and
 * is spelled out at orc_pack below).
 *
 * All arrays are caller-owned host memory; nothing is allocated that
 * outlives a call.
 */
#ifndef TBN_ORACLE_H
#define TBN_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Eq. 3 for one weight: returns -2, -1, 1 or 2. */
int orc_discretize_one(double w);

/* Eq. 3 over a filter of n weights: wt[i] = W~_i. */
void orc_discretize(const float *W, int64_t n, int8_t *wt);

/* Eq. 5: alpha* = (sum_{B1}|W_i| + 2 sum_{B2}|W_i|) / (|B1| + 4|B2|),
 * B1 = {i : |W_i| <= 1}, B2 = {i : |W_i| > 1}.  Sums are taken naively in
 * index order in double.  n >= 1. */
double orc_alpha(const float *W, int64_t n);

/* Algorithm 1 (quantization loop) for one layer: for each of the K filters
 * (row k of the row-major [K][n] matrix W) compute W~ by Eq. 3 and alpha by
 * Eq. 5.  wt is [K][n], alpha is [K]. */
void orc_quantize(const float *W, int64_t K, int64_t n, int8_t *wt, double *alpha);

/* Number of 32-bit words that hold one filter of n two-bit codes. */
int64_t orc_words_per_filter(int64_t n);

/* Two-bit storage format.  Each code is a 2-bit field (s, m):
 *   s = 1 when W~ < 0 (sign), m = 1 when |W~| = 2 (magnitude),
 *   field value = m + 2 s, i.e.  +1 -> 0, +2 -> 1, -1 -> 2, -2 -> 3,
 * and W~ = (1 - 2 s)(1 + m).  Code i of filter k lives in word
 * k * words_per_filter + i / 16.  With l = i mod 16, pair p = l / 2 and half
 * h = l mod 2, its m bit is bit 16 h + p of that word and its s bit is bit
 * 16 h + 8 + p ("byte-planar": byte 0 = m of the even codes, byte 1 = s of
 * the even codes, byte 2 = m of the odd codes, byte 3 = s of the odd codes).
 * Unused codes of the last word of a filter have m = s = 0.
 * words is [K][orc_words_per_filter(n)].  Returns 0, or -1 if some wt value
 * is not in {-2,-1,1,2}. */
int orc_pack(const int8_t *wt, int64_t K, int64_t n, uint32_t *words);

/* Inverse of orc_pack.  Returns 0, or -1 if a padding field is non-zero. */
int orc_unpack(const uint32_t *words, int64_t K, int64_t n, int8_t *wt);

/* Canonical two-bit layout (the interchange format): the same field
 * f = m + 2 s, code i of filter k at bits 2 (i mod 16) .. 2 (i mod 16) + 1 of
 * word k * words_per_filter + i / 16 (bit m low, bit s high), unused fields
 * 0.  Same return values as orc_pack / orc_unpack. */
int orc_pack_canonical(const int8_t *wt, int64_t K, int64_t n, uint32_t *words);
int orc_unpack_canonical(const uint32_t *words, int64_t K, int64_t n, int8_t *wt);

/* Eq. 2 objective evaluated directly: sum_i (W_i - alpha wt_i)^2. */
double orc_quant_error(const float *W, const int8_t *wt, int64_t n, double alpha);

/* Eq. 1, direct seven-loop cross-correlation in NCHW order with zero padding:
 *   acc[b,k,p,q] = sum_{c,r,s} x[b,c,p*sh-ph+r, q*sw-pw+s] * wt[k,c,r,s]
 *   y[b,k,p,q]   = alpha[k] * acc          (alpha applied to the output;
 *                                           Eq. 1 scales the input -- equal
 *                                           by linearity)
 *   bound[...]   = |alpha[k]| * sum of |x| over the taps inside the image
 * x is [N][C][H][W] (fp32 values, widened to double), wt [K][C][R][S],
 * y and bound are [N][K][P][Q] with P = (H + 2ph - R)/sh + 1 and
 * Q = (W + 2pw - S)/sw + 1.  bound may be NULL.
 * Parallel over (b, k) with OpenMP when built with it. */
void orc_conv2d_nchw(const float *x, int64_t N, int64_t C, int64_t H, int64_t W,
                     const int8_t *wt, const double *alpha, int64_t K, int64_t R,
                     int64_t S, int64_t sh, int64_t sw, int64_t ph, int64_t pw,
                     double *y, double *bound);

/* Same definition evaluated only at the npts output sites
 * sites[4 j .. 4 j + 3] = (b, k, p, q); results go to y[j], bound[j]. */
void orc_conv2d_nchw_sites(const float *x, int64_t N, int64_t C, int64_t H,
                           int64_t W, const int8_t *wt, const double *alpha,
                           int64_t K, int64_t R, int64_t S, int64_t sh,
                           int64_t sw, int64_t ph, int64_t pw,
                           const int64_t *sites, int64_t npts, double *y,
                           double *bound);

/* Algorithm 1, TwoBitBackward, through one convolution (Eq. 1) with the
 * approximate filters W^ = alpha[k] wt[k]:
 *   dx[b,c,h,w] = sum over (k, p, q, r, s) with p sh - ph + r = h and
 *                 q sw - pw + s = w of dy[b,k,p,q] * alpha[k] * wt[k,c,r,s]
 *   bound[...]  = the same sum of absolute values.
 * dy is [N][K][P][Q] (fp32 values), wt [K][C][R][S], dx and bound
 * [N][C][H][W]; bound may be NULL. */
void orc_conv2d_bwd_data_nchw(const float *dy, int64_t N, int64_t K, int64_t P,
                              int64_t Q, const int8_t *wt, const double *alpha,
                              int64_t C, int64_t H, int64_t W, int64_t R, int64_t S,
                              int64_t sh, int64_t sw, int64_t ph, int64_t pw,
                              double *dx, double *bound);

/*   dW^[k,c,r,s] = sum over (b, p, q) of dy[b,k,p,q] *
 *                  x[b, c, p sh - ph + r, q sw - pw + s]   (zero outside)
 *   bound[...]   = the same sum of absolute values.
 * x [N][C][H][W], dy [N][K][P][Q] (fp32 values), dw and bound [K][C][R][S];
 * bound may be NULL. */
void orc_conv2d_bwd_filter_nchw(const float *x, int64_t N, int64_t C, int64_t H,
                                int64_t W, const float *dy, int64_t K, int64_t P,
                                int64_t Q, int64_t R, int64_t S, int64_t sh, int64_t sw,
                                int64_t ph, int64_t pw, double *dw, double *bound);

/* Fully-connected layer (Section 3: treated as a convolution):
 *   y[b,k] = alpha[k] * sum_j x[b,j] * wt[k,j],
 *   bound[b,k] = |alpha[k]| * sum_j |x[b,j]|.
 * x [B][Kin], wt [Kout][Kin], y and bound [B][Kout]; bound may be NULL. */
void orc_linear(const float *x, int64_t B, int64_t Kin, const int8_t *wt,
                const double *alpha, int64_t Kout, double *y, double *bound);

/* Layer epilogue used by the benchmark networks (not part of the paper's
 * method): v = y + residual (if residual != NULL), then max(v, 0) if relu.
 * In place on y[count]. */
void orc_epilogue(double *y, const double *residual, int64_t count, int relu);

/* Max pooling in NCHW (network glue between TBN layers): window kh x kw,
 * stride sh x sw, padding ph x pw (taps outside the image are skipped, i.e.
 * padded with -infinity).  y is [N][C][Ho][Wo], Ho = (H + 2 ph - kh)/sh + 1. */
void orc_maxpool2d_nchw(const double *x, int64_t N, int64_t C, int64_t H,
                        int64_t W, int64_t kh, int64_t kw, int64_t sh,
                        int64_t sw, int64_t ph, int64_t pw, double *y);

/* Full-precision layers of the networks (first convolution and last
 * fully-connected layer of ResNet-18; not part of the paper's method):
 *   dense conv:   y[b,k,p,q] = sum_{c,r,s} x[b,c,p sh-ph+r,q sw-pw+s] w[k,c,r,s]
 *                 (zero padding), bound = the same sum of |products|;
 *                 x [N][C][H][W], w [K][C][R][S] fp32, y/bound [N][K][P][Q];
 *   global average pool: y[b,c] = mean of x[b,c,:,:]; x [N][C][H][W];
 *   dense linear: y[b,k] = sum_j x[b,j] w[k,j], bound = sum_j |x[b,j] w[k,j]|;
 *                 x [B][Kin], w [Kout][Kin] fp32.
 * bound may be NULL. */
void orc_dense_conv2d_nchw(const float *x, int64_t N, int64_t C, int64_t H, int64_t W,
                           const float *w, int64_t K, int64_t R, int64_t S, int64_t sh,
                           int64_t sw, int64_t ph, int64_t pw, double *y, double *bound);
void orc_avgpool_global_nchw(const double *x, int64_t N, int64_t C, int64_t H, int64_t W,
                             double *y);
void orc_dense_linear(const float *x, int64_t B, int64_t Kin, const float *w, int64_t Kout,
                      double *y, double *bound);

/* Threads the parallel loops use (1 without OpenMP). */
int orc_num_threads(void);

/* Set the thread count of the parallel loops (n >= 1; no effect without
 * OpenMP).  Used to time the oracle single-threaded beside all cores. */
void orc_set_num_threads(int n);

#ifdef __cplusplus
}
#endif

#endif /* TBN_ORACLE_H */
