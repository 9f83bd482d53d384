/*
 * tbn.h -- C ABI of the Two-Bit Networks (TBN) GPU library for GB300 (sm_103a).
 *
 * Two-Bit Networks (Meng, Gu, Zhang, Wu, arXiv:1701.00485) approximate each
 * real-valued filter W of a convolutional or fully-connected layer by
 * alpha * W~, with W~ in {-2,-1,1,2}^n stored at two bits per weight.  This
 * library provides the data-parallel hot path of the method:
 *
 *   tbn_quantize_pack   discretization (Eq. 3) + optimal scaling factor
 *                       (Eq. 5) for every filter of a layer, packed
 *   tbn_unpack          packed codes -> int8 W~ or dequantized alpha W~
 *   tbn_conv2d_fwd      convolution with alpha W~ (Eq. 1)
 *   tbn_linear_fwd      fully-connected layer, treated as a convolution
 *                       (Section 3); tbn_linear_fwd_ws with caller-owned
 *                       scratch for the batch-1 fp32 table-lookup GEMV
 *   tbn_conv2d_bwd_data, tbn_conv2d_bwd_filter   Algorithm 1's
 *                       TwoBitBackward through a convolution
 *   tbn_repack          byte-planar codes <-> the canonical interchange layout
 *   tbn_maxpool2d_nhwc, tbn_nchw_to_nhwc   network glue between layers
 *   tbn_dense_conv2d_fwd, tbn_avgpool2d_global_nhwc, tbn_dense_linear_fwd
 *                       the full-precision layers a network keeps around its
 *                       two-bit layers (first convolution, global average
 *                       pool, last fully-connected layer)
 *
 * Conventions shared by every call
 * --------------------------------
 * - Pointers to tensors are DEVICE pointers, allocated and owned by the
 *   caller.  The library allocates no device memory and keeps no state
 *   between calls except the per-device error word (tbn_device_error),
 *   per-process kernel attributes and the 4 MiB scratch array of
 *   tbn_linear_fwd_noalloc (one per device and process; calls of that entry
 *   point that could overlap must be serialized, see its declaration).
 * - One process drives one GPU (run one process per GPU for replicas): the
 *   kernels' shared-memory attributes are set on the device that is current
 *   at a kernel's first launch in the process, so a later launch of a
 *   large-shared-memory kernel on another device can fail with TBN_ERR_CUDA.
 * - Every compute call is asynchronous on `stream` (a cudaStream_t; NULL is
 *   the legacy default stream).  Arguments are validated on the host before
 *   anything is launched; an invalid call returns a status and launches
 *   nothing.  No call aborts the process or throws.
 * - Kernel-side waits are bounded in time.  A wait that expires sets a bit
 *   in the per-device error word and the kernel returns early; read it with
 *   tbn_device_error() after synchronizing.
 * - tbn_last_error() returns a human-readable detail string for the most
 *   recent failing call on the calling host thread.
 * - The convolutions are launched as programmatic dependents of the previous
 *   kernel on `stream`: their start-up may overlap that kernel's end, and
 *   they read activations and residuals only after it has completed.  Codes
 *   and alpha may be read earlier, while a previous convolution of this
 *   library (or tbn_nchw_to_nhwc) is still finishing, so they must not be
 *   the output of the immediately preceding call.  Everything older, and
 *   every other kind of preceding kernel, is complete before they start.
 *
 * Two-bit storage format (the paper fixes only that each of the four values
 * takes two bits, Section 1; the layout below is this library's):
 * - each code is a 2-bit field f = m + 2 s with s = 1 for a negative value and
 *   m = 1 for magnitude two:  +1 -> 0, +2 -> 1, -1 -> 2, -2 -> 3;
 *   W~ = (1 - 2 s)(1 + m);
 * - a filter of n codes occupies tbn_packed_words(n) = ceil(n / 16) uint32
 *   words; code i of filter k is in word k * ceil(n / 16) + i / 16;
 * - inside a word ("byte-planar"), code l = i mod 16 = 2p + h (pair p in
 *   0..7, half h in {0, 1}) has its m bit at bit 16h + p and its s bit at
 *   bit 16h + 8 + p: byte 0 = m of the even codes, byte 1 = s of the even
 *   codes, byte 2 = m of the odd codes, byte 3 = s of the odd codes.  A pair
 *   of codes then decodes to two bf16 values with one mask and one
 *   multiply-add (the tensor-core kernels), and the four (m, s) nibble pairs
 *   of a byte pair index the table-lookup GEMV's tables directly;
 * - unused codes of a filter's last word have m = s = 0;
 * - codes[K][ceil(n/16)] plus alpha[K] (fp32) is the complete inference
 *   form of a layer: inference reads nothing else of the layer (Section 3).
 * - The order of the n weights of a filter is the caller's choice; the
 *   convolution reads them in the activation layout's natural order:
 *   NCHW -> (c, r, s), NHWC and NCHW_NHWC -> (r, s, c).  Discretization is elementwise and
 *   alpha does not depend on the order, so permuting fp32 weights before
 *   tbn_quantize_pack is how either order is produced.
 */
#ifndef TBN_H
#define TBN_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define TBN_ABI_VERSION 9

typedef enum {
  TBN_OK = 0,
  TBN_ERR_INVALID_ARG = 1, /* null pointer, non-positive size, bad enum, overflow */
  TBN_ERR_UNSUPPORTED = 2, /* valid request that no kernel here implements       */
  TBN_ERR_MISALIGNED = 3,  /* a pointer violates the alignment the call needs    */
  TBN_ERR_CUDA = 4,        /* a CUDA runtime/driver call failed (see last_error) */
  TBN_ERR_TIMEOUT = 5      /* reserved for callers mapping the device error word */
} tbn_status;

typedef enum { TBN_F32 = 0, TBN_BF16 = 1 } tbn_dtype;

/* Activation layouts.  TBN_NCHW_NHWC (convolutions only) reads an NCHW x
 * and writes an NHWC y (and residual), with codes in the NHWC order
 * (r, s, c): the first layer of an NHWC network can read its NCHW input
 * batch without a converted copy (small-tap and direct kernels).
 * TBN_S2D_NHWC (convolutions only) reads x in the space-to-depth form that
 * tbn_space_to_depth writes for the same convolution and writes an NHWC y;
 * sizes, stride, padding and codes ((r, s, c) order) are those of the
 * convolution on the original input. */
typedef enum { TBN_NCHW = 0, TBN_NHWC = 1, TBN_NCHW_NHWC = 2, TBN_S2D_NHWC = 3 } tbn_layout;

typedef enum {
  TBN_UNPACK_I8 = 0,   /* int8 W~ in {-2,-1,1,2}                 */
  TBN_UNPACK_F32 = 1,  /* fp32 alpha[k] * W~                      */
  TBN_UNPACK_BF16 = 2  /* bf16 alpha[k] * W~ (round to nearest)   */
} tbn_unpack_format;

/* Convolution algorithms.  AUTO picks the fastest implemented one. */
typedef enum {
  TBN_CONV_AUTO = 0,
  TBN_CONV_DIRECT = 1,        /* CUDA-core direct convolution, any layout/dtype   */
  TBN_CONV_IMPLICIT_GEMM = 2, /* tcgen05 implicit GEMM, NHWC bf16 x; activations
                                 by TMA when C % 64 == 0, else gathered by threads */
  TBN_CONV_SMALL_TAPS = 3     /* tensor-core convolution for short filters,
                                 C*R*S <= 64, bf16 x in any layout, no fused
                                 pool: the input patch and its im2col
                                 expansion are staged in shared memory
                                 (tcgen05 for NHWC x and bf16 NHWC y without
                                 residual, K % 8 == 0; mma.sync otherwise)   */
} tbn_conv_algo;

/* Fused layer epilogue (network glue, not part of the paper's method):
 *   v = alpha[k] * acc;  if (residual) v += residual[same index];
 *   if (relu) v = max(v, 0);
 *   if (pool == 2) v = max of v over a 2x2 window, stride 2 (floor sizes);
 *   y = v rounded to y's dtype.
 * `residual` has y's layout, shape and dtype (not combinable with pool).
 * With pool == 2, y is [N][P/2][Q/2][K] (NHWC, NCHW_NHWC) / [N][K][P/2][Q/2]
 * (NCHW).
 * Pass NULL for no epilogue. */
typedef struct {
  int relu;
  const void *residual;
  int pool; /* 0: none, 2: 2x2 max pool, stride 2 */
} tbn_epilogue;

/* A cudaStream_t, passed as an opaque pointer. */
typedef void *tbn_stream;

/* ------------------------------------------------------------------------ */

/* ABI version of the loaded library (TBN_ABI_VERSION). */
int tbn_abi_version(void);

/* Words per filter for n codes: ceil(n / 16); -1 if n < 1. */
int64_t tbn_packed_words(int64_t n);

/* Static description of a status code. */
const char *tbn_status_string(tbn_status s);

/* Detail of the most recent failure on this host thread ("" if none). */
const char *tbn_last_error(void);

/* Reads and clears the error word of the current device (synchronous:
 * waits for the device's pending work; the read and the clear are one atomic
 * step on the device).  Bit 1: a kernel wait timed out;
 * bit 2: a kernel saw a launch shape it could not run.  *flags = 0 when no
 * error was recorded. */
tbn_status tbn_device_error(uint32_t *flags);

/* Self-check of the failure detection that every kernel's waits rely on:
 * launches one thread that waits, through the same bounded wait, on a
 * shared-memory mbarrier that nothing arrives at.  After limit_us
 * microseconds (1 .. 1000000) the wait gives up, sets bit 1 (timeout) of
 * the current device's error word and the kernel returns; the device stays
 * usable.  Asynchronous on `stream`; read the result with tbn_device_error.
 * TBN_ERR_INVALID_ARG for a limit out of range. */
tbn_status tbn_selftest_wait_timeout(uint32_t limit_us, tbn_stream stream);

/* Quantize and pack one layer -- Algorithm 1, quantization loop; Eq. 3
 * (discretization) and Eq. 5 (optimal scaling factor), Section 2.
 *
 *   W      [K][n] fp32, row k = filter k (device).  Any 4-byte alignment;
 *          16-byte alignment with n % 4 == 0 takes the vector-load path.
 *   codes  [K][tbn_packed_words(n)] uint32 (device, output), 4-byte aligned.
 *   alpha  [K] fp32 (device, output):
 *          alpha_k = (sum_{|W|<=1} |W| + 2 sum_{|W|>1} |W|) / (n + 3 |{|W|>1}|)
 *          the sum of 16 weights of a word in fp32, the word sums added
 *          exactly as fp32 pairs (two-float TwoSum; fp64 only when a word sum
 *          overflows fp32), rounded once to fp32.  An all-zero filter gets
 *          alpha = 0.
 *   Eq. 3 per weight: W < -1 -> -2; -1 <= W <= 0 -> -1 (including -0.0);
 *          0 < W <= 1 -> 1; W > 1 -> 2.  NaN weights are undefined input.
 * K >= 1, 1 <= n < 2^31, K * tbn_packed_words(n) < 2^40. */
tbn_status tbn_quantize_pack(const float *W, int64_t K, int64_t n, uint32_t *codes,
                             float *alpha, tbn_stream stream);

/* One layer of a grouped quantization call (see tbn_quantize_pack_group). */
typedef struct {
  const float *W;
  int64_t K;
  int64_t n;
  uint32_t *codes;
  float *alpha;
} tbn_quant_job;

/* Up to TBN_MAX_QUANT_JOBS layers quantized by one kernel launch (used to
 * re-quantize every layer of a network per forward pass, Algorithm 1).  Each
 * job follows tbn_quantize_pack's contract; jobs must not overlap in memory.
 * The job table is passed by value to the kernel; nothing is allocated. */
#define TBN_MAX_QUANT_JOBS 16
tbn_status tbn_quantize_pack_group(const tbn_quant_job *jobs, int njobs, tbn_stream stream);

/* Unpack codes [K][tbn_packed_words(n)] into out [K][n] as int8 W~, or as
 * fp32 / bf16 alpha[k] * W~ (alpha may be NULL only for TBN_UNPACK_I8).
 * Padding fields are ignored. */
tbn_status tbn_unpack(const uint32_t *codes, const float *alpha, int64_t K, int64_t n,
                      void *out, tbn_unpack_format fmt, tbn_stream stream);

/* Batch-1 two-bit linear layer on fp8 tensor cores (Section 3: y[k] =
 * alpha[k] sum_j x[j] W~[k, j]).  W~/2 in {+-0.5, +-1} is exact in e4m3; x
 * (bf16) is split exactly into three e4m3 terms under one power-of-two
 * scale, x 2^E = t1 + t2/16 + t3/256 + r with |r| <= 2^-25 max|x| per
 * element, so the result stays within 2e-3 alpha sum|x| for K_in <= 16384;
 * accumulation is fp32, and the partial sums of a row are added in a fixed
 * order (bitwise reproducible).
 *
 * tbn_linear_prepare_f8 rewrites codes [K_out][tbn_packed_words(K_in)]
 * (the byte-planar layout; K_in a multiple of 512) into this path's
 * prepared layout, once per weight matrix: "e4m3-planar" words (the 16
 * codes of a word, code 4j + b at bits 8b + j (m) and 8b + 4 + j (s)),
 * blocked by 128 rows x 512 codes (16 KiB contiguous per block, the 16-byte
 * chunks of a row permuted by the row's low 3 bits), rows past K_out zero.
 * prepared holds tbn_linear_f8_prepared_words(K_out, K_in) words (-1: the
 * shape is not taken), 16-byte aligned, not overlapping codes.
 *
 * tbn_linear_fwd_f8 runs it: x bf16 [1][K_in], K_in a multiple of 512 and at
 * most 16384, x 16-byte aligned, prepared codes of the same K_out and K_in, alpha fp32 [K_out], y [1][K_out]
 * bf16 or fp32, optional epilogue (ReLU, residual; no pool), and a caller
 * workspace (256-byte aligned, contents on entry irrelevant, at least
 * tbn_linear_f8_workspace_bytes) that calls which may run concurrently must
 * not share.  One launch when the 128-row tiles fill most SMs (each CTA
 * owns whole tiles), else two (the rows' K ranges are spread over CTAs and
 * a second kernel adds their partial sums in a fixed order).
 * tbn_linear_f8_workspace_bytes returns 0 for shapes this path does not
 * take (then tbn_linear_fwd_f8 returns TBN_ERR_UNSUPPORTED). */
int64_t tbn_linear_f8_prepared_words(int64_t K_out, int64_t K_in);
tbn_status tbn_linear_prepare_f8(const uint32_t *codes, int64_t K_out, int64_t K_in,
                                 uint32_t *prepared, tbn_stream stream);
size_t tbn_linear_f8_workspace_bytes(int64_t B, int64_t K_in, int64_t K_out);
tbn_status tbn_linear_fwd_f8(const void *x, tbn_dtype xdt, int64_t B, int64_t K_in,
                             const uint32_t *prepared, const float *alpha, int64_t K_out, void *y,
                             tbn_dtype ydt, const tbn_epilogue *epi, void *workspace,
                             size_t workspace_bytes, tbn_stream stream);

/* Canonical ("sequential") two-bit layout, the interchange format for codes
 * exchanged with other software: the same field f = m + 2 s per code (Section
 * 1: two bits per weight), code i of filter k in word
 * k * tbn_packed_words(n) + i / 16 at bits 2 (i mod 16) (m) and
 * 2 (i mod 16) + 1 (s), little-endian, unused fields 0.  The worked example
 * W~ = (-2, -1, -1, -1, 1, 1, 2, 2) is 0x000050AB in this layout and
 * 0x03080309 in the library's byte-planar one. */
typedef enum {
  TBN_REPACK_CANONICAL_TO_PLANAR = 0,
  TBN_REPACK_PLANAR_TO_CANONICAL = 1
} tbn_repack_direction;

/* Repack codes [K][tbn_packed_words(n)] between the two layouts (a fixed
 * permutation of the bits of each word; unused fields stay 0).  in and out
 * are 4-byte aligned device arrays of the same size; they may be the same
 * array (in place) but must not otherwise overlap.  Asynchronous on `stream`. */
tbn_status tbn_repack(const uint32_t *in, int64_t K, int64_t n, uint32_t *out,
                      tbn_repack_direction dir, tbn_stream stream);

/* Two-bit convolution, Eq. 1 (Section 2): cross-correlation with zero
 * padding, no bias, groups = 1, dilation = 1 (the paper states none of
 * these; they follow the Torch7 convention the paper's experiments used).
 *
 *   y[b,k,p,q] = alpha[k] * sum_{c,r,s} x[b,c,p*sh-ph+r,q*sw-pw+s] W~[k,c,r,s]
 *
 *   x      activations (device).  layout NCHW and NCHW_NHWC: [N][C][H][W];
 *          NHWC: [N][H][W][C].  dtype fp32 or bf16.
 *   codes  [K][tbn_packed_words(C*R*S)], filter order (c,r,s) for NCHW and
 *          (r,s,c) for NHWC and NCHW_NHWC.   alpha [K] fp32.
 *   y      [N][K][P][Q] (NCHW) or [N][P][Q][K] (NHWC, NCHW_NHWC), dtype
 *          fp32 or bf16, P = (H + 2 ph - R) / sh + 1, Q = (W + 2 pw - S) / sw + 1.
 *   epi    optional fused epilogue (NULL = none).
 * Accumulation is fp32; x * W~ products are exact.  y must not alias x.
 * The tensor-core implicit-GEMM path needs NHWC and bf16 x (16-byte aligned
 * x, y and residual; stride 1 or 2 when C % 64 == 0, any stride otherwise);
 * the small-tap path takes bf16 x with C*R*S <= 64 in any layout; AUTO falls
 * back to the CUDA-core direct kernel for every other case. */
tbn_status tbn_conv2d_fwd(const void *x, tbn_dtype xdt, tbn_layout layout, int64_t N,
                          int64_t C, int64_t H, int64_t W, const uint32_t *codes,
                          const float *alpha, int64_t K, int64_t R, int64_t S,
                          int64_t stride_h, int64_t stride_w, int64_t pad_h, int64_t pad_w,
                          void *y, tbn_dtype ydt, const tbn_epilogue *epi, tbn_stream stream);

/* Space-to-depth input of a strided convolution with few channels (not in
 * the paper; a layout change that lets a first layer such as AlexNet's
 * 11x11 stride-4 convolution over 3 channels run on the tensor-core
 * implicit GEMM).  With s = stride_h = stride_w >= 2, s*s*C <= 64,
 * P, Q the output size, R' = ceil(R / s), S' = ceil(S / s), it writes
 *   out [N][Hs][Ws][64] bf16,  Hs = P + R' - 1,  Ws = Q + S' - 1,
 *   out[n][Y][X][(dy s + dx) C + c] = x[n, c, s Y + dy - pad_h, s X + dx - pad_w]
 * (dy, dx in [0, s); zero outside the image and for channels >= s*s*C).
 * x is bf16, NCHW or NHWC, 2-byte aligned; out is 16-byte aligned and must
 * not overlap x.  The convolution of Eq. 1 over x then equals
 * tbn_conv2d_fwd with layout TBN_S2D_NHWC over out (a stride-1 R' x S'
 * convolution of the 64 channels, whose weights the kernel gathers from the
 * original codes; weights past the filter are zero).  That call needs
 * K <= 128, bf16 output or fp32, no pool and no residual, and R' S' K blocks
 * that fit in tensor memory beside the output tile (AlexNet's first layer:
 * R' = S' = 3).  Asynchronous on `stream`.
 * tbn_space_to_depth_elems returns the element count of out, or -1 when the
 * geometry is invalid or unsupported. */
int64_t tbn_space_to_depth_elems(int64_t N, int64_t C, int64_t H, int64_t W, int64_t R,
                                 int64_t S, int64_t stride_h, int64_t stride_w, int64_t pad_h,
                                 int64_t pad_w);
tbn_status tbn_space_to_depth(const void *x, tbn_dtype xdt, tbn_layout layout, int64_t N,
                              int64_t C, int64_t H, int64_t W, int64_t R, int64_t S,
                              int64_t stride_h, int64_t stride_w, int64_t pad_h, int64_t pad_w,
                              void *out, tbn_stream stream);

/* Algorithm 1's quantization loop fused with TwoBitForward in one launch
 * (Eq. 3, Eq. 5, Eq. 1): the CTAs of the implicit GEMM first quantize the
 * fp32 filters Wf [K][C*R*S] (in (r, s, c) order) into codes and alpha,
 * bitwise as tbn_quantize_pack writes them, meet at a grid-wide barrier (a
 * cooperative launch), then convolve as tbn_conv2d_fwd does with those
 * codes.  codes [K][tbn_packed_words(C*R*S)] and alpha [K] are outputs.
 * Takes the implicit GEMM's TMA activation shapes: NHWC bf16 x with
 * C % 32 == 0 and strides <= 2, C*R*S <= 32768 (else TBN_ERR_UNSUPPORTED).
 * Wf 4-byte aligned (16-byte aligned with C*R*S % 4 == 0 for vector loads).
 * workspace: at least 4 bytes, 4-byte aligned, zeroed by the call (a barrier
 * word: calls that may run concurrently must not share it).  Wf, codes and
 * alpha must not overlap.  The launch uses one CTA per SM and needs the
 * whole GPU (a cooperative launch: it fails with TBN_ERR_CUDA if the CTAs
 * cannot all be resident); a barrier that runs out of time sets
 * the timeout bit of the device error word.  It is launched plainly (not as
 * a programmatic dependent): it starts after the previous kernel on the
 * stream has completed, so Wf may be that kernel's output.  On this GPU it
 * is a few microseconds slower than tbn_quantize_pack + tbn_conv2d_fwd. */
tbn_status tbn_conv2d_fwd_quant(const void *x, tbn_dtype xdt, tbn_layout layout, int64_t N,
                                int64_t C, int64_t H, int64_t W, const float *Wf, int64_t K,
                                int64_t R, int64_t S, int64_t stride_h, int64_t stride_w,
                                int64_t pad_h, int64_t pad_w, uint32_t *codes, float *alpha,
                                void *y, tbn_dtype ydt, const tbn_epilogue *epi, void *workspace,
                                size_t workspace_bytes, tbn_stream stream);

/* tbn_conv2d_fwd with an explicit algorithm.  Returns TBN_ERR_UNSUPPORTED if
 * the requested algorithm cannot run this shape. */
tbn_status tbn_conv2d_fwd_algo(const void *x, tbn_dtype xdt, tbn_layout layout, int64_t N,
                               int64_t C, int64_t H, int64_t W, const uint32_t *codes,
                               const float *alpha, int64_t K, int64_t R, int64_t S,
                               int64_t stride_h, int64_t stride_w, int64_t pad_h,
                               int64_t pad_w, void *y, tbn_dtype ydt, const tbn_epilogue *epi,
                               tbn_conv_algo algo, tbn_stream stream);

/* The algorithm AUTO would choose for this shape (host-only query). */
tbn_conv_algo tbn_conv2d_select_algo(tbn_dtype xdt, tbn_layout layout, int64_t N, int64_t C,
                                     int64_t H, int64_t W, int64_t K, int64_t R, int64_t S,
                                     int64_t stride_h, int64_t stride_w, int64_t pad_h,
                                     int64_t pad_w);

/* TwoBitBackward (Algorithm 1) through one convolution of Eq. 1, whose
 * filters are the approximate filters W^ = alpha[k] W~[k] (the backward pass
 * uses them, not the real-valued weights).  Shapes as tbn_conv2d_fwd in NHWC:
 * x [N][H][W][C], dy = dC/dy [N][P][Q][K], codes [K][tbn_packed_words(R S C)]
 * in (r, s, c) order; pad_h <= R - 1 and pad_w <= S - 1 (else
 * TBN_ERR_UNSUPPORTED).  Both calls are asynchronous on `stream`, need a
 * caller workspace (256-byte aligned, contents on entry irrelevant; calls
 * that may run concurrently must not share one) and are bitwise
 * reproducible.
 *
 * Input gradient: dx[n,h,w,c] = sum over (k, p, q, r, s) with
 * p sh - pad_h + r = h and q sw - pad_w + s = w of dy[n,p,q,k] alpha[k]
 * W~[k,r,s,c], written to dx [N][H][W][C] (bf16 or fp32).  It runs as a
 * stride-1 convolution (this library's forward kernels) of
 * bf16(alpha[k] dy) dilated by the stride with the filters transposed and
 * mirrored; rounding alpha dy to bf16 adds at most 2^-9 relative per term
 * to the fp32 accumulation. */
size_t tbn_conv2d_bwd_data_workspace_bytes(int64_t N, int64_t C, int64_t H, int64_t W, int64_t K,
                                           int64_t R, int64_t S, int64_t stride_h,
                                           int64_t stride_w, int64_t pad_h, int64_t pad_w);
tbn_status tbn_conv2d_bwd_data(const void *dy, int64_t N, int64_t C, int64_t H, int64_t W,
                               const uint32_t *codes, const float *alpha, int64_t K, int64_t R,
                               int64_t S, int64_t stride_h, int64_t stride_w, int64_t pad_h,
                               int64_t pad_w, void *dx, tbn_dtype dxdt, void *workspace,
                               size_t workspace_bytes, tbn_stream stream);

/* Filter gradient: dW^[k,r,s,c] = sum over (n, p, q) of dy[n,p,q,k] *
 * x[n, p sh - pad_h + r, q sw - pad_w + s, c] (zero outside the image),
 * fp32 [K][R][S][C] (the codes' order), fp32 accumulation of exact bf16
 * products; Algorithm 1 applies it to the real-valued weights. */
size_t tbn_conv2d_bwd_filter_workspace_bytes(int64_t N, int64_t C, int64_t H, int64_t W,
                                             int64_t K, int64_t R, int64_t S, int64_t stride_h,
                                             int64_t stride_w, int64_t pad_h, int64_t pad_w);
tbn_status tbn_conv2d_bwd_filter(const void *x, const void *dy, int64_t N, int64_t C, int64_t H,
                                 int64_t W, int64_t K, int64_t R, int64_t S, int64_t stride_h,
                                 int64_t stride_w, int64_t pad_h, int64_t pad_w, float *dw,
                                 void *workspace, size_t workspace_bytes, tbn_stream stream);

/* Fully-connected layer (Section 3: treated as a convolution):
 *   y[b,k] = alpha[k] * sum_j x[b,j] W~[k,j]
 * x [B][K_in] (fp32 or bf16), codes [K_out][tbn_packed_words(K_in)],
 * alpha [K_out], y [B][K_out] (fp32 or bf16), optional epilogue (ReLU,
 * residual [B][K_out] of y's dtype; pool is invalid here).
 * Equivalent to tbn_linear_fwd_ws with no workspace: bf16 x with B <= 8,
 * K_in % 64 == 0 and 16-byte aligned x and codes runs the tensor-core GEMV;
 * fp32 x with B == 1 and K_in % 64 == 0 runs only on the table-lookup GEMV,
 * which needs no workspace for K_in <= 512 -- larger layers return
 * TBN_ERR_UNSUPPORTED here (use tbn_linear_fwd_ws or tbn_linear_fwd_noalloc);
 * every other shape runs as a 1x1 convolution (tensor cores for bf16 x). */
tbn_status tbn_linear_fwd(const void *x, tbn_dtype xdt, int64_t B, int64_t K_in,
                          const uint32_t *codes, const float *alpha, int64_t K_out, void *y,
                          tbn_dtype ydt, const tbn_epilogue *epi, tbn_stream stream);

/* Device scratch bytes tbn_linear_fwd_ws needs to run this shape on the
 * table-lookup GEMV (host-only query): 0 when that kernel does not apply
 * (it takes fp32 x, B == 1, K_in % 64 == 0) or needs no scratch
 * (K_in <= 512); otherwise 4 * ceil(K_in / 512) * 128 * ceil(K_out / 128)
 * bytes rounded up to 256. */
size_t tbn_linear_workspace_bytes(tbn_dtype xdt, int64_t B, int64_t K_in, int64_t K_out);

/* tbn_linear_fwd with caller-owned device scratch.  When x is fp32, B == 1,
 * K_in % 64 == 0, codes are 16-byte aligned and workspace_bytes >=
 * tbn_linear_workspace_bytes(...), the layer runs on the table-lookup GEMV:
 * for every group of four inputs the kernel tabulates the 256 possible sums
 * of the four two-bit weights times those inputs (fp32, products exact),
 * and each packed code word costs four table lookups.  The fp32 partial sum
 * of every row over each chunk of 512 inputs goes to `workspace` (256-byte
 * aligned, contents on entry irrelevant), and a second kernel on `stream`
 * adds them in chunk order, so results are bitwise reproducible.  Calls
 * that may run concurrently must not share a workspace.  Otherwise the call
 * behaves as tbn_linear_fwd and does not touch `workspace` (NULL allowed);
 * a batch-1 fp32 layer of the table kernel's shape with a smaller workspace
 * returns TBN_ERR_UNSUPPORTED (16-byte misaligned codes: TBN_ERR_MISALIGNED). */
tbn_status tbn_linear_fwd_ws(const void *x, tbn_dtype xdt, int64_t B, int64_t K_in,
                             const uint32_t *codes, const float *alpha, int64_t K_out, void *y,
                             tbn_dtype ydt, const tbn_epilogue *epi, void *workspace,
                             size_t workspace_bytes, tbn_stream stream);

/* tbn_linear_fwd_ws for callers that cannot allocate device memory (the
 * paper has no counterpart; this is a deployment variant of the same
 * computation).  It runs only the table-lookup GEMV (fp32 x, B == 1,
 * K_in % 64 == 0, 16-byte aligned codes; otherwise TBN_ERR_UNSUPPORTED) and
 * keeps its chunk partial sums in a 4 MiB array inside the library's own
 * device module instead of a caller's workspace: layers needing more,
 * tbn_linear_workspace_bytes(...) > 4 MiB (e.g. more than 32768 outputs at
 * 16384 inputs), return TBN_ERR_UNSUPPORTED before launching.  Nothing in
 * the array needs clearing between calls.  There is one array per device
 * and process: calls that could run concurrently (other streams, other
 * host threads) race on it and must be serialized by the caller.  The
 * first call on each device resolves the array's address
 * (cudaGetSymbolAddress); make it before any stream capture.  Results are
 * bitwise equal to tbn_linear_fwd_ws's. */
tbn_status tbn_linear_fwd_noalloc(const void *x, tbn_dtype xdt, int64_t B, int64_t K_in,
                                  const uint32_t *codes, const float *alpha, int64_t K_out,
                                  void *y, tbn_dtype ydt, const tbn_epilogue *epi,
                                  tbn_stream stream);

/* Max pooling over NHWC (network glue): window kh x kw, stride sh x sw,
 * padding ph x pw (taps in the padding are skipped, i.e. -infinity padding;
 * ph < kh and pw < kw); x [N][H][W][C] -> y [N][Ho][Wo][C],
 * Ho = (H + 2 ph - kh)/sh + 1, Wo = (W + 2 pw - kw)/sw + 1. */
tbn_status tbn_maxpool2d_nhwc(const void *x, tbn_dtype dt, int64_t N, int64_t H, int64_t W,
                              int64_t C, int64_t kh, int64_t kw, int64_t sh, int64_t sw,
                              int64_t ph, int64_t pw, void *y, tbn_stream stream);

/* Layout conversion NCHW -> NHWC with channel zero-padding to C_pad >= C
 * (network glue for the first layer).  x [N][C][H][W], y [N][H][W][C_pad],
 * same dtype. */
tbn_status tbn_nchw_to_nhwc(const void *x, tbn_dtype dt, int64_t N, int64_t C, int64_t H,
                            int64_t W, int64_t C_pad, void *y, tbn_stream stream);

/* ---- full-precision layers (network glue, not the paper's method) -------
 * Two-bit networks keep their first convolution and last fully-connected
 * layer in full precision (the ResNet-18 workload).  These calls compute
 * them on the CUDA cores in fp32: products x * w rounded to fp32 and added
 * in fp32. */

/* Dense convolution with fp32 weights w [K][C][R][S] (PyTorch order, any
 * activation layout): y = x cross-correlated with w, zero padding, no bias,
 * optional ReLU (relu != 0).  layout NCHW: x [N][C][H][W] -> y [N][K][P][Q];
 * NCHW_NHWC: x [N][C][H][W] -> y [N][P][Q][K]; NHWC: x [N][H][W][C] ->
 * y [N][P][Q][K].  x and y fp32 or bf16; w 4-byte aligned. */
tbn_status tbn_dense_conv2d_fwd(const void *x, tbn_dtype xdt, tbn_layout layout, int64_t N,
                                int64_t C, int64_t H, int64_t W, const float *w, int64_t K,
                                int64_t R, int64_t S, int64_t stride_h, int64_t stride_w,
                                int64_t pad_h, int64_t pad_w, void *y, tbn_dtype ydt, int relu,
                                tbn_stream stream);

/* Global average pool: x [N][H][W][C] -> y [N][C], y[b,c] = the fp32 mean of
 * x[b,:,:,c] (pixels added in order, times 1/(H W)). */
tbn_status tbn_avgpool2d_global_nhwc(const void *x, tbn_dtype xdt, int64_t N, int64_t H,
                                     int64_t W, int64_t C, void *y, tbn_dtype ydt,
                                     tbn_stream stream);

/* Dense fully-connected layer with fp32 weights: x [B][K_in] fp32,
 * w [K_out][K_in] fp32, y [B][K_out] (fp32 or bf16) = x w^T, optional ReLU. */
tbn_status tbn_dense_linear_fwd(const float *x, int64_t B, int64_t K_in, const float *w,
                                int64_t K_out, void *y, tbn_dtype ydt, int relu,
                                tbn_stream stream);

#ifdef __cplusplus
}
#endif

#endif /* TBN_H */
