// tbn_internal.h -- host-side declarations shared by the library's
// translation units: error reporting, argument helpers and the launchers
// each kernel file provides.  Not part of the public ABI (include/tbn.h).
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

#include "tbn.h"

namespace tbn {

// Record a failure detail for tbn_last_error() and return `s`.
tbn_status fail(tbn_status s, const char* fmt, ...);
const char* last_error_text();

// Map a failed CUDA call to TBN_ERR_CUDA with its message.
tbn_status cuda_fail(cudaError_t e, const char* what);

// cudaGetLastError() after a launch.
tbn_status check_launch(const char* what);

// Device address of the current device's error word (set up once per
// device); nullptr if it could not be resolved.
uint32_t* device_error_word();

// Multiprocessor count of the current device (cached per device).
int device_sm_count();

// cuTensorMapEncodeTiled resolved through the runtime's driver entry point
// (no link against libcuda); nullptr if unavailable.
using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                   const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                   const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn get_encode_tiled();

inline bool is_aligned(const void* p, size_t a) {
  return (reinterpret_cast<uintptr_t>(p) % a) == 0;
}

inline cudaStream_t as_stream(tbn_stream s) { return reinterpret_cast<cudaStream_t>(s); }

inline size_t dtype_size(tbn_dtype d) { return d == TBN_BF16 ? 2 : 4; }

// One convolution problem after validation.
struct ConvProblem {
  int64_t N, C, H, W, K, R, S, sh, sw, ph, pw, P, Q;
  tbn_layout layout;
  tbn_dtype xdt, ydt;
  const void* x;
  const uint32_t* codes;
  const float* alpha;
  void* y;
  int relu;
  const void* residual;
  int pool;  // 0 or 2 (2x2 max pool, stride 2, after ReLU)
  // split K (implicit GEMM only; set by tbn_linear_fwd_ws): ksplit > 1 K
  // ranges accumulate into fp32 `partial` [ksplit][N][P][Q][K], then a
  // second kernel adds them in order and applies the epilogue
  float* partial;
  int ksplit;
  // fused quantization (implicit GEMM only; set by tbn_conv2d_fwd_quant):
  // fp32 filters [K][C*R*S] quantized into codes and alpha by the same
  // launch; gbar is a 4-byte barrier word the launcher zeroes
  const float* wq;
  unsigned* gbar;
};

// Space-to-depth form of a strided convolution with few input channels
// (layout TBN_S2D_NHWC): with s = stride, R' = ceil(R / s), S' = ceil(S / s),
// the input becomes xs [N][Hs][Ws][64] bf16, Hs = P + R' - 1, Ws = Q + S' - 1,
//   xs[n][Y][X][(dy s + dx) C + c] = x[n][c][s Y + dy - ph][s X + dx - pw]
// (zero outside the image and for channels >= s^2 C), and the convolution
// becomes a stride-1 R' x S' convolution of xs whose weight for s2d channel
// (dy, dx, c) of tap (r', s') is W~[k][s r' + dy][s s' + dx][c] (zero where
// that reaches past the filter).
struct S2dGeom {
  int64_t s, Rp, Sp, Hs, Ws;
};
constexpr int64_t kS2dChannels = 64;
inline S2dGeom s2d_geom(int64_t R, int64_t S, int64_t stride, int64_t P, int64_t Q) {
  S2dGeom g;
  g.s = stride;
  g.Rp = (R + stride - 1) / stride;
  g.Sp = (S + stride - 1) / stride;
  g.Hs = P + g.Rp - 1;
  g.Ws = Q + g.Sp - 1;
  return g;
}

// The shape of one convolution for its backward pass (NHWC bf16).
struct BwdConvShape {
  int64_t N, C, H, W, K, R, S, sh, sw, ph, pw, P, Q;
};

// AUTO algorithm dispatch of tbn_conv2d_fwd for an already validated problem.
tbn_status run_conv_auto(const ConvProblem& p, cudaStream_t s);

// ---- launchers (each defined next to its kernels) ----
tbn_status launch_quantize_group(const tbn_quant_job* jobs, int njobs, cudaStream_t s);
tbn_status launch_unpack(const uint32_t* codes, const float* alpha, int64_t K, int64_t n,
                         void* out, tbn_unpack_format fmt, cudaStream_t s);

tbn_status launch_conv_direct(const ConvProblem& p, cudaStream_t s);

// Empty string when the implicit-GEMM kernel can run `p`, else the reason.
const char* conv_igemm_unsupported_reason(const ConvProblem& p);
tbn_status launch_conv_igemm(const ConvProblem& p, cudaStream_t s);
// Space-to-depth layout change of a bf16 NCHW or NHWC input for the
// convolution geometry (C, H, W, R, S, stride, pad) (see S2dGeom).
tbn_status launch_space_to_depth(const void* x, tbn_layout layout, int64_t N, int64_t C,
                                 int64_t H, int64_t W, const S2dGeom& g, int64_t ph, int64_t pw,
                                 void* out, cudaStream_t s);
// Split-K plan of the implicit GEMM for `p` (a layer whose output tiles
// leave most SMs idle, e.g. a fully-connected layer at batch 256): the number
// of K ranges (1 = no split) and the fp32 workspace bytes it needs.
int conv_igemm_splitk(const ConvProblem& p, size_t* workspace_bytes);
// True when the implicit-GEMM kernel would feed activations by TMA (its fast mode).
bool conv_igemm_uses_tma(const ConvProblem& p);

const char* conv_smalltap_unsupported_reason(const ConvProblem& p);
tbn_status launch_conv_smalltap(const ConvProblem& p, cudaStream_t s);

const char* gemv_unsupported_reason(const void* x, tbn_dtype xdt, int64_t B, int64_t K_in,
                                    const uint32_t* codes);
tbn_status launch_gemv(const void* x, int64_t B, int64_t K_in, const uint32_t* codes,
                       const float* alpha, int64_t K_out, void* y, tbn_dtype ydt, int relu,
                       const void* residual, cudaStream_t s);

// Batch-1 table-lookup GEMV for fp32 activations (tbn_gemv_lut.cu).
const char* gemv_lut_shape_reason(tbn_dtype xdt, int64_t B, int64_t K_in, int64_t K_out);
const char* gemv_lut_unsupported_reason(tbn_dtype xdt, int64_t B, int64_t K_in, int64_t K_out,
                                        const uint32_t* codes);
size_t gemv_lut_workspace_bytes(int64_t K_in, int64_t K_out);
// batch-1 fp8 tensor-core GEMV (csrc/tbn_gemv_f8.cu) on codes in the
// e4m3-planar layout written by launch_prepare_f8
const char* gemv_f8_unsupported_reason(int64_t B, int64_t K_in, int64_t K_out);
size_t gemv_f8_workspace_bytes(int64_t K_in, int64_t K_out);
int64_t gemv_f8_prepared_words(int64_t K_out, int64_t K_in);
tbn_status launch_prepare_f8(const uint32_t* codes, int64_t K_out, int64_t K_in, uint32_t* out,
                             cudaStream_t s);
tbn_status launch_gemv_f8(const void* x, int64_t K_in, const uint32_t* prepared, const float* alpha,
                          int64_t K_out, void* y, tbn_dtype ydt, const void* residual, int relu,
                          void* workspace, size_t workspace_bytes, cudaStream_t s);
tbn_status launch_gemv_lut(const void* x, int64_t K_in, const uint32_t* codes,
                           const float* alpha, int64_t K_out, void* y, tbn_dtype ydt, int relu,
                           const void* residual, void* workspace, size_t workspace_bytes,
                           cudaStream_t s);

// The table GEMV with its scratch in a file-scope device array.
size_t gemv_lut_static_scratch_bytes();
tbn_status launch_gemv_lut_static(const void* x, int64_t K_in, const uint32_t* codes,
                                  const float* alpha, int64_t K_out, void* y, tbn_dtype ydt,
                                  int relu, const void* residual, cudaStream_t s);

// Algorithm 1 TwoBitBackward through a convolution (tbn_conv_bwd.cu).
const char* bwd_shape_reason(const BwdConvShape& p);
size_t bwd_data_workspace_bytes(const BwdConvShape& p);
tbn_status launch_bwd_data(const BwdConvShape& p, const void* dy, const uint32_t* codes,
                           const float* alpha, void* dx, tbn_dtype dxdt, void* workspace,
                           cudaStream_t s);
size_t bwd_filter_workspace_bytes(const BwdConvShape& p);
tbn_status launch_bwd_filter(const BwdConvShape& p, const void* x, const void* dy, float* dw,
                             void* workspace, cudaStream_t s);

tbn_status launch_maxpool_nhwc(const void* x, tbn_dtype dt, int64_t N, int64_t H, int64_t W,
                               int64_t C, int64_t kh, int64_t kw, int64_t sh, int64_t sw,
                               int64_t ph, int64_t pw, void* y, cudaStream_t s);

// Canonical <-> byte-planar code words (tbn_quantize.cu).
tbn_status launch_repack(const uint32_t* in, int64_t words, uint32_t* out, bool to_planar,
                         cudaStream_t s);

// Full-precision layers around the two-bit ones (tbn_dense.cu).
tbn_status launch_dense_conv(const ConvProblem& p, const float* w, cudaStream_t s);
tbn_status launch_avgpool_global_nhwc(const void* x, tbn_dtype xdt, int64_t N, int64_t H,
                                      int64_t W, int64_t C, void* y, tbn_dtype ydt,
                                      cudaStream_t s);
tbn_status launch_dense_linear(const float* x, int64_t B, int64_t K_in, const float* w,
                               int64_t K_out, void* y, tbn_dtype ydt, int relu,
                               cudaStream_t s);
tbn_status launch_nchw_to_nhwc(const void* x, tbn_dtype dt, int64_t N, int64_t C, int64_t H,
                               int64_t W, int64_t C_pad, void* y, cudaStream_t s);

}  // namespace tbn
