// tbn_api.cu -- the library's extern "C" entry points (include/tbn.h):
// argument validation on the host, dispatch to the kernels, error reporting.
#include <cuda_runtime.h>

#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>

#include "tbn.h"
#include "tbn_device.cuh"
#include "tbn_internal.h"

namespace tbn {

// Per-device error word written by kernels (timeouts, bad launch shapes).
__device__ uint32_t g_tbn_device_error;
// Where tbn_device_error's one-thread kernel leaves the word it took.
__device__ uint32_t g_tbn_error_snapshot;

namespace {

thread_local char t_last_error[512] = "";

// One thread waits on a fresh mbarrier (phase 0 never completes: nothing
// arrives) through the library's bounded wait, which records the timeout in
// the error word after limit_ns and returns.
__global__ void selftest_wait_timeout_kernel(uint32_t* err, uint64_t limit_ns) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_mbar_init();
    mbar_wait(&bar, 0u, nullptr, err, limit_ns);
  }
}

// Reads and clears the error word in one atomic step, so that a bit a
// kernel of another stream sets meanwhile stays for the next read.
__global__ void take_error_kernel(uint32_t* err) {
  g_tbn_error_snapshot = atomicExch(err, 0u);
}

std::mutex g_error_read_mutex;   // one reader of the snapshot slot at a time

constexpr int kMaxDevices = 64;
uint32_t* g_err_ptr[kMaxDevices] = {};
int g_sm_count[kMaxDevices] = {};
std::mutex g_dev_mutex;

bool mul_ok(int64_t a, int64_t b, int64_t limit) {
  return a >= 0 && b >= 0 && (a == 0 || b <= limit / a);
}

}  // namespace

const char* last_error_text() { return t_last_error; }

tbn_status fail(tbn_status s, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  std::vsnprintf(t_last_error, sizeof(t_last_error), fmt, ap);
  va_end(ap);
  return s;
}

tbn_status cuda_fail(cudaError_t e, const char* what) {
  return fail(TBN_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

tbn_status check_launch(const char* what) {
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, what);
  return TBN_OK;
}

EncodeTiledFn get_encode_tiled() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

uint32_t* device_error_word() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> g(g_dev_mutex);
  if (g_err_ptr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_tbn_device_error) == cudaSuccess)
      g_err_ptr[dev] = static_cast<uint32_t*>(p);
  }
  return g_err_ptr[dev];
}

int device_sm_count() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return 132;
  std::lock_guard<std::mutex> g(g_dev_mutex);
  if (g_sm_count[dev] == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
      n = 132;
    g_sm_count[dev] = n;
  }
  return g_sm_count[dev];
}

}  // namespace tbn

using namespace tbn;

namespace {

tbn_status validate_conv(const void* x, tbn_dtype xdt, tbn_layout layout, int64_t N, int64_t C,
                         int64_t H, int64_t W, const uint32_t* codes, const float* alpha,
                         int64_t K, int64_t R, int64_t S, int64_t sh, int64_t sw, int64_t ph,
                         int64_t pw, void* y, tbn_dtype ydt, const tbn_epilogue* epi,
                         ConvProblem* out) {
  if (!x || !codes || !alpha || !y) return fail(TBN_ERR_INVALID_ARG, "conv: null pointer");
  if (xdt != TBN_F32 && xdt != TBN_BF16) return fail(TBN_ERR_INVALID_ARG, "conv: bad x dtype");
  if (ydt != TBN_F32 && ydt != TBN_BF16) return fail(TBN_ERR_INVALID_ARG, "conv: bad y dtype");
  if (layout != TBN_NCHW && layout != TBN_NHWC && layout != TBN_NCHW_NHWC &&
      layout != TBN_S2D_NHWC)
    return fail(TBN_ERR_INVALID_ARG, "conv: bad layout");
  if (N < 1 || C < 1 || H < 1 || W < 1 || K < 1 || R < 1 || S < 1)
    return fail(TBN_ERR_INVALID_ARG, "conv: sizes must be >= 1");
  if (sh < 1 || sw < 1 || ph < 0 || pw < 0) return fail(TBN_ERR_INVALID_ARG, "conv: bad stride/pad");
  // bounds first, so that no sum or product below can overflow
  const int64_t lim31 = int64_t(1) << 31;
  if (N >= lim31 || C >= lim31 || H >= lim31 || W >= lim31 || K >= lim31)
    return fail(TBN_ERR_UNSUPPORTED, "conv: a size is 2^31 or more");
  if (R > 0xFFFF || S > 0xFFFF || sh > 0xFFFF || sw > 0xFFFF || ph > 0xFFFF || pw > 0xFFFF)
    return fail(TBN_ERR_UNSUPPORTED, "conv: kernel/stride/pad above 65535");
  if (H + 2 * ph < R || W + 2 * pw < S)
    return fail(TBN_ERR_INVALID_ARG, "conv: kernel larger than padded input");
  const int64_t lim = int64_t(1) << 31;
  if (!mul_ok(C * R, S, lim) || !mul_ok(C, H * W, lim) || H * W >= lim)
    return fail(TBN_ERR_UNSUPPORTED, "conv: C*R*S or C*H*W exceeds 2^31");
  const int64_t P = (H + 2 * ph - R) / sh + 1, Q = (W + 2 * pw - S) / sw + 1;
  const int64_t lim46 = int64_t(1) << 46;
  if (!mul_ok(N, H * W * C, lim46) || !mul_ok(N, P, lim46) || !mul_ok(N * P, Q, lim46) ||
      !mul_ok(N * P * Q, K, lim46))
    return fail(TBN_ERR_UNSUPPORTED, "conv: tensor too large");
  const size_t xs = dtype_size(xdt), ys = dtype_size(ydt);
  if (!is_aligned(x, xs) || !is_aligned(y, ys) || !is_aligned(codes, 4) || !is_aligned(alpha, 4))
    return fail(TBN_ERR_MISALIGNED, "conv: pointer not aligned to its element size");
  if (epi && epi->residual && !is_aligned(epi->residual, ys))
    return fail(TBN_ERR_MISALIGNED, "conv: residual not aligned to its element size");
  const int pool = epi ? epi->pool : 0;
  if (pool != 0 && pool != 2) return fail(TBN_ERR_INVALID_ARG, "conv: pool must be 0 or 2");
  if (pool && (P < 2 || Q < 2)) return fail(TBN_ERR_INVALID_ARG, "conv: pool needs P, Q >= 2");
  if (pool && epi->residual)
    return fail(TBN_ERR_UNSUPPORTED, "conv: pool cannot be combined with a residual");
  ConvProblem& p = *out;
  p.N = N; p.C = C; p.H = H; p.W = W; p.K = K; p.R = R; p.S = S;
  p.sh = sh; p.sw = sw; p.ph = ph; p.pw = pw; p.P = P; p.Q = Q;
  p.layout = layout; p.xdt = xdt; p.ydt = ydt;
  p.x = x; p.codes = codes; p.alpha = alpha; p.y = y;
  p.relu = epi ? (epi->relu != 0) : 0;
  p.residual = epi ? epi->residual : nullptr;
  p.pool = pool;
  return TBN_OK;
}

// AUTO: the implicit GEMM when it can feed activations by TMA, else the
// small-tap kernel for short filters, else the implicit GEMM with gathered
// activations, else the CUDA-core direct kernel.
tbn_conv_algo pick_algo(const ConvProblem& p) {
  if (p.layout == TBN_S2D_NHWC) return TBN_CONV_IMPLICIT_GEMM;   // its only kernel
  const bool igemm = conv_igemm_unsupported_reason(p)[0] == '\0';
  if (igemm && conv_igemm_uses_tma(p)) return TBN_CONV_IMPLICIT_GEMM;
  if (conv_smalltap_unsupported_reason(p)[0] == '\0') return TBN_CONV_SMALL_TAPS;
  if (igemm) return TBN_CONV_IMPLICIT_GEMM;
  return TBN_CONV_DIRECT;
}

tbn_status run_conv(const ConvProblem& p, tbn_conv_algo algo, cudaStream_t s) {
  if (algo == TBN_CONV_AUTO) algo = pick_algo(p);
  if (p.layout == TBN_S2D_NHWC && algo != TBN_CONV_IMPLICIT_GEMM) {
    if (algo != TBN_CONV_SMALL_TAPS && algo != TBN_CONV_DIRECT)
      return fail(TBN_ERR_INVALID_ARG, "conv: bad algorithm %d", (int)algo);
    return fail(TBN_ERR_UNSUPPORTED, "conv: space-to-depth input runs on the implicit GEMM only");
  }
  if (algo == TBN_CONV_SMALL_TAPS) {
    const char* why = conv_smalltap_unsupported_reason(p);
    if (why[0] != '\0') return fail(TBN_ERR_UNSUPPORTED, "%s", why);
    return launch_conv_smalltap(p, s);
  }
  if (algo == TBN_CONV_IMPLICIT_GEMM) {
    const char* why = conv_igemm_unsupported_reason(p);
    if (why[0] != '\0') return fail(TBN_ERR_UNSUPPORTED, "%s", why);
    return launch_conv_igemm(p, s);
  }
  if (algo == TBN_CONV_DIRECT) return launch_conv_direct(p, s);
  return fail(TBN_ERR_INVALID_ARG, "conv: bad algorithm %d", (int)algo);
}

// Geometry checks of the space-to-depth layout change (shared by the size
// query and the call).
tbn_status validate_s2d(int64_t N, int64_t C, int64_t H, int64_t W, int64_t R, int64_t S,
                        int64_t sh, int64_t sw, int64_t ph, int64_t pw, S2dGeom* g) {
  if (N < 1 || C < 1 || H < 1 || W < 1 || R < 1 || S < 1 || ph < 0 || pw < 0)
    return fail(TBN_ERR_INVALID_ARG, "space_to_depth: bad sizes");
  if (sh != sw || sh < 2)
    return fail(TBN_ERR_UNSUPPORTED, "space_to_depth: needs equal strides >= 2");
  if (sh > 8 || sh * sh * C > kS2dChannels)
    return fail(TBN_ERR_UNSUPPORTED, "space_to_depth: needs stride^2 * C <= 64");
  const int64_t lim = int64_t(1) << 31;
  if (H >= lim || W >= lim || R > 0xFFFF || S > 0xFFFF || ph > 0xFFFF || pw > 0xFFFF)
    return fail(TBN_ERR_UNSUPPORTED, "space_to_depth: a size is too large");
  if (H + 2 * ph < R || W + 2 * pw < S)
    return fail(TBN_ERR_INVALID_ARG, "space_to_depth: kernel larger than padded input");
  const int64_t P = (H + 2 * ph - R) / sh + 1, Q = (W + 2 * pw - S) / sw + 1;
  *g = s2d_geom(R, S, sh, P, Q);
  if (N > 65535 || g->Hs > 65535 || !mul_ok(N, g->Hs * g->Ws, int64_t(1) << 40) ||
      !mul_ok(N, H * W * C, int64_t(1) << 46))
    return fail(TBN_ERR_UNSUPPORTED, "space_to_depth: tensor too large");
  return TBN_OK;
}

}  // namespace

namespace tbn {
tbn_status run_conv_auto(const ConvProblem& p, cudaStream_t s) {
  return run_conv(p, TBN_CONV_AUTO, s);
}
}  // namespace tbn

extern "C" {

int tbn_abi_version(void) { return TBN_ABI_VERSION; }

int64_t tbn_packed_words(int64_t n) { return n < 1 ? -1 : (n + 15) / 16; }

const char* tbn_status_string(tbn_status s) {
  switch (s) {
    case TBN_OK: return "ok";
    case TBN_ERR_INVALID_ARG: return "invalid argument";
    case TBN_ERR_UNSUPPORTED: return "unsupported";
    case TBN_ERR_MISALIGNED: return "misaligned pointer";
    case TBN_ERR_CUDA: return "CUDA error";
    case TBN_ERR_TIMEOUT: return "device wait timed out";
  }
  return "unknown status";
}

const char* tbn_last_error(void) { return last_error_text(); }

tbn_status tbn_device_error(uint32_t* flags) {
  if (!flags) return fail(TBN_ERR_INVALID_ARG, "device_error: null pointer");
  *flags = 0;
  uint32_t* p = device_error_word();
  if (!p) return fail(TBN_ERR_CUDA, "device_error: cannot resolve the error word");
  std::lock_guard<std::mutex> g(g_error_read_mutex);
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return cuda_fail(e, "device_error: synchronize");
  take_error_kernel<<<1, 1>>>(p);
  e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "device_error: launch");
  uint32_t v = 0;
  e = cudaMemcpyFromSymbol(&v, g_tbn_error_snapshot, sizeof(v));   // synchronous, after the kernel
  if (e != cudaSuccess) return cuda_fail(e, "device_error: read");
  *flags = v;
  return TBN_OK;
}

tbn_status tbn_selftest_wait_timeout(uint32_t limit_us, tbn_stream stream) {
  if (limit_us < 1 || limit_us > 1000000)
    return fail(TBN_ERR_INVALID_ARG, "selftest_wait_timeout: limit must be 1 .. 1000000 us");
  uint32_t* err = device_error_word();
  if (!err) return fail(TBN_ERR_CUDA, "selftest_wait_timeout: cannot resolve the error word");
  selftest_wait_timeout_kernel<<<1, 32, 0, as_stream(stream)>>>(err,
                                                                uint64_t(limit_us) * 1000u);
  return check_launch("selftest_wait_timeout_kernel");
}

tbn_status tbn_quantize_pack_group(const tbn_quant_job* jobs, int njobs, tbn_stream stream) {
  if (!jobs || njobs < 1 || njobs > TBN_MAX_QUANT_JOBS)
    return fail(TBN_ERR_INVALID_ARG, "quantize: need 1..%d jobs", TBN_MAX_QUANT_JOBS);
  for (int i = 0; i < njobs; ++i) {
    const tbn_quant_job& j = jobs[i];
    if (!j.W || !j.codes || !j.alpha) return fail(TBN_ERR_INVALID_ARG, "quantize: job %d null pointer", i);
    if (j.K < 1 || j.n < 1) return fail(TBN_ERR_INVALID_ARG, "quantize: job %d needs K, n >= 1", i);
    if (j.n >= (int64_t(1) << 31)) return fail(TBN_ERR_UNSUPPORTED, "quantize: job %d n >= 2^31", i);
    if (!mul_ok(j.K, (j.n + 15) / 16, int64_t(1) << 40) || !mul_ok(j.K, j.n, int64_t(1) << 44))
      return fail(TBN_ERR_UNSUPPORTED, "quantize: job %d too large", i);
    if (!is_aligned(j.W, 4) || !is_aligned(j.codes, 4) || !is_aligned(j.alpha, 4))
      return fail(TBN_ERR_MISALIGNED, "quantize: job %d pointers must be 4-byte aligned", i);
  }
  return launch_quantize_group(jobs, njobs, as_stream(stream));
}

tbn_status tbn_quantize_pack(const float* W, int64_t K, int64_t n, uint32_t* codes, float* alpha,
                             tbn_stream stream) {
  tbn_quant_job j{W, K, n, codes, alpha};
  return tbn_quantize_pack_group(&j, 1, stream);
}

tbn_status tbn_unpack(const uint32_t* codes, const float* alpha, int64_t K, int64_t n, void* out,
                      tbn_unpack_format fmt, tbn_stream stream) {
  if (!codes || !out) return fail(TBN_ERR_INVALID_ARG, "unpack: null pointer");
  if (fmt != TBN_UNPACK_I8 && fmt != TBN_UNPACK_F32 && fmt != TBN_UNPACK_BF16)
    return fail(TBN_ERR_INVALID_ARG, "unpack: bad format");
  if (fmt != TBN_UNPACK_I8 && !alpha) return fail(TBN_ERR_INVALID_ARG, "unpack: alpha required");
  if (K < 1 || n < 1) return fail(TBN_ERR_INVALID_ARG, "unpack: K, n must be >= 1");
  if (!mul_ok(K, n, int64_t(1) << 44)) return fail(TBN_ERR_UNSUPPORTED, "unpack: too large");
  const size_t es = fmt == TBN_UNPACK_I8 ? 1 : (fmt == TBN_UNPACK_F32 ? 4 : 2);
  if (!is_aligned(codes, 4) || !is_aligned(out, es) || (alpha && !is_aligned(alpha, 4)))
    return fail(TBN_ERR_MISALIGNED, "unpack: misaligned pointer");
  return launch_unpack(codes, alpha, K, n, out, fmt, as_stream(stream));
}

tbn_status tbn_conv2d_fwd_algo(const void* x, tbn_dtype xdt, tbn_layout layout, int64_t N,
                               int64_t C, int64_t H, int64_t W, const uint32_t* codes,
                               const float* alpha, int64_t K, int64_t R, int64_t S,
                               int64_t stride_h, int64_t stride_w, int64_t pad_h, int64_t pad_w,
                               void* y, tbn_dtype ydt, const tbn_epilogue* epi,
                               tbn_conv_algo algo, tbn_stream stream) {
  ConvProblem p{};
  const tbn_status st = validate_conv(x, xdt, layout, N, C, H, W, codes, alpha, K, R, S, stride_h,
                                      stride_w, pad_h, pad_w, y, ydt, epi, &p);
  if (st != TBN_OK) return st;
  return run_conv(p, algo, as_stream(stream));
}

tbn_status tbn_conv2d_fwd(const void* x, tbn_dtype xdt, tbn_layout layout, int64_t N, int64_t C,
                          int64_t H, int64_t W, const uint32_t* codes, const float* alpha,
                          int64_t K, int64_t R, int64_t S, int64_t stride_h, int64_t stride_w,
                          int64_t pad_h, int64_t pad_w, void* y, tbn_dtype ydt,
                          const tbn_epilogue* epi, tbn_stream stream) {
  return tbn_conv2d_fwd_algo(x, xdt, layout, N, C, H, W, codes, alpha, K, R, S, stride_h,
                             stride_w, pad_h, pad_w, y, ydt, epi, TBN_CONV_AUTO, stream);
}

tbn_status tbn_conv2d_fwd_quant(const void* x, tbn_dtype xdt, tbn_layout layout, int64_t N,
                                int64_t C, int64_t H, int64_t W, const float* Wf, int64_t K,
                                int64_t R, int64_t S, int64_t stride_h, int64_t stride_w,
                                int64_t pad_h, int64_t pad_w, uint32_t* codes, float* alpha,
                                void* y, tbn_dtype ydt, const tbn_epilogue* epi, void* workspace,
                                size_t workspace_bytes, tbn_stream stream) {
  if (!Wf) return fail(TBN_ERR_INVALID_ARG, "conv quant: null filters");
  ConvProblem p{};
  const tbn_status st = validate_conv(x, xdt, layout, N, C, H, W, codes, alpha, K, R, S, stride_h,
                                      stride_w, pad_h, pad_w, y, ydt, epi, &p);
  if (st != TBN_OK) return st;
  if (!workspace || workspace_bytes < 4) return fail(TBN_ERR_INVALID_ARG, "conv quant: workspace < 4 bytes");
  if (!is_aligned(Wf, 4) || !is_aligned(workspace, 4))
    return fail(TBN_ERR_MISALIGNED, "conv quant: filters and workspace need 4-byte alignment");
  if (layout == TBN_S2D_NHWC || C * R * S > 32768)
    return fail(TBN_ERR_UNSUPPORTED, "conv quant: needs C*R*S <= 32768 and no space-to-depth input");
  const int64_t nbytes = K * C * R * S * 4, cbytes = K * ((C * R * S + 15) / 16) * 4;
  const uintptr_t w0 = reinterpret_cast<uintptr_t>(Wf), c0 = reinterpret_cast<uintptr_t>(codes),
                  a0 = reinterpret_cast<uintptr_t>(alpha);
  if ((c0 < w0 + nbytes && w0 < c0 + cbytes) || (a0 < w0 + nbytes && w0 < a0 + K * 4) ||
      (a0 < c0 + cbytes && c0 < a0 + K * 4))
    return fail(TBN_ERR_INVALID_ARG, "conv quant: filters, codes and alpha must not overlap");
  p.wq = Wf;
  p.gbar = static_cast<unsigned*>(workspace);
  const char* why = conv_igemm_unsupported_reason(p);
  if (why[0] != '\0') return fail(TBN_ERR_UNSUPPORTED, "%s", why);
  return launch_conv_igemm(p, as_stream(stream));
}

int64_t tbn_space_to_depth_elems(int64_t N, int64_t C, int64_t H, int64_t W, int64_t R,
                                 int64_t S, int64_t stride_h, int64_t stride_w, int64_t pad_h,
                                 int64_t pad_w) {
  S2dGeom g{};
  if (validate_s2d(N, C, H, W, R, S, stride_h, stride_w, pad_h, pad_w, &g) != TBN_OK) return -1;
  return N * g.Hs * g.Ws * kS2dChannels;
}

tbn_status tbn_space_to_depth(const void* x, tbn_dtype xdt, tbn_layout layout, int64_t N,
                              int64_t C, int64_t H, int64_t W, int64_t R, int64_t S,
                              int64_t stride_h, int64_t stride_w, int64_t pad_h, int64_t pad_w,
                              void* out, tbn_stream stream) {
  if (!x || !out) return fail(TBN_ERR_INVALID_ARG, "space_to_depth: null pointer");
  if (xdt != TBN_BF16) return fail(TBN_ERR_UNSUPPORTED, "space_to_depth: x must be bf16");
  if (layout != TBN_NCHW && layout != TBN_NHWC)
    return fail(TBN_ERR_INVALID_ARG, "space_to_depth: x must be NCHW or NHWC");
  S2dGeom g{};
  const tbn_status st = validate_s2d(N, C, H, W, R, S, stride_h, stride_w, pad_h, pad_w, &g);
  if (st != TBN_OK) return st;
  if (!is_aligned(x, 2) || !is_aligned(out, 16))
    return fail(TBN_ERR_MISALIGNED, "space_to_depth: x needs 2-byte, out 16-byte alignment");
  const int64_t bytes = N * g.Hs * g.Ws * kS2dChannels * 2;
  const int64_t xbytes = N * C * H * W * 2;
  const uintptr_t a = reinterpret_cast<uintptr_t>(x), b = reinterpret_cast<uintptr_t>(out);
  if (a < b + static_cast<uintptr_t>(bytes) && b < a + static_cast<uintptr_t>(xbytes))
    return fail(TBN_ERR_INVALID_ARG, "space_to_depth: x and out overlap");
  return launch_space_to_depth(x, layout, N, C, H, W, g, pad_h, pad_w, out, as_stream(stream));
}

tbn_conv_algo tbn_conv2d_select_algo(tbn_dtype xdt, tbn_layout layout, int64_t N, int64_t C,
                                     int64_t H, int64_t W, int64_t K, int64_t R, int64_t S,
                                     int64_t stride_h, int64_t stride_w, int64_t pad_h,
                                     int64_t pad_w) {
  // Pointers only matter for alignment; use a 256-byte aligned dummy.
  static const uint32_t dummy[64] __attribute__((aligned(256))) = {};
  ConvProblem p{};
  const tbn_status st =
      validate_conv(dummy, xdt, layout, N, C, H, W, dummy, reinterpret_cast<const float*>(dummy),
                    K, R, S, stride_h, stride_w, pad_h, pad_w, const_cast<uint32_t*>(dummy), TBN_BF16,
                    nullptr, &p);
  if (st != TBN_OK) return TBN_CONV_DIRECT;
  return pick_algo(p);
}

}  // extern "C"

namespace {

// Host-side checks shared by the linear entry points.
tbn_status validate_linear(const void* x, tbn_dtype xdt, int64_t B, int64_t K_in,
                           const uint32_t* codes, const float* alpha, int64_t K_out, void* y,
                           tbn_dtype ydt, const tbn_epilogue* epi) {
  if (!x || !codes || !alpha || !y) return fail(TBN_ERR_INVALID_ARG, "linear: null pointer");
  if (xdt != TBN_F32 && xdt != TBN_BF16) return fail(TBN_ERR_INVALID_ARG, "linear: bad x dtype");
  if (ydt != TBN_F32 && ydt != TBN_BF16) return fail(TBN_ERR_INVALID_ARG, "linear: bad y dtype");
  if (B < 1 || K_in < 1 || K_out < 1) return fail(TBN_ERR_INVALID_ARG, "linear: sizes must be >= 1");
  if (B >= (int64_t(1) << 31) || K_in >= (int64_t(1) << 31) || K_out >= (int64_t(1) << 31))
    return fail(TBN_ERR_UNSUPPORTED, "linear: B / K_in / K_out >= 2^31");
  const size_t ys = dtype_size(ydt);
  if (!is_aligned(x, dtype_size(xdt)) || !is_aligned(y, ys) || !is_aligned(codes, 4) ||
      !is_aligned(alpha, 4) || (epi && epi->residual && !is_aligned(epi->residual, ys)))
    return fail(TBN_ERR_MISALIGNED, "linear: pointer not aligned to its element size");
  if (epi && epi->pool != 0) return fail(TBN_ERR_INVALID_ARG, "linear: pool is not defined");
  return TBN_OK;
}

// The 1x1-convolution form of a fully-connected layer (Section 3), with
// 256-byte aligned stand-in pointers for shape-only queries.
bool linear_as_conv(const void* x, tbn_dtype xdt, int64_t B, int64_t K_in, const uint32_t* codes,
                    const float* alpha, int64_t K_out, void* y, tbn_dtype ydt,
                    const tbn_epilogue* epi, ConvProblem* p) {
  return validate_conv(x, xdt, TBN_NHWC, B, K_in, 1, 1, codes, alpha, K_out, 1, 1, 1, 1, 0, 0, y,
                       ydt, epi, p) == TBN_OK;
}

bool linear_uses_table(tbn_dtype xdt, int64_t B, int64_t K_in, int64_t K_out,
                       const uint32_t* codes) {
  return gemv_lut_unsupported_reason(xdt, B, K_in, K_out, codes)[0] == '\0';
}

}  // namespace

extern "C" {

tbn_status tbn_linear_fwd(const void* x, tbn_dtype xdt, int64_t B, int64_t K_in,
                          const uint32_t* codes, const float* alpha, int64_t K_out, void* y,
                          tbn_dtype ydt, const tbn_epilogue* epi, tbn_stream stream) {
  return tbn_linear_fwd_ws(x, xdt, B, K_in, codes, alpha, K_out, y, ydt, epi, nullptr, 0, stream);
}

int64_t tbn_linear_f8_prepared_words(int64_t K_out, int64_t K_in) {
  if (K_out < 1 || K_in < 1 || K_in % 512 != 0 || K_in > (int64_t(1) << 30) ||
      K_out >= (int64_t(1) << 24))
    return -1;
  return gemv_f8_prepared_words(K_out, K_in);
}

tbn_status tbn_linear_prepare_f8(const uint32_t* codes, int64_t K_out, int64_t K_in,
                                 uint32_t* prepared, tbn_stream stream) {
  if (!codes || !prepared) return fail(TBN_ERR_INVALID_ARG, "prepare_f8: null pointer");
  if (K_out < 1 || K_in < 1) return fail(TBN_ERR_INVALID_ARG, "prepare_f8: sizes must be >= 1");
  const int64_t words = tbn_linear_f8_prepared_words(K_out, K_in);
  if (words < 0) return fail(TBN_ERR_UNSUPPORTED, "prepare_f8: K_in must be a multiple of 512");
  if (!is_aligned(codes, 4) || !is_aligned(prepared, 16))
    return fail(TBN_ERR_MISALIGNED, "prepare_f8: codes need 4-byte, prepared 16-byte alignment");
  const uintptr_t a = reinterpret_cast<uintptr_t>(codes), b = reinterpret_cast<uintptr_t>(prepared);
  const uintptr_t na = static_cast<uintptr_t>(K_out * (K_in / 16)) * 4;
  const uintptr_t nb = static_cast<uintptr_t>(words) * 4;
  if (a < b + nb && b < a + na) return fail(TBN_ERR_INVALID_ARG, "prepare_f8: codes and prepared overlap");
  return launch_prepare_f8(codes, K_out, K_in, prepared, as_stream(stream));
}

size_t tbn_linear_f8_workspace_bytes(int64_t B, int64_t K_in, int64_t K_out) {
  if (B != 1 || K_in < 1 || K_out < 1 || K_out >= (int64_t(1) << 24)) return 0;
  return gemv_f8_workspace_bytes(K_in, K_out);
}

tbn_status tbn_linear_fwd_f8(const void* x, tbn_dtype xdt, int64_t B, int64_t K_in,
                             const uint32_t* prepared, const float* alpha, int64_t K_out, void* y,
                             tbn_dtype ydt, const tbn_epilogue* epi, void* workspace,
                             size_t workspace_bytes, tbn_stream stream) {
  const tbn_status st = validate_linear(x, xdt, B, K_in, prepared, alpha, K_out, y, ydt, epi);
  if (st != TBN_OK) return st;
  if (xdt != TBN_BF16) return fail(TBN_ERR_UNSUPPORTED, "fp8 GEMV: x must be bf16");
  const char* why = gemv_f8_unsupported_reason(B, K_in, K_out);
  if (why[0] != '\0') return fail(TBN_ERR_UNSUPPORTED, "%s", why);
  if (!workspace) return fail(TBN_ERR_INVALID_ARG, "fp8 GEMV: null workspace");
  if (!is_aligned(x, 16) || !is_aligned(prepared, 16) || !is_aligned(workspace, 256))
    return fail(TBN_ERR_MISALIGNED,
                "fp8 GEMV: x and the codes need 16-byte, the workspace 256-byte alignment");
  if (workspace_bytes < gemv_f8_workspace_bytes(K_in, K_out))
    return fail(TBN_ERR_INVALID_ARG, "fp8 GEMV: workspace smaller than tbn_linear_f8_workspace_bytes");
  return launch_gemv_f8(x, K_in, prepared, alpha, K_out, y, ydt, epi ? epi->residual : nullptr,
                        epi ? epi->relu : 0, workspace, workspace_bytes, as_stream(stream));
}

size_t tbn_linear_workspace_bytes(tbn_dtype xdt, int64_t B, int64_t K_in, int64_t K_out) {
  if ((xdt != TBN_F32 && xdt != TBN_BF16) || B < 1 || K_in < 1 || K_out < 1) return 0;
  if (gemv_lut_shape_reason(xdt, B, K_in, K_out)[0] == '\0')
    return gemv_lut_workspace_bytes(K_in, K_out);
  if (xdt != TBN_BF16 || (B <= 8 && K_in % 64 == 0)) return 0;   // tensor-core GEMV, or no split
  static const uint32_t dummy[64] __attribute__((aligned(256))) = {};
  ConvProblem p{};
  if (!linear_as_conv(dummy, xdt, B, K_in, dummy, reinterpret_cast<const float*>(dummy), K_out,
                      const_cast<uint32_t*>(dummy), TBN_BF16, nullptr, &p))
    return 0;
  if (conv_igemm_unsupported_reason(p)[0] != '\0') return 0;
  size_t bytes = 0;
  return conv_igemm_splitk(p, &bytes) > 1 ? bytes : 0;
}

tbn_status tbn_linear_fwd_ws(const void* x, tbn_dtype xdt, int64_t B, int64_t K_in,
                             const uint32_t* codes, const float* alpha, int64_t K_out, void* y,
                             tbn_dtype ydt, const tbn_epilogue* epi, void* workspace,
                             size_t workspace_bytes, tbn_stream stream) {
  const tbn_status st = validate_linear(x, xdt, B, K_in, codes, alpha, K_out, y, ydt, epi);
  if (st != TBN_OK) return st;
  const int relu = epi ? epi->relu : 0;
  const void* residual = epi ? epi->residual : nullptr;
  if (gemv_lut_shape_reason(xdt, B, K_in, K_out)[0] == '\0') {
    // a batch-1 fp32 layer runs on the table-lookup GEMV only: the CUDA-core
    // 1x1 convolution it would fall back to reads the codes about a hundred
    // times slower than the table kernel, so that path is refused
    const size_t need = gemv_lut_workspace_bytes(K_in, K_out);
    if (workspace_bytes < need || (need > 0 && workspace == nullptr))
      return fail(TBN_ERR_UNSUPPORTED,
                  "linear: fp32 activations at batch 1 run on the table-lookup GEMV, which needs "
                  "%zu bytes of workspace for this shape: call tbn_linear_fwd_ws with "
                  "tbn_linear_workspace_bytes(...) bytes, or tbn_linear_fwd_noalloc",
                  need);
    if (!linear_uses_table(xdt, B, K_in, K_out, codes))
      return fail(TBN_ERR_MISALIGNED, "linear: the table-lookup GEMV needs 16-byte aligned codes");
    return launch_gemv_lut(x, K_in, codes, alpha, K_out, y, ydt, relu, residual, workspace,
                           workspace_bytes, as_stream(stream));
  }
  if (gemv_unsupported_reason(x, xdt, B, K_in, codes)[0] == '\0') {
    return launch_gemv(x, B, K_in, codes, alpha, K_out, y, ydt, relu, residual,
                       as_stream(stream));
  }
  // a fully-connected layer is a 1x1 convolution over a 1x1 image (Section 3);
  // with the workspace the query asks for, its K blocks are split over the
  // SMs its output tiles leave idle
  ConvProblem p{};
  const tbn_status vs = validate_conv(x, xdt, TBN_NHWC, B, K_in, 1, 1, codes, alpha, K_out, 1, 1,
                                      1, 1, 0, 0, y, ydt, epi, &p);
  if (vs != TBN_OK) return vs;
  if (workspace != nullptr && is_aligned(workspace, 16) &&
      conv_igemm_unsupported_reason(p)[0] == '\0') {
    size_t need = 0;
    const int splits = conv_igemm_splitk(p, &need);
    if (splits > 1 && workspace_bytes >= need) {
      p.partial = static_cast<float*>(workspace);
      p.ksplit = splits;
    }
  }
  return run_conv_auto(p, as_stream(stream));
}

tbn_status tbn_linear_fwd_noalloc(const void* x, tbn_dtype xdt, int64_t B, int64_t K_in,
                                  const uint32_t* codes, const float* alpha, int64_t K_out,
                                  void* y, tbn_dtype ydt, const tbn_epilogue* epi,
                                  tbn_stream stream) {
  const tbn_status st = validate_linear(x, xdt, B, K_in, codes, alpha, K_out, y, ydt, epi);
  if (st != TBN_OK) return st;
  const char* why = gemv_lut_unsupported_reason(xdt, B, K_in, K_out, codes);
  if (why[0] != '\0') return fail(TBN_ERR_UNSUPPORTED, "linear (no-alloc): %s", why);
  return launch_gemv_lut_static(x, K_in, codes, alpha, K_out, y, ydt, epi ? epi->relu : 0,
                                epi ? epi->residual : nullptr, as_stream(stream));
}

}  // extern "C"

namespace {

// Shape checks shared by the backward entry points; fills `sh`.
tbn_status validate_bwd(int64_t N, int64_t C, int64_t H, int64_t W, int64_t K, int64_t R,
                        int64_t S, int64_t sh, int64_t sw, int64_t ph, int64_t pw,
                        BwdConvShape* out) {
  if (N < 1 || C < 1 || H < 1 || W < 1 || K < 1 || R < 1 || S < 1)
    return fail(TBN_ERR_INVALID_ARG, "conv backward: sizes must be >= 1");
  if (sh < 1 || sw < 1 || ph < 0 || pw < 0)
    return fail(TBN_ERR_INVALID_ARG, "conv backward: bad stride/pad");
  // every size below 2^31 and pad below the kernel size before any sum or
  // product of them is formed
  const int64_t lim = int64_t(1) << 31;
  if (N >= lim || C >= lim || H >= lim || W >= lim || K >= lim || R >= lim || S >= lim ||
      sh >= lim || sw >= lim)
    return fail(TBN_ERR_UNSUPPORTED, "conv backward: size too large");
  if (ph > R - 1 || pw > S - 1)
    return fail(TBN_ERR_UNSUPPORTED, "conv backward: needs pad <= kernel size - 1");
  if (H + 2 * ph < R || W + 2 * pw < S)
    return fail(TBN_ERR_INVALID_ARG, "conv backward: kernel larger than padded input");
  BwdConvShape& p = *out;
  p.N = N; p.C = C; p.H = H; p.W = W; p.K = K; p.R = R; p.S = S;
  p.sh = sh; p.sw = sw; p.ph = ph; p.pw = pw;
  p.P = (H + 2 * ph - R) / sh + 1;
  p.Q = (W + 2 * pw - S) / sw + 1;
  const char* why = bwd_shape_reason(p);
  if (why[0] != '\0') return fail(TBN_ERR_UNSUPPORTED, "%s", why);
  return TBN_OK;
}

}  // namespace

extern "C" {

size_t tbn_conv2d_bwd_data_workspace_bytes(int64_t N, int64_t C, int64_t H, int64_t W, int64_t K,
                                           int64_t R, int64_t S, int64_t stride_h,
                                           int64_t stride_w, int64_t pad_h, int64_t pad_w) {
  BwdConvShape p{};
  if (validate_bwd(N, C, H, W, K, R, S, stride_h, stride_w, pad_h, pad_w, &p) != TBN_OK) return 0;
  return bwd_data_workspace_bytes(p);
}

tbn_status tbn_conv2d_bwd_data(const void* dy, int64_t N, int64_t C, int64_t H, int64_t W,
                               const uint32_t* codes, const float* alpha, int64_t K, int64_t R,
                               int64_t S, int64_t stride_h, int64_t stride_w, int64_t pad_h,
                               int64_t pad_w, void* dx, tbn_dtype dxdt, void* workspace,
                               size_t workspace_bytes, tbn_stream stream) {
  if (!dy || !codes || !alpha || !dx || !workspace)
    return fail(TBN_ERR_INVALID_ARG, "conv backward data: null pointer");
  if (dxdt != TBN_F32 && dxdt != TBN_BF16)
    return fail(TBN_ERR_INVALID_ARG, "conv backward data: bad dx dtype");
  BwdConvShape p{};
  const tbn_status st =
      validate_bwd(N, C, H, W, K, R, S, stride_h, stride_w, pad_h, pad_w, &p);
  if (st != TBN_OK) return st;
  if (workspace_bytes < bwd_data_workspace_bytes(p))
    return fail(TBN_ERR_INVALID_ARG, "conv backward data: workspace smaller than %zu bytes",
                bwd_data_workspace_bytes(p));
  if (!is_aligned(dy, 2) || !is_aligned(codes, 4) || !is_aligned(alpha, 4) ||
      !is_aligned(dx, dtype_size(dxdt)) || !is_aligned(workspace, 256))
    return fail(TBN_ERR_MISALIGNED, "conv backward data: misaligned pointer");
  return launch_bwd_data(p, dy, codes, alpha, dx, dxdt, workspace, as_stream(stream));
}

size_t tbn_conv2d_bwd_filter_workspace_bytes(int64_t N, int64_t C, int64_t H, int64_t W,
                                             int64_t K, int64_t R, int64_t S, int64_t stride_h,
                                             int64_t stride_w, int64_t pad_h, int64_t pad_w) {
  BwdConvShape p{};
  if (validate_bwd(N, C, H, W, K, R, S, stride_h, stride_w, pad_h, pad_w, &p) != TBN_OK) return 0;
  return bwd_filter_workspace_bytes(p);
}

tbn_status tbn_conv2d_bwd_filter(const void* x, const void* dy, int64_t N, int64_t C, int64_t H,
                                 int64_t W, int64_t K, int64_t R, int64_t S, int64_t stride_h,
                                 int64_t stride_w, int64_t pad_h, int64_t pad_w, float* dw,
                                 void* workspace, size_t workspace_bytes, tbn_stream stream) {
  if (!x || !dy || !dw || !workspace)
    return fail(TBN_ERR_INVALID_ARG, "conv backward filter: null pointer");
  BwdConvShape p{};
  const tbn_status st =
      validate_bwd(N, C, H, W, K, R, S, stride_h, stride_w, pad_h, pad_w, &p);
  if (st != TBN_OK) return st;
  if (workspace_bytes < bwd_filter_workspace_bytes(p))
    return fail(TBN_ERR_INVALID_ARG, "conv backward filter: workspace smaller than %zu bytes",
                bwd_filter_workspace_bytes(p));
  if (!is_aligned(x, 2) || !is_aligned(dy, 2) || !is_aligned(dw, 4) || !is_aligned(workspace, 256))
    return fail(TBN_ERR_MISALIGNED, "conv backward filter: misaligned pointer");
  return launch_bwd_filter(p, x, dy, dw, workspace, as_stream(stream));
}

tbn_status tbn_maxpool2d_nhwc(const void* x, tbn_dtype dt, int64_t N, int64_t H, int64_t W,
                              int64_t C, int64_t kh, int64_t kw, int64_t sh, int64_t sw,
                              int64_t ph, int64_t pw, void* y, tbn_stream stream) {
  if (!x || !y) return fail(TBN_ERR_INVALID_ARG, "maxpool: null pointer");
  if (dt != TBN_F32 && dt != TBN_BF16) return fail(TBN_ERR_INVALID_ARG, "maxpool: bad dtype");
  if (N < 1 || H < 1 || W < 1 || C < 1 || kh < 1 || kw < 1 || sh < 1 || sw < 1 || ph < 0 ||
      pw < 0)
    return fail(TBN_ERR_INVALID_ARG, "maxpool: bad sizes");
  const int64_t lim = int64_t(1) << 31;
  if (H >= lim || W >= lim || C >= lim || N >= lim || kh >= lim || kw >= lim || sh >= lim ||
      sw >= lim)
    return fail(TBN_ERR_UNSUPPORTED, "maxpool: a size is 2^31 or more");
  if (ph >= kh || pw >= kw) return fail(TBN_ERR_INVALID_ARG, "maxpool: padding must be below the window");
  if (kh > H + 2 * ph || kw > W + 2 * pw) return fail(TBN_ERR_INVALID_ARG, "maxpool: window larger than the padded input");
  if (!mul_ok(N * H, W * C, int64_t(1) << 46)) return fail(TBN_ERR_UNSUPPORTED, "maxpool: too large");
  if (!is_aligned(x, dtype_size(dt)) || !is_aligned(y, dtype_size(dt)))
    return fail(TBN_ERR_MISALIGNED, "maxpool: misaligned pointer");
  return launch_maxpool_nhwc(x, dt, N, H, W, C, kh, kw, sh, sw, ph, pw, y, as_stream(stream));
}

tbn_status tbn_nchw_to_nhwc(const void* x, tbn_dtype dt, int64_t N, int64_t C, int64_t H,
                            int64_t W, int64_t C_pad, void* y, tbn_stream stream) {
  if (!x || !y) return fail(TBN_ERR_INVALID_ARG, "nchw_to_nhwc: null pointer");
  if (dt != TBN_F32 && dt != TBN_BF16) return fail(TBN_ERR_INVALID_ARG, "nchw_to_nhwc: bad dtype");
  if (N < 1 || C < 1 || H < 1 || W < 1 || C_pad < C)
    return fail(TBN_ERR_INVALID_ARG, "nchw_to_nhwc: bad sizes");
  if (!mul_ok(N * H, W * C_pad, int64_t(1) << 46)) return fail(TBN_ERR_UNSUPPORTED, "nchw_to_nhwc: too large");
  if (!is_aligned(x, dtype_size(dt)) || !is_aligned(y, dtype_size(dt)))
    return fail(TBN_ERR_MISALIGNED, "nchw_to_nhwc: misaligned pointer");
  return launch_nchw_to_nhwc(x, dt, N, C, H, W, C_pad, y, as_stream(stream));
}

}  // extern "C"

extern "C" {

tbn_status tbn_repack(const uint32_t* in, int64_t K, int64_t n, uint32_t* out,
                      tbn_repack_direction dir, tbn_stream stream) {
  if (!in || !out) return fail(TBN_ERR_INVALID_ARG, "repack: null pointer");
  if (dir != TBN_REPACK_CANONICAL_TO_PLANAR && dir != TBN_REPACK_PLANAR_TO_CANONICAL)
    return fail(TBN_ERR_INVALID_ARG, "repack: bad direction");
  if (K < 1 || n < 1) return fail(TBN_ERR_INVALID_ARG, "repack: K, n must be >= 1");
  if (n >= (int64_t(1) << 31) || !mul_ok(K, (n + 15) / 16, int64_t(1) << 40))
    return fail(TBN_ERR_UNSUPPORTED, "repack: too large");
  if (!is_aligned(in, 4) || !is_aligned(out, 4))
    return fail(TBN_ERR_MISALIGNED, "repack: pointers must be 4-byte aligned");
  const int64_t words = K * ((n + 15) / 16);
  const uintptr_t a = reinterpret_cast<uintptr_t>(in), b = reinterpret_cast<uintptr_t>(out);
  const uintptr_t bytes = static_cast<uintptr_t>(words) * 4u;
  if (a != b && a < b + bytes && b < a + bytes)
    return fail(TBN_ERR_INVALID_ARG, "repack: in and out overlap (only in == out is allowed)");
  return launch_repack(in, words, out, dir == TBN_REPACK_CANONICAL_TO_PLANAR, as_stream(stream));
}

tbn_status tbn_dense_conv2d_fwd(const void* x, tbn_dtype xdt, tbn_layout layout, int64_t N,
                                int64_t C, int64_t H, int64_t W, const float* w, int64_t K,
                                int64_t R, int64_t S, int64_t stride_h, int64_t stride_w,
                                int64_t pad_h, int64_t pad_w, void* y, tbn_dtype ydt, int relu,
                                tbn_stream stream) {
  if (!w) return fail(TBN_ERR_INVALID_ARG, "dense conv: null pointer");
  if (layout == TBN_S2D_NHWC)
    return fail(TBN_ERR_UNSUPPORTED, "dense conv: no space-to-depth input");
  // the shape, dtype, layout and alignment checks of the two-bit convolution;
  // the weights stand in for its codes and alpha (both only checked for
  // being non-null and 4-byte aligned)
  const tbn_epilogue epi{relu != 0 ? 1 : 0, nullptr, 0};
  ConvProblem p{};
  const tbn_status st =
      validate_conv(x, xdt, layout, N, C, H, W, reinterpret_cast<const uint32_t*>(w), w, K, R, S,
                    stride_h, stride_w, pad_h, pad_w, y, ydt, &epi, &p);
  if (st != TBN_OK) return st;
  if (!mul_ok(K, C * R * S, int64_t(1) << 40))
    return fail(TBN_ERR_UNSUPPORTED, "dense conv: weights too large");
  return launch_dense_conv(p, w, as_stream(stream));
}

tbn_status tbn_avgpool2d_global_nhwc(const void* x, tbn_dtype xdt, int64_t N, int64_t H,
                                     int64_t W, int64_t C, void* y, tbn_dtype ydt,
                                     tbn_stream stream) {
  if (!x || !y) return fail(TBN_ERR_INVALID_ARG, "avgpool: null pointer");
  if ((xdt != TBN_F32 && xdt != TBN_BF16) || (ydt != TBN_F32 && ydt != TBN_BF16))
    return fail(TBN_ERR_INVALID_ARG, "avgpool: bad dtype");
  if (N < 1 || H < 1 || W < 1 || C < 1) return fail(TBN_ERR_INVALID_ARG, "avgpool: bad sizes");
  const int64_t lim = int64_t(1) << 31;
  if (N >= lim || H >= lim || W >= lim || C >= lim || !mul_ok(N * C, H * W, int64_t(1) << 46))
    return fail(TBN_ERR_UNSUPPORTED, "avgpool: too large");
  if (!is_aligned(x, dtype_size(xdt)) || !is_aligned(y, dtype_size(ydt)))
    return fail(TBN_ERR_MISALIGNED, "avgpool: misaligned pointer");
  return launch_avgpool_global_nhwc(x, xdt, N, H, W, C, y, ydt, as_stream(stream));
}

tbn_status tbn_dense_linear_fwd(const float* x, int64_t B, int64_t K_in, const float* w,
                                int64_t K_out, void* y, tbn_dtype ydt, int relu,
                                tbn_stream stream) {
  if (!x || !w || !y) return fail(TBN_ERR_INVALID_ARG, "dense linear: null pointer");
  if (ydt != TBN_F32 && ydt != TBN_BF16) return fail(TBN_ERR_INVALID_ARG, "dense linear: bad y dtype");
  if (B < 1 || K_in < 1 || K_out < 1) return fail(TBN_ERR_INVALID_ARG, "dense linear: sizes must be >= 1");
  const int64_t lim = int64_t(1) << 31;
  if (B >= lim || K_in >= lim || K_out >= lim || !mul_ok(K_out, K_in, int64_t(1) << 46) ||
      !mul_ok(B, K_in, int64_t(1) << 46))
    return fail(TBN_ERR_UNSUPPORTED, "dense linear: too large");
  if (!is_aligned(x, 4) || !is_aligned(w, 4) || !is_aligned(y, dtype_size(ydt)))
    return fail(TBN_ERR_MISALIGNED, "dense linear: misaligned pointer");
  return launch_dense_linear(x, B, K_in, w, K_out, y, ydt, relu, as_stream(stream));
}

}  // extern "C"
