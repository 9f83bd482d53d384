// tbn_conv_direct.cu -- CUDA-core direct two-bit convolution (Eq. 1) for
// every layout / dtype / stride / padding, plus the network glue kernels
// (NHWC max pooling with optional padding, NCHW -> NHWC with channel padding).
//
// Direct convolution: a CTA computes 128 output pixels x 32 filters.  The
// filters' codes are decoded once per CTA into shared memory as fp32 W~ (a
// chunk of taps at a time, tap-major so that all threads read the same
// 32 weights -- a broadcast); each thread owns one pixel, walks the taps in
// the codes' order, loads one activation per tap and does 32 FMAs.  This is
// the path for small-channel layers (the first layer of a network, where
// the implicit GEMM would pad C up to its tile) and the fallback for shapes
// the tensor-core kernel does not take.  x * W~ is exact in fp32; the sum is
// accumulated in fp32 in tap order.
#include <cuda_bf16.h>

#include <algorithm>
#include <mutex>
#include <cstdint>

#include "tbn_device.cuh"
#include "tbn_internal.h"

namespace tbn {
namespace {

constexpr int kPix = 128;    // pixels (threads) per CTA
constexpr int kFilt = 32;    // filters per CTA
constexpr int kTapChunk = 128;

template <typename T>
__device__ __forceinline__ float to_f32(T v);
template <>
__device__ __forceinline__ float to_f32<float>(float v) { return v; }
template <>
__device__ __forceinline__ float to_f32<__nv_bfloat16>(__nv_bfloat16 v) {
  return __bfloat162float(v);
}

template <typename T>
__device__ __forceinline__ T from_f32(float v);
template <>
__device__ __forceinline__ float from_f32<float>(float v) { return v; }
template <>
__device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float v) {
  return __float2bfloat16_rn(v);
}

struct DirectArgs {
  int64_t N, C, H, W, K, R, S, sh, sw, ph, pw, P, Q;
  int64_t Po, Qo;  // output extent (P/2, Q/2 with the fused 2x2 pool)
  int64_t wpf;     // words per filter
  const void* x;
  const uint32_t* codes;
  const float* alpha;
  void* y;
  const void* residual;
  int relu;
};

// kWin = 1: one conv output per thread, 32 filters.  kWin = 4: one 2x2-pooled
// output per thread (four conv outputs, max after ReLU), 8 filters.
// kLayout (tbn_layout): x is NHWC only for TBN_NHWC; the codes are in
// (r, s, c) order and y is NHWC for TBN_NHWC and TBN_NCHW_NHWC.
template <typename TX, typename TY, int kLayout, int kWin>
__global__ void __launch_bounds__(kPix) conv_direct_kernel(const DirectArgs a) {
  constexpr int kF = kWin == 1 ? kFilt : 8;
  constexpr bool kXNhwc = kLayout == TBN_NHWC, kRsc = kLayout != TBN_NCHW;
  constexpr bool kYNhwc = kLayout != TBN_NCHW;
  __shared__ __align__(16) float s_w[kTapChunk][kF];
  __shared__ int32_t s_off[kTapChunk];
  __shared__ int32_t s_rs[kTapChunk];

  const TX* __restrict__ x = static_cast<const TX*>(a.x);
  const int64_t npix = a.N * a.Po * a.Qo;
  const int64_t pix = static_cast<int64_t>(blockIdx.x) * kPix + threadIdx.x;
  const int64_t k0 = static_cast<int64_t>(blockIdx.y) * kF;
  const bool active = pix < npix;
  const int64_t pc = active ? pix : 0;
  const int64_t b = pc / (a.Po * a.Qo);
  const int64_t po = (pc / a.Qo) % a.Po;
  const int64_t qo = pc % a.Qo;
  int h0[kWin], w0[kWin];
  int64_t base[kWin];
#pragma unroll
  for (int wdx = 0; wdx < kWin; ++wdx) {
    const int64_t p = kWin == 1 ? po : 2 * po + wdx / 2;
    const int64_t q = kWin == 1 ? qo : 2 * qo + wdx % 2;
    h0[wdx] = static_cast<int>(p * a.sh - a.ph);
    w0[wdx] = static_cast<int>(q * a.sw - a.pw);
    // element offset of (b, c = 0, h0, w0)
    base[wdx] = kXNhwc ? ((b * a.H + h0[wdx]) * a.W + w0[wdx]) * a.C
                      : ((b * a.C) * a.H + h0[wdx]) * a.W + w0[wdx];
  }
  const int H = static_cast<int>(a.H), W = static_cast<int>(a.W);

  float acc[kWin][kF];
#pragma unroll
  for (int wdx = 0; wdx < kWin; ++wdx)
#pragma unroll
    for (int f = 0; f < kF; ++f) acc[wdx][f] = 0.0f;

  const int64_t ntaps = a.C * a.R * a.S;
  for (int64_t t0 = 0; t0 < ntaps; t0 += kTapChunk) {
    const int tc = (ntaps - t0 < kTapChunk) ? static_cast<int>(ntaps - t0) : kTapChunk;
    __syncthreads();
    // decode W~ for this tap chunk: s_w[t][f]
    for (int i = threadIdx.x; i < tc * kF; i += kPix) {
      const int t = i / kF, f = i % kF;
      const int64_t k = k0 + f;
      float v = 0.0f;
      if (k < a.K) {
        const int64_t ti = t0 + t;
        const uint32_t w = a.codes[k * a.wpf + (ti >> 4)];
        v = code_value(code_field(w, static_cast<int>(ti & 15)));
      }
      s_w[t][f] = v;
    }
    for (int t = threadIdx.x; t < tc; t += kPix) {
      const int64_t ti = t0 + t;
      int64_t c, r, s;
      if (kRsc) {
        r = ti / (a.S * a.C);
        s = (ti / a.C) % a.S;
        c = ti % a.C;
      } else {
        c = ti / (a.R * a.S);
        r = (ti / a.S) % a.R;
        s = ti % a.S;
      }
      s_off[t] = static_cast<int32_t>(kXNhwc ? (r * a.W + s) * a.C + c : (c * a.H + r) * a.W + s);
      s_rs[t] = static_cast<int32_t>((r << 16) | s);
    }
    __syncthreads();
    if (active) {
      for (int t = 0; t < tc; ++t) {
        const int32_t rs = s_rs[t];
        const int off = s_off[t];
        const float4* wr = reinterpret_cast<const float4*>(&s_w[t][0]);
#pragma unroll
        for (int wdx = 0; wdx < kWin; ++wdx) {
          const int h = h0[wdx] + (rs >> 16), w = w0[wdx] + (rs & 0xFFFF);
          float xv = 0.0f;
          if (h >= 0 && h < H && w >= 0 && w < W) xv = to_f32<TX>(x[base[wdx] + off]);
#pragma unroll
          for (int f4 = 0; f4 < kF / 4; ++f4) {
            const float4 wv = wr[f4];
            acc[wdx][4 * f4 + 0] = fmaf(xv, wv.x, acc[wdx][4 * f4 + 0]);
            acc[wdx][4 * f4 + 1] = fmaf(xv, wv.y, acc[wdx][4 * f4 + 1]);
            acc[wdx][4 * f4 + 2] = fmaf(xv, wv.z, acc[wdx][4 * f4 + 2]);
            acc[wdx][4 * f4 + 3] = fmaf(xv, wv.w, acc[wdx][4 * f4 + 3]);
          }
        }
      }
    }
  }
  if (!active) return;

  TY* __restrict__ y = static_cast<TY*>(a.y);
  const TY* __restrict__ res = static_cast<const TY*>(a.residual);
#pragma unroll
  for (int f = 0; f < kF; ++f) {
    const int64_t k = k0 + f;
    if (k < a.K) {
      const int64_t o = kYNhwc ? pix * a.K + k : ((b * a.K + k) * a.Po + po) * a.Qo + qo;
      float best = -INFINITY;
#pragma unroll
      for (int wdx = 0; wdx < kWin; ++wdx) {
        float v = a.alpha[k] * acc[wdx][f];
        if (res != nullptr) v += to_f32<TY>(res[o]);
        if (a.relu) v = fmaxf(v, 0.0f);
        best = fmaxf(best, v);
      }
      y[o] = from_f32<TY>(best);
    }
  }
}

template <typename TX, typename TY, int kLayout, int kWin>
tbn_status launch_direct_t(const DirectArgs& a, cudaStream_t s) {
  constexpr int kF = kWin == 1 ? kFilt : 8;
  const int64_t npix = a.N * a.Po * a.Qo;
  const int64_t gx = (npix + kPix - 1) / kPix;
  const int64_t gy = (a.K + kF - 1) / kF;
  if (gx > 0x7fffffffLL || gy > 65535)
    return fail(TBN_ERR_UNSUPPORTED, "conv direct: grid too large (%lld x %lld)", (long long)gx,
                (long long)gy);
  if (a.H >= (1 << 30) || a.W >= (1 << 30))
    return fail(TBN_ERR_UNSUPPORTED, "conv direct: image too large");
  conv_direct_kernel<TX, TY, kLayout, kWin><<<dim3((unsigned)gx, (unsigned)gy), kPix, 0, s>>>(a);
  return check_launch("conv_direct_kernel");
}

template <typename TX, typename TY, int kLayout>
tbn_status launch_direct_w(const DirectArgs& a, bool pool, cudaStream_t s) {
  return pool ? launch_direct_t<TX, TY, kLayout, 4>(a, s) : launch_direct_t<TX, TY, kLayout, 1>(a, s);
}

template <int kLayout>
tbn_status launch_direct_l(const DirectArgs& a, bool xb, bool yb, bool pool, cudaStream_t s) {
  using bf = __nv_bfloat16;
  if (xb && yb) return launch_direct_w<bf, bf, kLayout>(a, pool, s);
  if (xb && !yb) return launch_direct_w<bf, float, kLayout>(a, pool, s);
  if (!xb && yb) return launch_direct_w<float, bf, kLayout>(a, pool, s);
  return launch_direct_w<float, float, kLayout>(a, pool, s);
}

// Windows that reach into the padding skip those taps (-infinity padding).
template <typename T>
__global__ void __launch_bounds__(256) maxpool_nhwc_kernel(const T* __restrict__ x, int64_t N,
                                                           int64_t H, int64_t W, int64_t C,
                                                           int64_t kh, int64_t kw, int64_t sh,
                                                           int64_t sw, int64_t ph, int64_t pw,
                                                           int64_t Ho, int64_t Wo,
                                                           T* __restrict__ y) {
  const int64_t total = N * Ho * Wo * C;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < total;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t c = i % C;
    const int64_t wo = (i / C) % Wo;
    const int64_t ho = (i / (C * Wo)) % Ho;
    const int64_t b = i / (C * Wo * Ho);
    float m = -INFINITY;
    for (int64_t u = 0; u < kh; ++u) {
      const int64_t h = ho * sh - ph + u;
      if (h < 0 || h >= H) continue;
      for (int64_t v = 0; v < kw; ++v) {
        const int64_t w = wo * sw - pw + v;
        if (w < 0 || w >= W) continue;
        const float t = to_f32<T>(x[((b * H + h) * W + w) * C + c]);
        if (t > m) m = t;
      }
    }
    y[i] = from_f32<T>(m);
  }
}

// 8 channels (16 bytes) of bf16 per thread.
__global__ void __launch_bounds__(256) maxpool_nhwc_bf16x8_kernel(
    const uint4* __restrict__ x, int64_t N, int64_t H, int64_t W, int64_t C8, int64_t kh,
    int64_t kw, int64_t sh, int64_t sw, int64_t ph, int64_t pw, int64_t Ho, int64_t Wo,
    uint4* __restrict__ y) {
  const int64_t total = N * Ho * Wo * C8;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < total;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t c = i % C8;
    const int64_t wo = (i / C8) % Wo;
    const int64_t ho = (i / (C8 * Wo)) % Ho;
    const int64_t b = i / (C8 * Wo * Ho);
    float m[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) m[e] = -INFINITY;
    for (int64_t u = 0; u < kh; ++u) {
      const int64_t h = ho * sh - ph + u;
      if (h < 0 || h >= H) continue;
      for (int64_t v = 0; v < kw; ++v) {
        const int64_t w = wo * sw - pw + v;
        if (w < 0 || w >= W) continue;
        const uint4 t = x[((b * H + h) * W + w) * C8 + c];
        const __nv_bfloat16* tb = reinterpret_cast<const __nv_bfloat16*>(&t);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const float f = __bfloat162float(tb[e]);
          if (f > m[e]) m[e] = f;
        }
      }
    }
    uint4 o;
    __nv_bfloat16* ob = reinterpret_cast<__nv_bfloat16*>(&o);
#pragma unroll
    for (int e = 0; e < 8; ++e) ob[e] = __float2bfloat16_rn(m[e]);
    y[i] = o;
  }
}

// One output row (image b, row ho) per block, bf16 NHWC with C % 8 == 0: a
// thread takes (column, 8-channel vector) items, so consecutive threads read
// consecutive 16-byte vectors of each tap; the max is taken on bf16 pairs
// (exact: max of two bf16 values is one of them).  Taps in the padding are
// skipped.
// kK > 0: a kK x kK window, all of its loads issued before the first max
// (taps in the padding load nothing and count as -infinity).
template <int kK>
__global__ void __launch_bounds__(256) maxpool_row_bf16x8_kernel(
    const uint4* __restrict__ x, int H, int W, int C8, int kh, int kw, int sh, int sw, int ph,
    int pw, int Ho, int Wo, uint4* __restrict__ y) {
  const int b = blockIdx.x / Ho, ho = blockIdx.x - b * Ho;
  const int items = Wo * C8;
  const uint4* xb = x + static_cast<int64_t>(b) * H * W * C8;
  uint4* yrow = y + (static_cast<int64_t>(b) * Ho + ho) * Wo * C8;
  const int h_lo = max(0, ho * sh - ph), h_hi = min(H, ho * sh - ph + kh);
  if constexpr (kK > 0) {
    const uint4 ninf4 = make_uint4(0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u);
    for (int i = threadIdx.x; i < items; i += 256) {
      const int wo = i / C8, c = i - wo * C8;
      const int h0 = ho * sh - ph, w0 = wo * sw - pw;
      uint4 t[kK * kK];
#pragma unroll
      for (int u = 0; u < kK; ++u)
#pragma unroll
        for (int v = 0; v < kK; ++v) {
          const int h = h0 + u, w = w0 + v;
          t[u * kK + v] = (h >= 0 && h < H && w >= 0 && w < W)
                              ? __ldg(xb + (static_cast<int64_t>(h) * W + w) * C8 + c)
                              : ninf4;
        }
      __nv_bfloat162 m[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) m[e] = reinterpret_cast<const __nv_bfloat162*>(&t[0])[e];
#pragma unroll
      for (int j = 1; j < kK * kK; ++j)
#pragma unroll
        for (int e = 0; e < 4; ++e)
          m[e] = __hmax2(m[e], reinterpret_cast<const __nv_bfloat162*>(&t[j])[e]);
      yrow[i] = *reinterpret_cast<const uint4*>(m);
    }
    return;
  }
  for (int i = threadIdx.x; i < items; i += 256) {
    const int wo = i / C8, c = i - wo * C8;
    const int w_lo = max(0, wo * sw - pw), w_hi = min(W, wo * sw - pw + kw);
    __nv_bfloat162 m[4];
    const __nv_bfloat162 ninf = __floats2bfloat162_rn(-INFINITY, -INFINITY);
#pragma unroll
    for (int e = 0; e < 4; ++e) m[e] = ninf;
    for (int h = h_lo; h < h_hi; ++h) {
      const uint4* xr = xb + (static_cast<int64_t>(h) * W) * C8 + c;
      for (int w = w_lo; w < w_hi; ++w) {
        const uint4 t = __ldg(xr + static_cast<int64_t>(w) * C8);
        const __nv_bfloat162* tb = reinterpret_cast<const __nv_bfloat162*>(&t);
#pragma unroll
        for (int e = 0; e < 4; ++e) m[e] = __hmax2(m[e], tb[e]);
      }
    }
    yrow[i] = *reinterpret_cast<const uint4*>(m);
  }
}

// NCHW -> NHWC for any H*W (the vector kernel below needs H*W % 8 == 0):
// a block moves 1024 pixels of one image through shared memory, reading
// each channel plane with consecutive 2-byte loads and writing the pixels'
// Cp channels as one contiguous run of 2-byte stores.
constexpr int kT2Pix = 1024;

__global__ void __launch_bounds__(256) nchw_to_nhwc_tiled_kernel(
    const uint16_t* __restrict__ x, int C, int HW, int Cp, uint16_t* __restrict__ y) {
  extern __shared__ uint16_t t2[];   // [kT2Pix][Cp]
  grid_dependents_launch();
  const int b = blockIdx.y;
  const int p0 = blockIdx.x * kT2Pix;
  const int np = min(kT2Pix, HW - p0);
  const uint16_t* xb = x + static_cast<int64_t>(b) * C * HW + p0;
  for (int c = 0; c < Cp; ++c)
    for (int i = threadIdx.x; i < np; i += 256)
      t2[i * Cp + c] = c < C ? __ldg(xb + static_cast<int64_t>(c) * HW + i) : uint16_t(0);
  __syncthreads();
  uint16_t* yb = y + (static_cast<int64_t>(b) * HW + p0) * Cp;
  for (int i = threadIdx.x; i < np * Cp; i += 256) yb[i] = t2[i];
}

// One thread per pixel of one image (blockIdx.y): reads the pixel's C
// values from the C planes (coalesced across the warp's consecutive pixels)
// and writes its Cp channels contiguously; no index divisions.
template <typename T>
__global__ void __launch_bounds__(256) nchw_to_nhwc_kernel(const T* __restrict__ x, int C, int HW,
                                                           int Cp, T* __restrict__ y) {
  const int hw = blockIdx.x * 256 + threadIdx.x;
  if (hw >= HW) return;
  const int64_t b = blockIdx.y;
  const T* src = x + b * C * static_cast<int64_t>(HW) + hw;
  T* dst = y + (b * HW + hw) * static_cast<int64_t>(Cp);
  for (int c = 0; c < Cp; ++c)
    dst[c] = c < C ? src[static_cast<int64_t>(c) * HW] : from_f32<T>(0.0f);
}

// bf16 with H*W % 8 == 0 and 16-byte aligned tensors, Cp <= 8: one thread
// per 8 consecutive pixels of one image reads one 16-byte vector from each of
// the C planes and writes the 8 pixels' Cp channels as Cp 16-byte vectors.
template <int kCp>
__global__ void __launch_bounds__(256) nchw_to_nhwc_bf16x8_kernel(const uint4* __restrict__ x,
                                                                  int C, int HW8, int64_t total,
                                                                  uint4* __restrict__ y) {
  // the next kernel (a convolution launched as a programmatic dependent)
  // may start its set-up now; it reads this kernel's output only after
  // this grid has completed
  grid_dependents_launch();
  const int64_t t = static_cast<int64_t>(blockIdx.x) * 256 + threadIdx.x;
  if (t >= total) return;
  const int64_t b = t / HW8;
  const int hw8 = static_cast<int>(t - b * HW8);
  uint32_t in[kCp][4];
#pragma unroll
  for (int c = 0; c < kCp; ++c) {
    uint4 v = make_uint4(0u, 0u, 0u, 0u);
    if (c < C) v = x[(b * C + c) * HW8 + hw8];
    in[c][0] = v.x;
    in[c][1] = v.y;
    in[c][2] = v.z;
    in[c][3] = v.w;
  }
  uint4* dst = y + t * kCp;
#pragma unroll
  for (int o = 0; o < kCp; ++o) {
    uint32_t w[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      // output elements e = 8 o + 2 k, 8 o + 2 k + 1 -> (pixel e / kCp, channel e % kCp)
      const int e0 = 8 * o + 2 * k, e1 = e0 + 1;
      const uint32_t lo = (in[e0 % kCp][(e0 / kCp) >> 1] >> (16 * ((e0 / kCp) & 1))) & 0xFFFFu;
      const uint32_t hi = (in[e1 % kCp][(e1 / kCp) >> 1] >> (16 * ((e1 / kCp) & 1))) & 0xFFFFu;
      w[k] = lo | (hi << 16);
    }
    dst[o] = make_uint4(w[0], w[1], w[2], w[3]);
  }
}

int64_t grid_for(int64_t total) {
  const int64_t cap = static_cast<int64_t>(device_sm_count()) * 16;
  return std::max<int64_t>(1, std::min<int64_t>((total + 255) / 256, cap));
}

// Space-to-depth layout change (see S2dGeom): block (xc, Y, n) writes
// space-to-depth pixels X in [pix xc, pix xc + pix) of row Y, pix = 256 / s.
// The s input rows s Y + dy - ph, columns [pix s xc - pw, + pix s), all C
// channels, are first staged in shared memory as [dy][column][c] (zero
// outside the image): a warp copies one input row segment at a time
// (NCHW: a channel's row; NHWC: all channels of a row, one contiguous
// range of x).  In that layout the s C channels of dy-row dy of pixel X are
// one run of the tile, so when s C % 4 == 0 a 16-byte output chunk is two
// aligned 8-byte shared loads; otherwise it is gathered 2 bytes at a time
// through a 64-entry offset table.  kNchw: x is [N][C][H][W], else
// [N][H][W][C].
constexpr int kS2dThreads = 256;

template <bool kNchw>
__global__ void __launch_bounds__(kS2dThreads) space_to_depth_kernel(
    const uint16_t* __restrict__ x, int C, int H, int W, int s, int ph, int pw, int Hs, int Ws,
    uint4* __restrict__ out) {
  extern __shared__ __align__(16) uint16_t s2d_tile[];   // [s][pix s][C]
  __shared__ int s2d_off[64];              // channel j -> tile offset of pixel 0, or -1
  const int xc = blockIdx.x, Y = blockIdx.y, n = blockIdx.z;
  const int pix = kS2dThreads / s;
  const int cols = pix * s;                // <= 256
  const int w0 = xc * cols - pw;
  const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
  const int sc = s * C;                    // channels of one dy-row of a pixel
  const bool runs = (sc & 3) == 0;
  if (!runs && t < 64) {
    int o = -1;
    if (t < s * sc) {
      const int dy = t / sc, dx = (t / C) % s, c = t % C;
      o = (dy * cols + dx) * C + c;
    }
    s2d_off[t] = o;
  }
  // stage: segment rows, 4 loads per lane in flight before their stores
  const int nrows = kNchw ? C * s : s;
  const int len = kNchw ? cols : cols * C;      // elements per segment row
  for (int r = warp; r < nrows; r += kS2dThreads / 32) {
    const int c = kNchw ? r / s : 0, dy = kNchw ? r - c * s : r;
    const int h = s * Y + dy - ph;
    const bool hin = h >= 0 && h < H;
    const uint16_t* xr =
        kNchw ? x + ((static_cast<int64_t>(n) * C + c) * H + (hin ? h : 0)) * W + w0
              : x + ((static_cast<int64_t>(n) * H + (hin ? h : 0)) * W + w0) * static_cast<int64_t>(C);
    // in-image elements of the segment row: [lo, hi)
    const int lo = max(0, -w0) * (kNchw ? 1 : C);
    const int hi = max(lo, min(cols, W - w0) * (kNchw ? 1 : C));
    uint16_t* tr = s2d_tile + dy * cols * C + c;
    const int tstride = kNchw ? C : 1;
    for (int e0 = 0; e0 < len; e0 += 128) {
      uint16_t v[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int e = e0 + lane + 32 * i;
        v[i] = (hin && e >= lo && e < hi) ? xr[e] : static_cast<uint16_t>(0);
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int e = e0 + lane + 32 * i;
        if (e < len) tr[e * tstride] = v[i];
      }
    }
  }
  __syncthreads();
  const int npix = min(pix, Ws - xc * pix);
  const int q = t & 7;   // this thread's 16-byte chunk: channels 8 q .. 8 q + 7
  uint4* orow = out + ((static_cast<int64_t>(n) * Hs + Y) * Ws + xc * pix) * 8;
  if (runs) {
    // channels 4 p .. 4 p + 3 (p = 2 q, 2 q + 1): dy = 4 p / sc, at element
    // offset 4 p % sc of dy-row dy's run, which starts at (dy cols + s X) C
    int po[2];
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      const int j = 4 * (2 * q + u);
      po[u] = j < s * sc ? (j / sc) * cols * C + j % sc : -1;
    }
    const uint2* tile8 = reinterpret_cast<const uint2*>(s2d_tile);
    for (int xi = t >> 3; xi < npix; xi += kS2dThreads / 8) {
      uint2 a = make_uint2(0u, 0u), b = make_uint2(0u, 0u);
      if (po[0] >= 0) a = tile8[(po[0] + xi * sc) >> 2];
      if (po[1] >= 0) b = tile8[(po[1] + xi * sc) >> 2];
      orow[xi * 8 + q] = make_uint4(a.x, a.y, b.x, b.y);
    }
  } else {
    int off[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) off[i] = s2d_off[8 * q + i];
    for (int xi = t >> 3; xi < npix; xi += kS2dThreads / 8) {
      uint32_t hv[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) hv[i] = off[i] >= 0 ? s2d_tile[off[i] + xi * sc] : 0u;
      orow[xi * 8 + q] = make_uint4(hv[0] | (hv[1] << 16), hv[2] | (hv[3] << 16),
                                    hv[4] | (hv[5] << 16), hv[6] | (hv[7] << 16));
    }
  }
}

// The same layout change specialized for NCHW x with stride kS and kC
// channels, kS kC % 4 == 0 (AlexNet's first layer: 4, 3): block (Y, n)
// writes all Ws pixels of row Y (Ws <= 256 / kS, checked by the caller).
// Thread t owns input column t - pw of the kC kS rows and issues all its
// loads before its stores; the tile offsets are compile-time constants.
template <int kS, int kC>
__global__ void __launch_bounds__(kS2dThreads) space_to_depth_nchw_kernel(
    const uint16_t* __restrict__ x, int H, int W, int ph, int pw, int Hs, int Ws,
    uint4* __restrict__ out) {
  constexpr int kCols = (kS2dThreads / kS) * kS;
  constexpr int kSc = kS * kC;
  static_assert(kSc % 4 == 0 && kS * kSc <= 64, "specialization");
  __shared__ __align__(16) uint16_t tile[kS * kCols * kC];   // [dy][column][c]
  const int Y = blockIdx.x, n = blockIdx.y;
  const int t = threadIdx.x;
  if (t < kCols) {
    const int w = t - pw;
    const bool win = w >= 0 && w < W;
    const int64_t HW = static_cast<int64_t>(H) * W;
    const uint16_t* xc = x + static_cast<int64_t>(n) * kC * HW + w;
    const int hb = kS * Y - ph;
    uint16_t v[kC][kS];
#pragma unroll
    for (int dy = 0; dy < kS; ++dy) {
      const int h = hb + dy;
      const bool ok = win && h >= 0 && h < H;
#pragma unroll
      for (int c = 0; c < kC; ++c)
        v[c][dy] = ok ? xc[c * HW + static_cast<int64_t>(h) * W] : static_cast<uint16_t>(0);
    }
#pragma unroll
    for (int dy = 0; dy < kS; ++dy)
#pragma unroll
      for (int c = 0; c < kC; ++c) tile[(dy * kCols + t) * kC + c] = v[c][dy];
  }
  __syncthreads();
  const int q = t & 7;
  int po[2];
#pragma unroll
  for (int u = 0; u < 2; ++u) {
    const int j = 4 * (2 * q + u);
    po[u] = j < kS * kSc ? (j / kSc) * kCols * kC + j % kSc : -1;
  }
  const uint2* tile8 = reinterpret_cast<const uint2*>(tile);
  uint4* orow = out + (static_cast<int64_t>(n) * Hs + Y) * Ws * 8;
  for (int xi = t >> 3; xi < Ws; xi += kS2dThreads / 8) {
    uint2 a = make_uint2(0u, 0u), b = make_uint2(0u, 0u);
    if (po[0] >= 0) a = tile8[(po[0] + xi * kSc) >> 2];
    if (po[1] >= 0) b = tile8[(po[1] + xi * kSc) >> 2];
    orow[xi * 8 + q] = make_uint4(a.x, a.y, b.x, b.y);
  }
}

}  // namespace

tbn_status launch_conv_direct(const ConvProblem& p, cudaStream_t s) {
  DirectArgs a{};
  a.N = p.N; a.C = p.C; a.H = p.H; a.W = p.W; a.K = p.K; a.R = p.R; a.S = p.S;
  a.sh = p.sh; a.sw = p.sw; a.ph = p.ph; a.pw = p.pw; a.P = p.P; a.Q = p.Q;
  a.Po = p.pool ? p.P / 2 : p.P;
  a.Qo = p.pool ? p.Q / 2 : p.Q;
  a.wpf = (p.C * p.R * p.S + 15) / 16;
  a.x = p.x; a.codes = p.codes; a.alpha = p.alpha; a.y = p.y;
  a.residual = p.residual; a.relu = p.relu;
  const bool pool = p.pool != 0;
  const bool xb = p.xdt == TBN_BF16, yb = p.ydt == TBN_BF16;
  if (p.layout == TBN_NHWC) return launch_direct_l<TBN_NHWC>(a, xb, yb, pool, s);
  if (p.layout == TBN_NCHW_NHWC) return launch_direct_l<TBN_NCHW_NHWC>(a, xb, yb, pool, s);
  return launch_direct_l<TBN_NCHW>(a, xb, yb, pool, s);
}

tbn_status launch_maxpool_nhwc(const void* x, tbn_dtype dt, int64_t N, int64_t H, int64_t W,
                               int64_t C, int64_t kh, int64_t kw, int64_t sh, int64_t sw,
                               int64_t ph, int64_t pw, void* y, cudaStream_t s) {
  const int64_t Ho = (H + 2 * ph - kh) / sh + 1, Wo = (W + 2 * pw - kw) / sw + 1;
  if (dt == TBN_BF16 && C % 8 == 0 && is_aligned(x, 16) && is_aligned(y, 16) &&
      N * Ho < (int64_t(1) << 31) && H * W * C < (int64_t(1) << 31)) {
    if (kh == 3 && kw == 3)
      maxpool_row_bf16x8_kernel<3><<<static_cast<unsigned>(N * Ho), 256, 0, s>>>(
          static_cast<const uint4*>(x), (int)H, (int)W, (int)(C / 8), (int)kh, (int)kw, (int)sh,
          (int)sw, (int)ph, (int)pw, (int)Ho, (int)Wo, static_cast<uint4*>(y));
    else if (kh == 2 && kw == 2)
      maxpool_row_bf16x8_kernel<2><<<static_cast<unsigned>(N * Ho), 256, 0, s>>>(
          static_cast<const uint4*>(x), (int)H, (int)W, (int)(C / 8), (int)kh, (int)kw, (int)sh,
          (int)sw, (int)ph, (int)pw, (int)Ho, (int)Wo, static_cast<uint4*>(y));
    else
      maxpool_row_bf16x8_kernel<0><<<static_cast<unsigned>(N * Ho), 256, 0, s>>>(
          static_cast<const uint4*>(x), (int)H, (int)W, (int)(C / 8), (int)kh, (int)kw, (int)sh,
          (int)sw, (int)ph, (int)pw, (int)Ho, (int)Wo, static_cast<uint4*>(y));
  } else if (dt == TBN_BF16 && C % 8 == 0 && is_aligned(x, 16) && is_aligned(y, 16)) {
    const int64_t total = N * Ho * Wo * (C / 8);
    maxpool_nhwc_bf16x8_kernel<<<(unsigned)grid_for(total), 256, 0, s>>>(
        static_cast<const uint4*>(x), N, H, W, C / 8, kh, kw, sh, sw, ph, pw, Ho, Wo,
        static_cast<uint4*>(y));
  } else if (dt == TBN_BF16) {
    const int64_t total = N * Ho * Wo * C;
    maxpool_nhwc_kernel<__nv_bfloat16><<<(unsigned)grid_for(total), 256, 0, s>>>(
        static_cast<const __nv_bfloat16*>(x), N, H, W, C, kh, kw, sh, sw, ph, pw, Ho, Wo,
        static_cast<__nv_bfloat16*>(y));
  } else {
    const int64_t total = N * Ho * Wo * C;
    maxpool_nhwc_kernel<float><<<(unsigned)grid_for(total), 256, 0, s>>>(
        static_cast<const float*>(x), N, H, W, C, kh, kw, sh, sw, ph, pw, Ho, Wo,
        static_cast<float*>(y));
  }
  return check_launch("maxpool_nhwc_kernel");
}

tbn_status launch_nchw_to_nhwc(const void* x, tbn_dtype dt, int64_t N, int64_t C, int64_t H,
                               int64_t W, int64_t C_pad, void* y, cudaStream_t s) {
  if (N > 65535 || H * W >= (int64_t(1) << 31) - 256 || C_pad >= (int64_t(1) << 31))
    return fail(TBN_ERR_UNSUPPORTED, "nchw_to_nhwc: N > 65535 or H*W too large");
  // the shared-memory split of the kernels around it in a network (which
  // need nearly all of it): no SM reconfiguration between launches
  static std::once_flag attr_once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(attr_once, [] {
    const void* fns[11] = {(const void*)nchw_to_nhwc_bf16x8_kernel<1>,
                           (const void*)nchw_to_nhwc_bf16x8_kernel<2>,
                           (const void*)nchw_to_nhwc_bf16x8_kernel<3>,
                           (const void*)nchw_to_nhwc_bf16x8_kernel<4>,
                           (const void*)nchw_to_nhwc_bf16x8_kernel<5>,
                           (const void*)nchw_to_nhwc_bf16x8_kernel<6>,
                           (const void*)nchw_to_nhwc_bf16x8_kernel<7>,
                           (const void*)nchw_to_nhwc_bf16x8_kernel<8>,
                           (const void*)nchw_to_nhwc_kernel<__nv_bfloat16>,
                           (const void*)nchw_to_nhwc_kernel<float>,
                           (const void*)nchw_to_nhwc_tiled_kernel};
    for (const void* f : fns) {
      const cudaError_t e = cudaFuncSetAttribute(f, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
      if (e != cudaSuccess && attr_err == cudaSuccess) attr_err = e;
    }
  });
  if (attr_err != cudaSuccess) return cuda_fail(attr_err, "cudaFuncSetAttribute(nchw_to_nhwc)");
  if (dt == TBN_BF16 && (H * W) % 8 == 0 && C_pad <= 8 && is_aligned(x, 16) && is_aligned(y, 16)) {
    const int HW8 = static_cast<int>(H * W / 8);
    const int64_t total = N * HW8;
    const unsigned blocks = static_cast<unsigned>((total + 255) / 256);
    const uint4* xv = static_cast<const uint4*>(x);
    uint4* yv = static_cast<uint4*>(y);
    const int c = static_cast<int>(C);
    switch (C_pad) {
      case 1: nchw_to_nhwc_bf16x8_kernel<1><<<blocks, 256, 0, s>>>(xv, c, HW8, total, yv); break;
      case 2: nchw_to_nhwc_bf16x8_kernel<2><<<blocks, 256, 0, s>>>(xv, c, HW8, total, yv); break;
      case 3: nchw_to_nhwc_bf16x8_kernel<3><<<blocks, 256, 0, s>>>(xv, c, HW8, total, yv); break;
      case 4: nchw_to_nhwc_bf16x8_kernel<4><<<blocks, 256, 0, s>>>(xv, c, HW8, total, yv); break;
      case 5: nchw_to_nhwc_bf16x8_kernel<5><<<blocks, 256, 0, s>>>(xv, c, HW8, total, yv); break;
      case 6: nchw_to_nhwc_bf16x8_kernel<6><<<blocks, 256, 0, s>>>(xv, c, HW8, total, yv); break;
      case 7: nchw_to_nhwc_bf16x8_kernel<7><<<blocks, 256, 0, s>>>(xv, c, HW8, total, yv); break;
      default: nchw_to_nhwc_bf16x8_kernel<8><<<blocks, 256, 0, s>>>(xv, c, HW8, total, yv); break;
    }
    return check_launch("nchw_to_nhwc_bf16x8_kernel");
  }
  if (dt == TBN_BF16 && C_pad <= 16) {
    const dim3 grid(static_cast<unsigned>((H * W + kT2Pix - 1) / kT2Pix), static_cast<unsigned>(N));
    nchw_to_nhwc_tiled_kernel<<<grid, 256, kT2Pix * C_pad * 2, s>>>(
        static_cast<const uint16_t*>(x), (int)C, (int)(H * W), (int)C_pad,
        static_cast<uint16_t*>(y));
    return check_launch("nchw_to_nhwc_tiled_kernel");
  }
  const dim3 grid(static_cast<unsigned>((H * W + 255) / 256), static_cast<unsigned>(N));
  if (dt == TBN_BF16)
    nchw_to_nhwc_kernel<__nv_bfloat16><<<grid, 256, 0, s>>>(
        static_cast<const __nv_bfloat16*>(x), (int)C, (int)(H * W), (int)C_pad,
        static_cast<__nv_bfloat16*>(y));
  else
    nchw_to_nhwc_kernel<float><<<grid, 256, 0, s>>>(
        static_cast<const float*>(x), (int)C, (int)(H * W), (int)C_pad, static_cast<float*>(y));
  return check_launch("nchw_to_nhwc_kernel");
}

tbn_status launch_space_to_depth(const void* x, tbn_layout layout, int64_t N, int64_t C,
                                 int64_t H, int64_t W, const S2dGeom& g, int64_t ph, int64_t pw,
                                 void* out, cudaStream_t s) {
  const int64_t pix = kS2dThreads / g.s;
  if (layout == TBN_NCHW && g.s == 4 && C == 3 && g.Ws <= pix) {
    space_to_depth_nchw_kernel<4, 3><<<dim3(static_cast<unsigned>(g.Hs), static_cast<unsigned>(N)),
                                       kS2dThreads, 0, s>>>(
        static_cast<const uint16_t*>(x), (int)H, (int)W, (int)ph, (int)pw, (int)g.Hs, (int)g.Ws,
        static_cast<uint4*>(out));
    return check_launch("space_to_depth_nchw_kernel");
  }
  const dim3 grid(static_cast<unsigned>((g.Ws + pix - 1) / pix), static_cast<unsigned>(g.Hs),
                  static_cast<unsigned>(N));
  const size_t smem = static_cast<size_t>(g.s * pix * g.s * C) * 2;   // <= 512 s C <= 16 KiB
  if (layout == TBN_NCHW)
    space_to_depth_kernel<true><<<grid, kS2dThreads, smem, s>>>(
        static_cast<const uint16_t*>(x), (int)C, (int)H, (int)W, (int)g.s, (int)ph, (int)pw,
        (int)g.Hs, (int)g.Ws, static_cast<uint4*>(out));
  else
    space_to_depth_kernel<false><<<grid, kS2dThreads, smem, s>>>(
        static_cast<const uint16_t*>(x), (int)C, (int)H, (int)W, (int)g.s, (int)ph, (int)pw,
        (int)g.Hs, (int)g.Ws, static_cast<uint4*>(out));
  return check_launch("space_to_depth_kernel");
}

}  // namespace tbn
