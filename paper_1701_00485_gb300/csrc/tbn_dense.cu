// tbn_dense.cu -- the full-precision layers a two-bit network keeps around
// its TBN layers (network glue, not the paper's method): the first
// convolution with fp32 weights, the global average pool and the last
// fully-connected layer with fp32 weights (the ResNet-18 workload keeps
// both ends in full precision).  All arithmetic is fp32 on the CUDA cores:
// x * w products are rounded to fp32 and accumulated in fp32, which is what
// "kept in fp32" means for these layers.
//
// Dense convolution: a persistent CTA takes tiles of 4 output rows x 32
// output columns of one image for 64 filters.  Per chunk of input channels it
// stages the fp32 weights [tap][64 filters] and the input patch the tile
// reads (zero outside the image) in shared memory; each warp owns 8
// filters (its weight reads are broadcasts), each lane one output column of
// the four rows (4 pixels x 8 filters = 32 accumulators per thread), so a
// tap costs 4 activation reads, 2 vector weight reads and 32 FMAs.
#include <cuda_bf16.h>

#include <algorithm>
#include <cstdint>
#include <mutex>

#include "tbn_device.cuh"
#include "tbn_internal.h"

namespace tbn {
namespace {

constexpr int kDcRows = 4;      // output rows per tile
constexpr int kDcCols = 32;     // output columns per tile (= lanes)
constexpr int kDcFilt = 64;     // filters per CTA (8 warps x 8)
constexpr int kDcThreads = 256;
constexpr int kDcSmemMax = 200 * 1024;

template <typename T>
__device__ __forceinline__ float ld_f32(const T* p, int64_t i);
template <>
__device__ __forceinline__ float ld_f32<float>(const float* p, int64_t i) { return __ldg(p + i); }
template <>
__device__ __forceinline__ float ld_f32<__nv_bfloat16>(const __nv_bfloat16* p, int64_t i) {
  return __bfloat162float(p[i]);
}

struct DenseConvArgs {
  int N, C, H, W, K, R, S, sh, sw, ph, pw, P, Q;
  int cc;            // input channels per chunk
  int prows, pcols;  // staged patch extent
  int tiles_q, tiles_p;
  const void* x;
  const float* w;    // [K][C][R][S]
  void* y;
  int relu;
  int stage_out;     // bf16 NHWC output, K % 8 == 0, y 16-byte aligned: the tile's
                     // outputs go through shared memory and leave as 16-byte stores
};

// kXNhwc: x is [N][H][W][C] (else [N][C][H][W]); kYNhwc: y is [N][P][Q][K]
// (else [N][K][P][Q]).  kR, kS, kSH, kSW > 0 fix the kernel extent and
// stride at compile time (the 7x7/2 first layer of ResNet-18): the tap loop
// unrolls and every shared-memory address is an immediate offset; 0 = taken
// from the arguments.
template <typename TX, typename TY, bool kXNhwc, bool kYNhwc, int kR = 0, int kS = 0,
          int kSH = 0, int kSW = 0>
__global__ void __launch_bounds__(kDcThreads) dense_conv_kernel(const DenseConvArgs a) {
  extern __shared__ __align__(16) float dsm[];
  const int RS = a.R * a.S;
  float* s_w = dsm;                                   // [cc * R * S][64]
  float* s_x = dsm + static_cast<size_t>(a.cc) * RS * kDcFilt;   // [cc][prows][pcols]
  // staged outputs [4 rows x 32 columns][64 filters] bf16, 128 bytes per
  // pixel with its 16-byte filter chunks permuted by the pixel's low 3 bits
  // (after the weights and the patch, rounded up to 128 bytes)
  uint8_t* s_o = reinterpret_cast<uint8_t*>(
      dsm + ((static_cast<size_t>(a.cc) * (RS * kDcFilt + a.prows * a.pcols) + 31) & ~size_t(31)));
  const TX* __restrict__ x = static_cast<const TX*>(a.x);

  const int k0 = blockIdx.y * kDcFilt;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int f0 = warp * 8;
  const int R = kR > 0 ? kR : a.R, S = kS > 0 ? kS : a.S;
  const int sh = kSH > 0 ? kSH : a.sh, sw = kSW > 0 ? kSW : a.sw;
  const int patch = a.prows * a.pcols;
  const int ntiles = a.N * a.tiles_p * a.tiles_q;
  // column stride 2 (compile time): each patch row keeps its even columns,
  // then its odd ones, so that for a tap the 32 lanes (output columns) read
  // 32 consecutive words instead of every other one (no bank conflicts)
  constexpr bool kSplit = kSW == 2;
  const int half = (a.pcols + 1) / 2;
  // all input channels in one chunk: the CTA's weights are staged once and
  // serve every tile it takes (persistent grid)
  const bool w_once = a.cc >= a.C;
  auto load_weights = [&](int c0, int cn) {
    for (int i = threadIdx.x; i < cn * RS * kDcFilt; i += kDcThreads) {
      const int f = i % kDcFilt, tap = i / kDcFilt;
      const int k = k0 + f;
      s_w[i] = k < a.K ? __ldg(a.w + (static_cast<int64_t>(k) * a.C + c0) * RS + tap) : 0.0f;
    }
  };
  if (w_once) load_weights(0, a.C);
  TY* __restrict__ y = static_cast<TY*>(a.y);

  for (int t0 = blockIdx.x; t0 < ntiles; t0 += gridDim.x) {
    int t = t0;
    const int tq = t % a.tiles_q;
    t /= a.tiles_q;
    const int tp = t % a.tiles_p;
    const int b = t / a.tiles_p;
    const int q0 = tq * kDcCols, p0 = tp * kDcRows;
    const int h_base = p0 * sh - a.ph, w_base = q0 * sw - a.pw;

    float acc[kDcRows][8];
#pragma unroll
    for (int i = 0; i < kDcRows; ++i)
#pragma unroll
      for (int f = 0; f < 8; ++f) acc[i][f] = 0.0f;

    for (int c0 = 0; c0 < a.C; c0 += a.cc) {
      const int cn = min(a.cc, a.C - c0);
      __syncthreads();   // the previous chunk / tile is done with the buffers
      if (!w_once) load_weights(c0, cn);
      // input patch of this channel chunk, zero outside the image
      for (int i = threadIdx.x; i < cn * patch; i += kDcThreads) {
        const int c = i / patch, rem = i - c * patch;
        const int pr = rem / a.pcols, pc = rem - pr * a.pcols;
        const int h = h_base + pr, w = w_base + pc;
        float v = 0.0f;
        if (h >= 0 && h < a.H && w >= 0 && w < a.W) {
          const int64_t o = kXNhwc
                                ? ((static_cast<int64_t>(b) * a.H + h) * a.W + w) * a.C + c0 + c
                                : ((static_cast<int64_t>(b) * a.C + c0 + c) * a.H + h) * a.W + w;
          v = ld_f32<TX>(x, o);
        }
        if constexpr (kSplit)
          s_x[c * patch + pr * a.pcols + ((pc & 1) ? half + (pc >> 1) : (pc >> 1))] = v;
        else
          s_x[i] = v;
      }
      __syncthreads();
      for (int c = 0; c < cn; ++c) {
        const float* xc = s_x + c * patch + (kSplit ? lane : lane * sw);
#pragma unroll 1
        for (int r = 0; r < R; ++r) {
          const float* xr = xc + r * a.pcols;
          const float* wr = s_w + ((c * R + r) * S) * kDcFilt + f0;
#pragma unroll
          for (int s = 0; s < S; ++s) {
            const float4 w0 = *reinterpret_cast<const float4*>(wr + s * kDcFilt);
            const float4 w1 = *reinterpret_cast<const float4*>(wr + s * kDcFilt + 4);
#pragma unroll
            for (int i = 0; i < kDcRows; ++i) {
              const float xv =
                  kSplit ? xr[i * sh * a.pcols + (s & 1) * half + (s >> 1)] : xr[i * sh * a.pcols + s];
              acc[i][0] = fmaf(xv, w0.x, acc[i][0]);
              acc[i][1] = fmaf(xv, w0.y, acc[i][1]);
              acc[i][2] = fmaf(xv, w0.z, acc[i][2]);
              acc[i][3] = fmaf(xv, w0.w, acc[i][3]);
              acc[i][4] = fmaf(xv, w1.x, acc[i][4]);
              acc[i][5] = fmaf(xv, w1.y, acc[i][5]);
              acc[i][6] = fmaf(xv, w1.z, acc[i][6]);
              acc[i][7] = fmaf(xv, w1.w, acc[i][7]);
            }
          }
        }
      }
    }

    if constexpr (kYNhwc && sizeof(TY) == 2) {
      if (a.stage_out) {
        // lane = output column, this warp's 8 filters = one 16-byte chunk
        const uint32_t o_base = smem_addr(s_o);
#pragma unroll
        for (int i = 0; i < kDcRows; ++i) {
          float v[8];
#pragma unroll
          for (int f = 0; f < 8; ++f) v[f] = a.relu ? fmaxf(acc[i][f], 0.0f) : acc[i][f];
          const int px = i * kDcCols + lane;
          const uint32_t addr = o_base + static_cast<uint32_t>(px * 128 + ((warp ^ (lane & 7)) << 4));
          asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr),
                       "r"(pack_bf16x2(v[0], v[1])), "r"(pack_bf16x2(v[2], v[3])),
                       "r"(pack_bf16x2(v[4], v[5])), "r"(pack_bf16x2(v[6], v[7]))
                       : "memory");
        }
        __syncthreads();
        // 4 x 32 pixels x 8 chunks of 8 filters: consecutive threads take a
        // pixel's chunks, so a warp writes four whole 128-byte pixel rows
        for (int c = threadIdx.x; c < kDcRows * kDcCols * 8; c += kDcThreads) {
          const int px = c >> 3, ch = c & 7;
          const int col = px % kDcCols, p = p0 + px / kDcCols, q = q0 + col;
          const int k = k0 + ch * 8;
          if (p >= a.P || q >= a.Q || k >= a.K) continue;
          uint4 v;
          asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
                       : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                       : "r"(o_base + static_cast<uint32_t>(px * 128 + ((ch ^ (col & 7)) << 4)))
                       : "memory");
          *reinterpret_cast<uint4*>(y + ((static_cast<int64_t>(b) * a.P + p) * a.Q + q) * a.K + k) = v;
        }
        continue;
      }
    }
    const int q = q0 + lane;
    if (q >= a.Q) continue;
#pragma unroll
    for (int i = 0; i < kDcRows; ++i) {
      const int p = p0 + i;
      if (p >= a.P) continue;
#pragma unroll
      for (int f = 0; f < 8; ++f) {
        const int k = k0 + f0 + f;
        if (k >= a.K) continue;
        float v = acc[i][f];
        if (a.relu) v = fmaxf(v, 0.0f);
        const int64_t o = kYNhwc ? ((static_cast<int64_t>(b) * a.P + p) * a.Q + q) * a.K + k
                                 : ((static_cast<int64_t>(b) * a.K + k) * a.P + p) * a.Q + q;
        if constexpr (sizeof(TY) == 2)
          y[o] = __float2bfloat16_rn(v);
        else
          y[o] = v;
      }
    }
  }
}

template <typename TX, typename TY, bool kXNhwc, bool kYNhwc, int kR = 0, int kS = 0,
          int kSH = 0, int kSW = 0>
tbn_status launch_dense_conv_t(const DenseConvArgs& a, size_t smem, cudaStream_t s) {
  auto kern = dense_conv_kernel<TX, TY, kXNhwc, kYNhwc, kR, kS, kSH, kSW>;
  static std::once_flag once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(once, [&] {
    attr_err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kDcSmemMax);
  });
  if (attr_err != cudaSuccess) return cuda_fail(attr_err, "cudaFuncSetAttribute(dense_conv_kernel)");
  const int64_t tiles = static_cast<int64_t>(a.N) * a.tiles_p * a.tiles_q;
  const int64_t gy = (a.K + kDcFilt - 1) / kDcFilt;
  if (tiles > 0x7fffffffLL || gy > 65535)
    return fail(TBN_ERR_UNSUPPORTED, "dense conv: grid too large");
  // persistent: as many CTAs as fit at once (the weights are staged once per CTA)
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kDcThreads, smem) !=
          cudaSuccess ||
      per_sm < 1)
    per_sm = 1;
  const int64_t slots = static_cast<int64_t>(device_sm_count()) * per_sm;
  const int64_t gx = std::max<int64_t>(1, std::min<int64_t>(tiles, (slots + gy - 1) / gy));
  kern<<<dim3(static_cast<unsigned>(gx), static_cast<unsigned>(gy)), kDcThreads, smem, s>>>(a);
  return check_launch("dense_conv_kernel");
}

template <typename TX, typename TY>
tbn_status launch_dense_conv_l(const DenseConvArgs& a, size_t smem, bool xn, bool yn,
                               cudaStream_t s) {
  if (!xn && yn && a.R == 7 && a.S == 7 && a.sh == 2 && a.sw == 2)
    return launch_dense_conv_t<TX, TY, false, true, 7, 7, 2, 2>(a, smem, s);
  if (xn && yn) return launch_dense_conv_t<TX, TY, true, true>(a, smem, s);
  if (!xn && yn) return launch_dense_conv_t<TX, TY, false, true>(a, smem, s);
  if (!xn && !yn) return launch_dense_conv_t<TX, TY, false, false>(a, smem, s);
  return fail(TBN_ERR_UNSUPPORTED, "dense conv: NHWC input with NCHW output");
}

// ---------------------------------------------------------------- avg pool
// One thread per (image, channel): the mean over H*W in fp32, pixels in order.
template <typename TX, typename TY>
__global__ void __launch_bounds__(256) avgpool_global_nhwc_kernel(const TX* __restrict__ x,
                                                                  int64_t N, int64_t HW,
                                                                  int64_t C, float inv,
                                                                  TY* __restrict__ y) {
  const int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x;
  if (i >= N * C) return;
  const int64_t b = i / C, c = i - b * C;
  const TX* p = x + b * HW * C + c;
  float acc = 0.0f;
  for (int64_t j = 0; j < HW; ++j) acc += ld_f32<TX>(p, j * C);
  const float v = acc * inv;
  if constexpr (sizeof(TY) == 2)
    y[i] = __float2bfloat16_rn(v);
  else
    y[i] = v;
}

// ---------------------------------------------------------------- dense linear
// y[b, k] = sum_j x[b, j] w[k, j]: a CTA computes 64 rows (b) x 64 columns (k),
// 256 threads with 4 x 4 outputs each, K_in in chunks of 32 staged in shared
// memory (both operands transposed to [j][.] so the inner loop reads rows).
constexpr int kLinTile = 64, kLinK = 32;

template <typename TY>
__global__ void __launch_bounds__(256) dense_linear_kernel(const float* __restrict__ x,
                                                           int B, int Kin,
                                                           const float* __restrict__ w,
                                                           int Kout, TY* __restrict__ y,
                                                           int relu) {
  __shared__ float sx[kLinK][kLinTile + 4];
  __shared__ float sw[kLinK][kLinTile + 4];
  const int b0 = blockIdx.y * kLinTile, k0 = blockIdx.x * kLinTile;
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  float acc[4][4] = {};
  for (int j0 = 0; j0 < Kin; j0 += kLinK) {
    __syncthreads();
    for (int i = threadIdx.x; i < kLinK * kLinTile; i += 256) {
      const int row = i / kLinK, j = i % kLinK;
      const int gb = b0 + row, gk = k0 + row, gj = j0 + j;
      sx[j][row] = (gb < B && gj < Kin) ? __ldg(x + static_cast<int64_t>(gb) * Kin + gj) : 0.0f;
      sw[j][row] = (gk < Kout && gj < Kin) ? __ldg(w + static_cast<int64_t>(gk) * Kin + gj) : 0.0f;
    }
    __syncthreads();
#pragma unroll 8
    for (int j = 0; j < kLinK; ++j) {
      float xv[4], wv[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        xv[u] = sx[j][ty * 4 + u];
        wv[u] = sw[j][tx * 4 + u];
      }
#pragma unroll
      for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int v = 0; v < 4; ++v) acc[u][v] = fmaf(xv[u], wv[v], acc[u][v]);
    }
  }
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const int gb = b0 + ty * 4 + u;
    if (gb >= B) continue;
#pragma unroll
    for (int v = 0; v < 4; ++v) {
      const int gk = k0 + tx * 4 + v;
      if (gk >= Kout) continue;
      float o = acc[u][v];
      if (relu) o = fmaxf(o, 0.0f);
      if constexpr (sizeof(TY) == 2)
        y[static_cast<int64_t>(gb) * Kout + gk] = __float2bfloat16_rn(o);
      else
        y[static_cast<int64_t>(gb) * Kout + gk] = o;
    }
  }
}

}  // namespace

tbn_status launch_dense_conv(const ConvProblem& p, const float* w, cudaStream_t s) {
  DenseConvArgs a{};
  a.N = (int)p.N; a.C = (int)p.C; a.H = (int)p.H; a.W = (int)p.W; a.K = (int)p.K;
  a.R = (int)p.R; a.S = (int)p.S; a.sh = (int)p.sh; a.sw = (int)p.sw;
  a.ph = (int)p.ph; a.pw = (int)p.pw; a.P = (int)p.P; a.Q = (int)p.Q;
  a.x = p.x; a.w = w; a.y = p.y; a.relu = p.relu;
  a.prows = (kDcRows - 1) * a.sh + a.R;
  a.pcols = (kDcCols - 1) * a.sw + a.S;
  const int64_t per_c = static_cast<int64_t>(a.R) * a.S * kDcFilt + int64_t(a.prows) * a.pcols;
  const int64_t cc = std::min<int64_t>(a.C, (kDcSmemMax / 4) / per_c);
  if (cc < 1) return fail(TBN_ERR_UNSUPPORTED, "dense conv: kernel or stride too large");
  a.cc = static_cast<int>(cc);
  a.tiles_q = static_cast<int>((p.Q + kDcCols - 1) / kDcCols);
  a.tiles_p = static_cast<int>((p.P + kDcRows - 1) / kDcRows);
  const bool xn = p.layout == TBN_NHWC, yn = p.layout != TBN_NCHW;
  const bool xb = p.xdt == TBN_BF16, yb = p.ydt == TBN_BF16;
  constexpr size_t kStageOutBytes = kDcRows * kDcCols * kDcFilt * 2;
  const size_t in_bytes = ((static_cast<size_t>(cc * per_c) + 31) & ~size_t(31)) * 4;
  a.stage_out = (yn && yb && p.K % 8 == 0 && is_aligned(p.y, 16) &&
                 in_bytes + kStageOutBytes <= static_cast<size_t>(kDcSmemMax))
                    ? 1 : 0;
  const size_t smem = a.stage_out ? in_bytes + kStageOutBytes : static_cast<size_t>(cc * per_c) * 4;
  using bf = __nv_bfloat16;
  if (xb && yb) return launch_dense_conv_l<bf, bf>(a, smem, xn, yn, s);
  if (xb && !yb) return launch_dense_conv_l<bf, float>(a, smem, xn, yn, s);
  if (!xb && yb) return launch_dense_conv_l<float, bf>(a, smem, xn, yn, s);
  return launch_dense_conv_l<float, float>(a, smem, xn, yn, s);
}

tbn_status launch_avgpool_global_nhwc(const void* x, tbn_dtype xdt, int64_t N, int64_t H,
                                      int64_t W, int64_t C, void* y, tbn_dtype ydt,
                                      cudaStream_t s) {
  const int64_t total = N * C;
  const unsigned blocks = static_cast<unsigned>((total + 255) / 256);
  const float inv = 1.0f / static_cast<float>(H * W);
  using bf = __nv_bfloat16;
  if (xdt == TBN_BF16 && ydt == TBN_F32)
    avgpool_global_nhwc_kernel<bf, float><<<blocks, 256, 0, s>>>(
        static_cast<const bf*>(x), N, H * W, C, inv, static_cast<float*>(y));
  else if (xdt == TBN_BF16)
    avgpool_global_nhwc_kernel<bf, bf><<<blocks, 256, 0, s>>>(
        static_cast<const bf*>(x), N, H * W, C, inv, static_cast<bf*>(y));
  else if (ydt == TBN_F32)
    avgpool_global_nhwc_kernel<float, float><<<blocks, 256, 0, s>>>(
        static_cast<const float*>(x), N, H * W, C, inv, static_cast<float*>(y));
  else
    avgpool_global_nhwc_kernel<float, bf><<<blocks, 256, 0, s>>>(
        static_cast<const float*>(x), N, H * W, C, inv, static_cast<bf*>(y));
  return check_launch("avgpool_global_nhwc_kernel");
}

tbn_status launch_dense_linear(const float* x, int64_t B, int64_t K_in, const float* w,
                               int64_t K_out, void* y, tbn_dtype ydt, int relu,
                               cudaStream_t s) {
  const int64_t gx = (K_out + kLinTile - 1) / kLinTile, gy = (B + kLinTile - 1) / kLinTile;
  if (gx > 0x7fffffffLL || gy > 65535) return fail(TBN_ERR_UNSUPPORTED, "dense linear: grid too large");
  const dim3 grid(static_cast<unsigned>(gx), static_cast<unsigned>(gy));
  if (ydt == TBN_BF16)
    dense_linear_kernel<__nv_bfloat16><<<grid, 256, 0, s>>>(
        x, (int)B, (int)K_in, w, (int)K_out, static_cast<__nv_bfloat16*>(y), relu);
  else
    dense_linear_kernel<float><<<grid, 256, 0, s>>>(x, (int)B, (int)K_in, w, (int)K_out,
                                                    static_cast<float*>(y), relu);
  return check_launch("dense_linear_kernel");
}

}  // namespace tbn
