// tbn_conv_bwd.cu -- Algorithm 1's TwoBitBackward through a two-bit
// convolution (Eq. 1 with the approximate filters W^ = alpha W~), NHWC bf16:
//
// * Input gradient dx.  The adjoint of a stride-sigma convolution is a
//   stride-1 convolution of dy dilated by sigma (zeros between the rows and
//   columns) with the filters transposed (input and output channels swapped)
//   and mirrored (tap r -> R - 1 - r), padded by R - 1 - pad.  alpha_k is a
//   factor of the reduction index k there, so it goes into the dilated
//   input: dyd[u, v, k] = alpha_k dy[u / sigma, v / sigma, k], rounded to
//   bf16, and the transposed two-bit filters get scale 1.  The convolution
//   then runs on this library's forward kernels (tensor cores whenever the
//   forward pass of that shape would).
// * Filter gradient dW^[k, r, s, c] = sum over (n, p, q) of dy[n, p, q, k]
//   x[n, p sigma - pad + r, q sigma - pad + s, c]: a product of dy^T
//   (K x pixels) and the im2col view of x (pixels x R S C).  Each CTA
//   computes a 64 x 64 tile over a slice of the pixels with fp32 FMA on
//   CUDA cores (bf16 x bf16 products are exact in fp32); a second kernel
//   adds the slices in slice order, so results are bitwise reproducible.
#include <cuda_bf16.h>

#include <algorithm>
#include <cstdint>

#include "tbn_device.cuh"
#include "tbn_internal.h"

namespace tbn {
namespace {

// ------------------------------------------------------------ input grad
// Field (m + 2 s) of code i of a filter row of byte-planar words.
__device__ __forceinline__ uint32_t field_of_code(const uint32_t* row, int64_t i) {
  const uint32_t w = __ldg(row + (i >> 4));
  const int l = static_cast<int>(i & 15);
  const int b = 16 * (l & 1) + (l >> 1);
  return ((w >> b) & 1u) | (((w >> (b + 8)) & 1u) << 1);
}

// codes [K][R][S][C] -> codes_t [C][R][S][K] with the taps mirrored:
// W'[c, r, s, k] = W~[k, R-1-r, S-1-s, c].  One thread per output word.
__global__ void __launch_bounds__(256) transpose_codes_kernel(
    const uint32_t* __restrict__ codes, int64_t wpf_in, uint32_t* __restrict__ out,
    int64_t wpf_out, int K, int C, int R, int S) {
  const int64_t n_out = static_cast<int64_t>(R) * S * K;
  const int64_t total = static_cast<int64_t>(C) * wpf_out;
  for (int64_t wi = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; wi < total;
       wi += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int c = static_cast<int>(wi / wpf_out);
    const int64_t j = wi - static_cast<int64_t>(c) * wpf_out;
    uint32_t o = 0u;
    for (int l = 0; l < 16; ++l) {
      const int64_t i = 16 * j + l;
      if (i >= n_out) break;
      const int k = static_cast<int>(i % K);
      const int64_t rs = i / K;
      const int s = static_cast<int>(rs % S), r = static_cast<int>(rs / S);
      const int64_t src = (static_cast<int64_t>(R - 1 - r) * S + (S - 1 - s)) * C + c;
      const uint32_t f = field_of_code(codes + static_cast<int64_t>(k) * wpf_in, src);
      const int b = 16 * (l & 1) + (l >> 1);
      o |= ((f & 1u) << b) | ((f >> 1) << (b + 8));
    }
    out[wi] = o;
  }
}

// dyd [N][Hd][Wd][K] bf16 = alpha_k dy at (u / sh, v / sw) where both divide,
// zero elsewhere; also ones[c] = 1 for the transposed filters' scales.
__global__ void __launch_bounds__(256) dilate_scale_kernel(
    const __nv_bfloat16* __restrict__ dy, const float* __restrict__ alpha, int N, int P, int Q,
    int K, int Hd, int Wd, int sh, int sw, __nv_bfloat16* __restrict__ dyd,
    float* __restrict__ ones, int C) {
  const int64_t total = static_cast<int64_t>(N) * Hd * Wd * K;
  const int64_t tid = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (tid < C) ones[tid] = 1.0f;
  for (int64_t e = tid; e < total; e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int k = static_cast<int>(e % K);
    int64_t t = e / K;
    const int v = static_cast<int>(t % Wd);
    t /= Wd;
    const int u = static_cast<int>(t % Hd);
    const int n = static_cast<int>(t / Hd);
    float val = 0.0f;
    if (u % sh == 0 && v % sw == 0) {
      const int p = u / sh, q = v / sw;
      if (p < P && q < Q)
        val = __ldg(alpha + k) *
              __bfloat162float(dy[((static_cast<int64_t>(n) * P + p) * Q + q) * K + k]);
    }
    dyd[e] = __float2bfloat16_rn(val);
  }
}

// ------------------------------------------------------------ filter grad
constexpr int kTileM = 64;    // filters k
constexpr int kTileN = 64;    // (r, s, c) columns
constexpr int kChunk = 32;    // pixels per shared-memory chunk
constexpr int kBwdThreads = 256;

struct BwdFilterArgs {
  const __nv_bfloat16* x;
  const __nv_bfloat16* dy;
  float* part;   // [slices][K][RSC]
  int N, C, H, W, K, R, S, sh, sw, ph, pw, P, Q;
  int64_t npix;  // N P Q
  int rsc;       // R S C
  int slices;
  int64_t pix_per_slice;
};

// CTA (bx, by, bz): filters 64 bx .., columns 64 by .., pixels of slice bz.
// Thread (ty, tx) = (tid / 16, tid % 16) accumulates filters 4 ty .. and
// columns 4 tx .. of the tile.
__global__ void __launch_bounds__(kBwdThreads) bwd_filter_kernel(const BwdFilterArgs a) {
  __shared__ __align__(16) float sdy[kChunk][kTileM];
  __shared__ __align__(16) float sx[kChunk][kTileN];
  __shared__ int col_r[kTileN], col_s[kTileN], col_c[kTileN];
  __shared__ int px_n[kChunk], px_h[kChunk], px_w[kChunk];
  const int tid = threadIdx.x;
  const int k0 = blockIdx.x * kTileM, j0 = blockIdx.y * kTileN;
  if (tid < kTileN) {
    const int j = j0 + tid;
    const int c = j % a.C, rs = j / a.C;
    col_c[tid] = c;
    col_s[tid] = rs % a.S;
    col_r[tid] = j < a.rsc ? rs / a.S : -1;   // -1: column past R S C
  }
  const int ty = tid >> 4, tx = tid & 15;
  float acc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.0f;
  const int64_t pbeg = static_cast<int64_t>(blockIdx.z) * a.pix_per_slice;
  const int64_t pend = min(a.npix, pbeg + a.pix_per_slice);
  for (int64_t p0 = pbeg; p0 < pend; p0 += kChunk) {
    __syncthreads();   // previous chunk consumed; column tables written
    if (tid < kChunk) {
      const int64_t pix = p0 + tid;
      int n = -1, h = 0, w = 0;
      if (pix < pend) {
        const int64_t pq = static_cast<int64_t>(a.P) * a.Q;
        n = static_cast<int>(pix / pq);
        const int rem = static_cast<int>(pix - static_cast<int64_t>(n) * pq);
        h = (rem / a.Q) * a.sh - a.ph;
        w = (rem % a.Q) * a.sw - a.pw;
      }
      px_n[tid] = n;
      px_h[tid] = h;
      px_w[tid] = w;
    }
    // dy chunk: 32 pixels x 64 filters (rows of dy are K-contiguous)
    for (int e = tid; e < kChunk * kTileM; e += kBwdThreads) {
      const int pr = e / kTileM, kc = e % kTileM;
      const int64_t pix = p0 + pr;
      const int k = k0 + kc;
      sdy[pr][kc] = (pix < pend && k < a.K) ? __bfloat162float(a.dy[pix * a.K + k]) : 0.0f;
    }
    __syncthreads();   // pixel table ready
    // im2col chunk: 32 pixels x 64 (r, s, c) columns of x
    for (int e = tid; e < kChunk * kTileN; e += kBwdThreads) {
      const int pr = e / kTileN, jc = e % kTileN;
      const int n = px_n[pr], r = col_r[jc];
      float v = 0.0f;
      if (n >= 0 && r >= 0) {
        const int h = px_h[pr] + r, w = px_w[pr] + col_s[jc];
        if (h >= 0 && h < a.H && w >= 0 && w < a.W)
          v = __bfloat162float(
              a.x[((static_cast<int64_t>(n) * a.H + h) * a.W + w) * a.C + col_c[jc]]);
      }
      sx[pr][jc] = v;
    }
    __syncthreads();
#pragma unroll 8
    for (int pr = 0; pr < kChunk; ++pr) {
      const float4 d4 = *reinterpret_cast<const float4*>(&sdy[pr][4 * ty]);
      const float4 x4 = *reinterpret_cast<const float4*>(&sx[pr][4 * tx]);
      const float dv[4] = {d4.x, d4.y, d4.z, d4.w}, xv[4] = {x4.x, x4.y, x4.z, x4.w};
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(dv[i], xv[j], acc[i][j]);
    }
  }
  float* part = a.part + static_cast<int64_t>(blockIdx.z) * a.K * a.rsc;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int k = k0 + 4 * ty + i;
    if (k >= a.K) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int jj = j0 + 4 * tx + j;
      if (jj < a.rsc) part[static_cast<int64_t>(k) * a.rsc + jj] = acc[i][j];
    }
  }
}

// dw[e] = sum of the slices' partial values, in slice order.
__global__ void __launch_bounds__(256) bwd_filter_reduce_kernel(const float* __restrict__ part,
                                                                int slices, int64_t count,
                                                                float* __restrict__ dw) {
  for (int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; e < count;
       e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    float s = part[e];
    for (int z = 1; z < slices; ++z) s += part[static_cast<int64_t>(z) * count + e];
    dw[e] = s;
  }
}

size_t align256(size_t v) { return (v + 255) & ~static_cast<size_t>(255); }

struct BwdDataPlan {
  int64_t Hd, Wd, pad_h, pad_w, wpf_t;
  size_t off_ones, off_dyd, bytes;
};

BwdDataPlan plan_bwd_data(const BwdConvShape& p) {
  BwdDataPlan b{};
  b.pad_h = p.R - 1 - p.ph;
  b.pad_w = p.S - 1 - p.pw;
  b.Hd = p.H + 2 * p.ph - p.R + 1;
  b.Wd = p.W + 2 * p.pw - p.S + 1;
  b.wpf_t = (p.R * p.S * p.K + 15) / 16;
  b.off_ones = align256(static_cast<size_t>(p.C) * b.wpf_t * 4);
  b.off_dyd = b.off_ones + align256(static_cast<size_t>(p.C) * 4);
  b.bytes = b.off_dyd + align256(static_cast<size_t>(p.N) * b.Hd * b.Wd * p.K * 2);
  return b;
}

int bwd_filter_slices(const BwdConvShape& p) {
  const int64_t tiles = ((p.K + kTileM - 1) / kTileM) * ((p.R * p.S * p.C + kTileN - 1) / kTileN);
  const int64_t want = 4 * static_cast<int64_t>(device_sm_count());
  const int64_t npix = p.N * p.P * p.Q;
  int64_t s = std::max<int64_t>(1, want / std::max<int64_t>(tiles, 1));
  s = std::min<int64_t>(s, std::max<int64_t>(1, npix / (4 * kChunk)));
  return static_cast<int>(std::min<int64_t>(s, 64));
}

}  // namespace

const char* bwd_shape_reason(const BwdConvShape& p) {
  if (p.ph > p.R - 1 || p.pw > p.S - 1) return "backward needs pad <= kernel size - 1";
  if (p.N * p.H * p.W * p.C >= (1ll << 40) || p.N * p.P * p.Q * p.K >= (1ll << 40))
    return "backward: tensor too large";
  if (p.C >= (1 << 30) || p.K >= (1 << 30) || p.R * p.S * p.C >= (1ll << 30) ||
      p.R * p.S * p.K >= (1ll << 30))
    return "backward: filter too large";
  return "";
}

size_t bwd_data_workspace_bytes(const BwdConvShape& p) { return plan_bwd_data(p).bytes; }

tbn_status launch_bwd_data(const BwdConvShape& p, const void* dy, const uint32_t* codes,
                           const float* alpha, void* dx, tbn_dtype dxdt, void* workspace,
                           cudaStream_t s) {
  const BwdDataPlan b = plan_bwd_data(p);
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  uint32_t* codes_t = reinterpret_cast<uint32_t*>(ws);
  float* ones = reinterpret_cast<float*>(ws + b.off_ones);
  __nv_bfloat16* dyd = reinterpret_cast<__nv_bfloat16*>(ws + b.off_dyd);
  const int64_t wpf_in = (p.R * p.S * p.C + 15) / 16;
  {
    const int64_t total = p.C * b.wpf_t;
    const int64_t blocks = std::min<int64_t>((total + 255) / 256, 65536);
    transpose_codes_kernel<<<static_cast<unsigned>(blocks), 256, 0, s>>>(
        codes, wpf_in, codes_t, b.wpf_t, static_cast<int>(p.K), static_cast<int>(p.C),
        static_cast<int>(p.R), static_cast<int>(p.S));
    const tbn_status st = check_launch("transpose_codes_kernel");
    if (st != TBN_OK) return st;
  }
  {
    const int64_t total = p.N * b.Hd * b.Wd * p.K;
    const int64_t blocks =
        std::max<int64_t>(1, std::min<int64_t>((std::max<int64_t>(total, p.C) + 255) / 256,
                                               static_cast<int64_t>(device_sm_count()) * 16));
    dilate_scale_kernel<<<static_cast<unsigned>(blocks), 256, 0, s>>>(
        static_cast<const __nv_bfloat16*>(dy), alpha, static_cast<int>(p.N),
        static_cast<int>(p.P), static_cast<int>(p.Q), static_cast<int>(p.K),
        static_cast<int>(b.Hd), static_cast<int>(b.Wd), static_cast<int>(p.sh),
        static_cast<int>(p.sw), dyd, ones, static_cast<int>(p.C));
    const tbn_status st = check_launch("dilate_scale_kernel");
    if (st != TBN_OK) return st;
  }
  // dx = the forward convolution of dyd with the transposed filters
  ConvProblem q{};
  q.N = p.N; q.C = p.K; q.H = b.Hd; q.W = b.Wd; q.K = p.C; q.R = p.R; q.S = p.S;
  q.sh = 1; q.sw = 1; q.ph = b.pad_h; q.pw = b.pad_w;
  q.P = b.Hd + 2 * b.pad_h - p.R + 1;
  q.Q = b.Wd + 2 * b.pad_w - p.S + 1;
  q.layout = TBN_NHWC;
  q.xdt = TBN_BF16;
  q.ydt = dxdt;
  q.x = dyd;
  q.codes = codes_t;
  q.alpha = ones;
  q.y = dx;
  q.relu = 0;
  q.residual = nullptr;
  q.pool = 0;
  return run_conv_auto(q, s);
}

size_t bwd_filter_workspace_bytes(const BwdConvShape& p) {
  const int slices = bwd_filter_slices(p);
  return align256(static_cast<size_t>(slices) * p.K * p.R * p.S * p.C * 4);
}

tbn_status launch_bwd_filter(const BwdConvShape& p, const void* x, const void* dy, float* dw,
                             void* workspace, cudaStream_t s) {
  BwdFilterArgs a{};
  a.x = static_cast<const __nv_bfloat16*>(x);
  a.dy = static_cast<const __nv_bfloat16*>(dy);
  a.part = static_cast<float*>(workspace);
  a.N = static_cast<int>(p.N); a.C = static_cast<int>(p.C); a.H = static_cast<int>(p.H);
  a.W = static_cast<int>(p.W); a.K = static_cast<int>(p.K); a.R = static_cast<int>(p.R);
  a.S = static_cast<int>(p.S); a.sh = static_cast<int>(p.sh); a.sw = static_cast<int>(p.sw);
  a.ph = static_cast<int>(p.ph); a.pw = static_cast<int>(p.pw); a.P = static_cast<int>(p.P);
  a.Q = static_cast<int>(p.Q);
  a.npix = p.N * p.P * p.Q;
  a.rsc = static_cast<int>(p.R * p.S * p.C);
  a.slices = bwd_filter_slices(p);
  a.pix_per_slice = (a.npix + a.slices - 1) / a.slices;
  const dim3 grid(static_cast<unsigned>((p.K + kTileM - 1) / kTileM),
                  static_cast<unsigned>((a.rsc + kTileN - 1) / kTileN),
                  static_cast<unsigned>(a.slices));
  if (grid.y > 65535) return fail(TBN_ERR_UNSUPPORTED, "backward filter: R S C too large");
  bwd_filter_kernel<<<grid, kBwdThreads, 0, s>>>(a);
  tbn_status st = check_launch("bwd_filter_kernel");
  if (st != TBN_OK) return st;
  const int64_t count = p.K * a.rsc;
  const int64_t blocks = std::min<int64_t>((count + 255) / 256, 65536);
  bwd_filter_reduce_kernel<<<static_cast<unsigned>(blocks), 256, 0, s>>>(a.part, a.slices, count,
                                                                          dw);
  return check_launch("bwd_filter_reduce_kernel");
}

}  // namespace tbn
