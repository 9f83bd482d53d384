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
//   computes a tile over a slice of the pixels: 128 x 128 on tcgen05 with
//   the accumulator in tensor memory when K and C are multiples of 8, else
//   64 x 64 on mma.sync (bf16 products exact, fp32 accumulation); a second
//   kernel adds the slices in a fixed order, so results are bitwise
//   reproducible.
#include <cuda_bf16.h>

#include <algorithm>
#include <cstdint>
#include <mutex>

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
    if (K % 16 == 0) {
      // the word's 16 codes share the tap (r, s); input channels k0 .. k0+15
      const int64_t i0 = 16 * j;
      const int k0 = static_cast<int>(i0 % K);
      const int64_t rs = i0 / K;
      const int s = static_cast<int>(rs % S), r = static_cast<int>(rs / S);
      const int64_t src = (static_cast<int64_t>(R - 1 - r) * S + (S - 1 - s)) * C + c;
#pragma unroll
      for (int l = 0; l < 16; ++l) {
        const uint32_t f = field_of_code(codes + static_cast<int64_t>(k0 + l) * wpf_in, src);
        const int b = 16 * (l & 1) + (l >> 1);
        o |= ((f & 1u) << b) | ((f >> 1) << (b + 8));
      }
      out[wi] = o;
      continue;
    }
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
// zero elsewhere; also ones[c] = 1 for the transposed filters' scales.  One
// thread per output pixel, eight channels per step (16-byte loads and
// stores when K % 8 == 0 and dy, dyd are 16-byte aligned).
__global__ void __launch_bounds__(256) dilate_scale_kernel(
    const __nv_bfloat16* __restrict__ dy, const float* __restrict__ alpha, int N, int P, int Q,
    int K, int Hd, int Wd, int sh, int sw, __nv_bfloat16* __restrict__ dyd,
    float* __restrict__ ones, int C, int vec) {
  const int64_t npix = static_cast<int64_t>(N) * Hd * Wd;
  const int64_t tid = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  const int64_t nthreads = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t c = tid; c < C; c += nthreads) ones[c] = 1.0f;
  // one item = 8 channels of one pixel (vec) or one pixel (scalar path)
  const int per_pix = vec ? K / 8 : 1;
  for (int64_t e = tid; e < npix * per_pix; e += nthreads) {
    const int64_t pix = e / per_pix;
    const int kv = static_cast<int>(e - pix * per_pix);
    const int v = static_cast<int>(pix % Wd);
    const int64_t t = pix / Wd;
    const int u = static_cast<int>(t % Hd);
    const int n = static_cast<int>(t / Hd);
    const bool hit = u % sh == 0 && v % sw == 0 && u / sh < P && v / sw < Q;
    const __nv_bfloat16* src =
        hit ? dy + ((static_cast<int64_t>(n) * P + u / sh) * Q + v / sw) * K : nullptr;
    __nv_bfloat16* dst = dyd + pix * K;
    if (vec) {
      const int k = 8 * kv;
      uint4 o = make_uint4(0u, 0u, 0u, 0u);
      if (hit) {
        const uint4 i4 = __ldg(reinterpret_cast<const uint4*>(src + k));
        const float4 a0 = __ldg(reinterpret_cast<const float4*>(alpha + k));
        const float4 a1 = __ldg(reinterpret_cast<const float4*>(alpha + k + 4));
        const float al[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
        const uint32_t iw[4] = {i4.x, i4.y, i4.z, i4.w};
        uint32_t ow[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&iw[q]));
          const __nv_bfloat162 r = __floats2bfloat162_rn(al[2 * q] * f.x, al[2 * q + 1] * f.y);
          ow[q] = *reinterpret_cast<const uint32_t*>(&r);
        }
        o = make_uint4(ow[0], ow[1], ow[2], ow[3]);
      }
      *reinterpret_cast<uint4*>(dst + k) = o;
    } else {
      for (int k = 0; k < K; ++k)
        dst[k] = __float2bfloat16_rn(hit ? __ldg(alpha + k) * __bfloat162float(src[k]) : 0.0f);
    }
  }
}

// ------------------------------------------------------------ filter grad
constexpr int kTileM = 64;    // filters k
constexpr int kTileN = 64;    // (r, s, c) columns
constexpr int kChunk = 64;    // pixels per shared-memory chunk
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
  int dy_vec, x_vec;   // 16-byte loads possible (K % 8 == 0 / C % 8 == 0, aligned)
  uint32_t* err;       // device error word (bounded waits)
  int part_vec;        // 16-byte partial stores possible (rsc % 4 == 0, aligned)
};

__device__ __forceinline__ void ldsm_x4_trans(uint32_t (&r)[4], uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr)
               : "memory");
}

__device__ __forceinline__ void mma_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                          uint32_t b1) {
  asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
      "{%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Pixel index n P Q + p Q + q of one tile row, advanced by kChunk pixels per
// chunk with the carries of kChunk = dn P Q + dp Q + dq (no divisions in
// the loop).  Rows past the slice keep advancing but are never loaded.
struct PixelRow {
  int64_t pix;
  int n, p, q;
  __device__ __forceinline__ void init(int64_t pixel, int P, int Q) {
    pix = pixel;
    const int64_t pq = static_cast<int64_t>(P) * Q;
    n = static_cast<int>(pixel / pq);
    const int rem = static_cast<int>(pixel - static_cast<int64_t>(n) * pq);
    p = rem / Q;
    q = rem - p * Q;
  }
  __device__ __forceinline__ void advance(int dn, int dp, int dq, int P, int Q) {
    pix += kChunk;
    q += dq;
    if (q >= Q) { q -= Q; ++p; }
    p += dp;
    if (p >= P) { p -= P; ++n; }
    n += dn;
  }
};

// Shared tiles are [pixel][64 bf16]: 128-byte rows of eight 16-byte chunks,
// chunk c of row r stored at c ^ (r & 7) (conflict-free ldmatrix).
__device__ __forceinline__ uint32_t tile_off(int row, int chunk) {
  return static_cast<uint32_t>(row * 128 + ((chunk ^ (row & 7)) << 4));
}

// CTA (bx, by, bz): filters 64 bx .., columns 64 by .., pixels of slice bz.
// dW^ tile = dy^T (filters x pixels) * im2col(x) (pixels x columns) on
// mma.m16n8k16 (bf16 products exact, fp32 accumulation): warp w owns
// filters 16 (w % 4) .. and columns 32 (w / 4) .. (four 8-column n-tiles).
// Both operands come from the pixel-major tiles by ldmatrix.trans.  Thread
// i fills chunk i % 8 of pixel row i / 8 (and row i / 8 + 32) of both
// tiles; the next chunk's loads are issued before the current MMAs.
__global__ void __launch_bounds__(kBwdThreads, 4) bwd_filter_kernel(const BwdFilterArgs a) {
  __shared__ __align__(128) uint8_t sdy[kChunk * 128];
  __shared__ __align__(128) uint8_t sx[kChunk * 128];
  __shared__ int col_r[kTileN], col_s[kTileN], col_c[kTileN];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int k0 = blockIdx.x * kTileM, j0 = blockIdx.y * kTileN;
  if (tid < kTileN) {
    const int j = j0 + tid;
    const int c = j % a.C, rs = j / a.C;
    col_c[tid] = c;
    col_s[tid] = rs % a.S;
    col_r[tid] = j < a.rsc ? rs / a.S : -1;   // -1: column past R S C
  }
  __syncthreads();
  const int my_chunk = tid & 7, my_row = tid >> 3;   // rows my_row and my_row + 32
  const int64_t pbeg = static_cast<int64_t>(blockIdx.z) * a.pix_per_slice;
  const int64_t pend = min(a.npix, pbeg + a.pix_per_slice);
  const int64_t pq = static_cast<int64_t>(a.P) * a.Q;
  const int dq = kChunk % a.Q, dp = (kChunk / a.Q) % a.P, dn = static_cast<int>(kChunk / pq);
  PixelRow rows[2];
  rows[0].init(pbeg + my_row, a.P, a.Q);
  rows[1].init(pbeg + my_row + 32, a.P, a.Q);

  // global loads of the next chunk into registers: 8 filters of dy and 8
  // im2col columns of x for its pixels my_row and my_row + 32
  auto load = [&](uint4 (&vd)[2], uint4 (&vx)[2]) {
#pragma unroll
    for (int h2 = 0; h2 < 2; ++h2) {
      const int64_t pix = rows[h2].pix;
      uint32_t d[4] = {0u, 0u, 0u, 0u}, xv[4] = {0u, 0u, 0u, 0u};
      if (pix < pend) {
        const int kb = k0 + 8 * my_chunk;
        const __nv_bfloat16* dyp = a.dy + pix * a.K + kb;
        if (a.dy_vec && kb + 8 <= a.K) {
          const uint4 v = __ldg(reinterpret_cast<const uint4*>(dyp));
          d[0] = v.x; d[1] = v.y; d[2] = v.z; d[3] = v.w;
        } else {
#pragma unroll
          for (int e = 0; e < 8; ++e)
            if (kb + e < a.K)
              d[e >> 1] |= static_cast<uint32_t>(__bfloat16_as_ushort(dyp[e])) << (16 * (e & 1));
        }
        const int n = rows[h2].n;
        const int h0 = rows[h2].p * a.sh - a.ph, w0 = rows[h2].q * a.sw - a.pw;
        const int jc = 8 * my_chunk;
        const int r = col_r[jc];
        if (a.x_vec && r >= 0 && jc + 7 < kTileN && col_r[jc + 7] == r && col_s[jc + 7] == col_s[jc]) {
          // eight consecutive channels of one tap
          const int hh = h0 + r, ww = w0 + col_s[jc];
          if (hh >= 0 && hh < a.H && ww >= 0 && ww < a.W) {
            const uint4 v = __ldg(reinterpret_cast<const uint4*>(
                a.x + ((static_cast<int64_t>(n) * a.H + hh) * a.W + ww) * a.C + col_c[jc]));
            xv[0] = v.x; xv[1] = v.y; xv[2] = v.z; xv[3] = v.w;
          }
        } else {
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const int re = col_r[jc + e];
            if (re < 0) continue;
            const int hh = h0 + re, ww = w0 + col_s[jc + e];
            if (hh >= 0 && hh < a.H && ww >= 0 && ww < a.W)
              xv[e >> 1] |= static_cast<uint32_t>(__bfloat16_as_ushort(
                                a.x[((static_cast<int64_t>(n) * a.H + hh) * a.W + ww) * a.C +
                                    col_c[jc + e]]))
                            << (16 * (e & 1));
          }
        }
      }
      vd[h2] = make_uint4(d[0], d[1], d[2], d[3]);
      vx[h2] = make_uint4(xv[0], xv[1], xv[2], xv[3]);
      rows[h2].advance(dn, dp, dq, a.P, a.Q);
    }
  };

  float acc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.0f;
  const uint32_t sdy_s = smem_addr(sdy), sx_s = smem_addr(sx);
  const int wf = 16 * (warp & 3), wj = 32 * (warp >> 2);
  const int mi = lane >> 3, lr = lane & 7;
  uint4 vd[2], vx[2];
  if (pbeg < pend) load(vd, vx);
  for (int64_t p0 = pbeg; p0 < pend; p0 += kChunk) {
    __syncthreads();   // the previous chunk's fragments have been read
#pragma unroll
    for (int h2 = 0; h2 < 2; ++h2) {
      *reinterpret_cast<uint4*>(sdy + tile_off(my_row + 32 * h2, my_chunk)) = vd[h2];
      *reinterpret_cast<uint4*>(sx + tile_off(my_row + 32 * h2, my_chunk)) = vx[h2];
    }
    __syncthreads();
    if (p0 + kChunk < pend) load(vd, vx);
#pragma unroll
    for (int ks = 0; ks < kChunk / 16; ++ks) {
      // A: filters wf .. wf+15 x pixels 16 ks ..; matrix mi = (pixel half
      // mi >> 1, filter half mi & 1)
      uint32_t af[4];
      ldsm_x4_trans(af, sdy_s + tile_off(16 * ks + 8 * (mi >> 1) + lr, (wf >> 3) + (mi & 1)));
#pragma unroll
      for (int nb = 0; nb < 2; ++nb) {
        // B: pixels 16 ks .. x columns wj + 16 nb ..; matrix mi = (pixel
        // half mi & 1, column half mi >> 1)
        uint32_t bf[4];
        ldsm_x4_trans(bf, sx_s + tile_off(16 * ks + 8 * (mi & 1) + lr,
                                          ((wj + 16 * nb) >> 3) + (mi >> 1)));
        mma_16816(acc[2 * nb], af, bf[0], bf[1]);
        mma_16816(acc[2 * nb + 1], af, bf[2], bf[3]);
      }
    }
  }
  // lane (g, t): filters wf + g (+8), columns wj + 8 nt + 2t (+1)
  float* part = a.part + static_cast<int64_t>(blockIdx.z) * a.K * a.rsc;
  const int g = lane >> 2, t = lane & 3;
#pragma unroll
  for (int nt = 0; nt < 4; ++nt) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int k = k0 + wf + g + 8 * (i >> 1);
      const int jj = j0 + wj + 8 * nt + 2 * t + (i & 1);
      if (k < a.K && jj < a.rsc) part[static_cast<int64_t>(k) * a.rsc + jj] = acc[nt][i];
    }
  }
}

// The same product for aligned operands (K % 8 == 0, C % 8 == 0, 16-byte
// aligned x and dy), on tiles of 128 filters x 128 columns: every 16-byte
// chunk is 8 filters of one pixel or 8 channels of one tap, copied by
// cp.async into a kStages-deep ring (out-of-image taps and pixels past the
// slice are zero-filled by a copy of source size 0), so several chunks'
// loads are in flight per CTA.
constexpr int kTileMA = 128;
constexpr int kTileNA = 128;
constexpr int kStages = 3;
constexpr int kHalfTile = kChunk * 128;           // 64 pixels x 64 bf16
constexpr int kStageBytes = 4 * kHalfTile;        // dy: 2 halves, x: 2 halves

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, bool valid) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src),
               "r"(valid ? 16 : 0)
               : "memory");
}

// The product runs on the 5th-generation tensor cores (tcgen05).  The
// pixel-major tiles are MN-major operands with the 128-byte swizzle: 64
// filters (or columns) of one pixel are a 128-byte row, 8 pixel rows an
// atom (SBO = 1 KB apart along the pixels), and the two 64-wide halves
// LBO = 8 KB apart.  One thread issues four
// M 128 x N 128 x K 16 MMAs per 64-pixel chunk into a 128-column fp32
// accumulator in tensor memory and commits them to the stage's mbarrier;
// a stage is refilled only after the MMAs reading it have completed.
constexpr uint64_t kBwdWaitLimitNs = 1000000000ull;

__device__ __forceinline__ uint64_t smem_desc_sw128_mn(uint32_t saddr) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
  d |= static_cast<uint64_t>(8192u >> 4) << 16;   // LBO: next 64-wide MN half
  d |= static_cast<uint64_t>(1024u >> 4) << 32;   // SBO: next 8 pixel rows
  d |= static_cast<uint64_t>(1u) << 46;
  d |= static_cast<uint64_t>(2u) << 61;          // 128-byte swizzle
  return d;
}

__global__ void __launch_bounds__(kBwdThreads, 2) bwd_filter_tc_kernel(const BwdFilterArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* ring = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  __shared__ int col_r[kTileNA], col_s[kTileNA], col_c[kTileNA];
  __shared__ uint64_t bar[kStages];
  __shared__ uint32_t tmem_slot;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int k0 = blockIdx.x * kTileMA, j0 = blockIdx.y * kTileNA;
  if (tid < kTileNA) {
    const int j = j0 + tid;
    const int c = j % a.C, rs = j / a.C;
    col_c[tid] = c;
    col_s[tid] = rs % a.S;
    col_r[tid] = j < a.rsc ? rs / a.S : -1;
  }
  if (warp == 0) {
    tmem_alloc(&tmem_slot, 128);
    tmem_relinquish();
  }
  if (tid == 0) {
    for (int i = 0; i < kStages; ++i) mbar_init(&bar[i], 1);
    fence_mbar_init();
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t acc = tmem_slot;
  const int my_chunk = tid & 7, my_row = tid >> 3;
  const int64_t pbeg = static_cast<int64_t>(blockIdx.z) * a.pix_per_slice;
  const int64_t pend = min(a.npix, pbeg + a.pix_per_slice);
  const int64_t pq = static_cast<int64_t>(a.P) * a.Q;
  const int nchunks = pend > pbeg ? static_cast<int>((pend - pbeg + kChunk - 1) / kChunk) : 0;
  const uint32_t ring_s = smem_addr(ring);
  // this thread's two im2col columns: tap (r, s) and channel, and their
  // offset from the tap-(0, 0) element in x
  int tap_r[2], tap_s[2];
  int64_t tap_off[2];
#pragma unroll
  for (int hx = 0; hx < 2; ++hx) {
    const int jc = 64 * hx + 8 * my_chunk;
    tap_r[hx] = col_r[jc];
    tap_s[hx] = col_s[jc];
    tap_off[hx] = (static_cast<int64_t>(tap_r[hx]) * a.W + tap_s[hx]) * a.C + col_c[jc];
  }
  const int dq = kChunk % a.Q, dp = (kChunk / a.Q) % a.P, dn = static_cast<int>(kChunk / pq);
  PixelRow rows[2];
  rows[0].init(pbeg + my_row, a.P, a.Q);
  rows[1].init(pbeg + my_row + 32, a.P, a.Q);
  // chunks are issued once each, in order, so the rows advance by kChunk
  auto issue = [&](int ci) {
    const uint32_t st = ring_s + static_cast<uint32_t>((ci % kStages) * kStageBytes);
#pragma unroll
    for (int h2 = 0; h2 < 2; ++h2) {
      const int row = my_row + 32 * h2;
      const bool pv = rows[h2].pix < pend;
      const int64_t dy_row = pv ? rows[h2].pix * a.K : 0;
#pragma unroll
      for (int hf = 0; hf < 2; ++hf) {
        const int kb = k0 + 64 * hf + 8 * my_chunk;
        cp_async16(st + hf * kHalfTile + tile_off(row, my_chunk),
                   a.dy + dy_row + (kb < a.K ? kb : 0), pv && kb < a.K);
      }
      const int h0 = rows[h2].p * a.sh - a.ph, w0 = rows[h2].q * a.sw - a.pw;
      const int64_t x_row = ((static_cast<int64_t>(rows[h2].n) * a.H + h0) * a.W + w0) * a.C;
#pragma unroll
      for (int hx = 0; hx < 2; ++hx) {
        const int hh = h0 + tap_r[hx], ww = w0 + tap_s[hx];
        const bool xv = pv && tap_r[hx] >= 0 && hh >= 0 && hh < a.H && ww >= 0 && ww < a.W;
        cp_async16(st + (2 + hx) * kHalfTile + tile_off(row, my_chunk),
                   a.x + (xv ? x_row + tap_off[hx] : 0), xv);
      }
      rows[h2].advance(dn, dp, dq, a.P, a.Q);
    }
  };
  constexpr uint32_t idesc = idesc_bf16_f32(128, 128) | (1u << 15) | (1u << 16);   // MN-major
#pragma unroll
  for (int ci = 0; ci < kStages - 1; ++ci) {
    if (ci < nchunks) issue(ci);
    asm volatile("cp.async.commit_group;" ::: "memory");
  }
  bool ok = true;
  for (int ci = 0; ci < nchunks; ++ci) {
    asm volatile("cp.async.wait_group %0;" ::"n"(kStages - 2) : "memory");
    fence_proxy_async_smem();   // this thread's copies -> visible to the tensor core
    __syncthreads();
    if (tid == 0) {
      tc_fence_after_sync();
      const uint32_t st = ring_s + static_cast<uint32_t>((ci % kStages) * kStageBytes);
#pragma unroll
      for (int ks = 0; ks < kChunk / 16; ++ks)
        tc_mma_ss(acc, smem_desc_sw128_mn(st + ks * 2048), smem_desc_sw128_mn(st + 2 * kHalfTile + ks * 2048),
                  idesc, (ci | ks) != 0 ? 1u : 0u);
      tc_commit(&bar[ci % kStages]);
    }
    if (ci + kStages - 1 < nchunks) {
      // the refilled stage held chunk ci - 1: its MMAs must have finished
      if (ci >= 1 && tid == 0)
        ok = mbar_wait(&bar[(ci - 1) % kStages], static_cast<uint32_t>((ci - 1) / kStages) & 1u,
                       nullptr, a.err, kBwdWaitLimitNs);
      if (!__syncthreads_and(ok)) break;
      issue(ci + kStages - 1);
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  }
  asm volatile("cp.async.wait_group 0;" ::: "memory");
  if (nchunks > 0 && tid == 0)
    ok = mbar_wait(&bar[(nchunks - 1) % kStages],
                   static_cast<uint32_t>((nchunks - 1) / kStages) & 1u, nullptr, a.err,
                   kBwdWaitLimitNs) && ok;
  ok = __syncthreads_and(ok);
  tc_fence_after_sync();
  // epilogue: warp w reads lanes 32 (w % 4) .. (filters) and columns 64 (w / 4) ..
  float* part = a.part + static_cast<int64_t>(blockIdx.z) * a.K * a.rsc;
  const int k = k0 + 32 * (warp & 3) + lane;
#pragma unroll
  for (int q = 0; q < 2; ++q) {
    const int jb = 64 * (warp >> 2) + 32 * q;
    uint32_t v[32];
    tmem_ld_32x32b_x32(acc + (static_cast<uint32_t>(32 * (warp & 3)) << 16) +
                           static_cast<uint32_t>(jb),
                       v);
    tmem_wait_ld();
    if (nchunks == 0) {
#pragma unroll
      for (int i = 0; i < 32; ++i) v[i] = 0u;
    }
    if (ok && k < a.K) {
      float* row = part + static_cast<int64_t>(k) * a.rsc + j0 + jb;
      if (a.part_vec && j0 + jb + 32 <= a.rsc) {
#pragma unroll
        for (int i = 0; i < 32; i += 4)
          *reinterpret_cast<uint4*>(row + i) = make_uint4(v[i], v[i + 1], v[i + 2], v[i + 3]);
      } else {
#pragma unroll
        for (int i = 0; i < 32; ++i)
          if (j0 + jb + i < a.rsc) row[i] = __uint_as_float(v[i]);
      }
    }
  }
  tc_fence_before_sync();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after_sync();
    tmem_dealloc(acc, 128);
  }
}

// dw[e] = sum of the slices' partial values in a fixed order.  The block's
// threads form `groups` (1, 2, 4 or 8, a function of the slice count) groups
// of 256 / groups; group g sums slices g, g + groups, ... in order for one
// element per thread, and group 0 adds the group sums in group order.
__global__ void __launch_bounds__(kBwdThreads) bwd_filter_reduce_kernel(
    const float* __restrict__ part, int slices, int groups, int64_t count,
    float* __restrict__ dw) {
  __shared__ float sums[kBwdThreads];
  const int per = kBwdThreads / groups;
  const int li = threadIdx.x % per, g = threadIdx.x / per;
  const int64_t e = static_cast<int64_t>(blockIdx.x) * per + li;
  float s = 0.0f;
  if (e < count) {
#pragma unroll 4
    for (int z = g; z < slices; z += groups) s += part[static_cast<int64_t>(z) * count + e];
  }
  sums[threadIdx.x] = s;
  __syncthreads();
  if (g == 0 && e < count) {
    float t = sums[li];
    for (int h = 1; h < groups; ++h) t += sums[h * per + li];
    dw[e] = t;
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

// Pixel slices of the filter gradient: one wave of CTAs over the tiles of
// the kernel the shape selects (2 resident per SM for the 96 KB ring, 4 for
// the register path), each slice's partial tile costing a write and a read
// in the reduction.  A function of the shape only, so the workspace query
// agrees with the launch.
int bwd_filter_slices(const BwdConvShape& p) {
  const bool big = p.K % 8 == 0 && p.C % 8 == 0;
  const int tm = big ? kTileMA : kTileM, tn = big ? kTileNA : kTileN;
  const int64_t tiles = ((p.K + tm - 1) / tm) * ((p.R * p.S * p.C + tn - 1) / tn);
  const int64_t want = (big ? 2 : 4) * static_cast<int64_t>(device_sm_count());
  const int64_t npix = p.N * p.P * p.Q;
  int64_t s = std::max<int64_t>(1, want / std::max<int64_t>(tiles, 1));
  s = std::min<int64_t>(s, std::max<int64_t>(1, npix / (4 * kChunk)));
  // at most 64 MB of partial tiles
  const int64_t per_slice = std::max<int64_t>(1, p.K * p.R * p.S * p.C);
  s = std::min<int64_t>(s, std::max<int64_t>(1, (int64_t{16} << 20) / per_slice));
  return static_cast<int>(std::min<int64_t>(s, 1024));
}

}  // namespace

const char* bwd_shape_reason(const BwdConvShape& p) {
  if (p.ph > p.R - 1 || p.pw > p.S - 1) return "backward needs pad <= kernel size - 1";
  // the sizes are below 2^31 here, so each pairwise product fits in int64
  const int64_t lim = int64_t(1) << 40;
  const auto prod_below = [lim](int64_t a, int64_t b, int64_t c, int64_t d) {
    const int64_t ab = a * b, cd = c * d;
    return ab < lim && cd < lim && (ab == 0 || cd < lim / ab);
  };
  if (!prod_below(p.N, p.H, p.W, p.C) || !prod_below(p.N, p.P, p.Q, p.K))
    return "backward: tensor too large";
  if (p.C >= (1 << 30) || p.K >= (1 << 30) || !prod_below(p.R, p.S, p.C, 1024) ||
      !prod_below(p.R, p.S, p.K, 1024))
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
    const int64_t total = p.N * b.Hd * b.Wd * (p.K % 8 == 0 ? p.K / 8 : 1);
    const int64_t blocks =
        std::max<int64_t>(1, std::min<int64_t>((std::max<int64_t>(total, p.C) + 255) / 256,
                                               static_cast<int64_t>(device_sm_count()) * 16));
    // dyd is 256-aligned; alpha is read as float4 pairs
    const int vec = (p.K % 8 == 0 && is_aligned(dy, 16) && is_aligned(alpha, 16)) ? 1 : 0;
    dilate_scale_kernel<<<static_cast<unsigned>(blocks), 256, 0, s>>>(
        static_cast<const __nv_bfloat16*>(dy), alpha, static_cast<int>(p.N),
        static_cast<int>(p.P), static_cast<int>(p.Q), static_cast<int>(p.K),
        static_cast<int>(b.Hd), static_cast<int>(b.Wd), static_cast<int>(p.sh),
        static_cast<int>(p.sw), dyd, ones, static_cast<int>(p.C), vec);
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
  a.part_vec = (p.R * p.S * p.C) % 4 == 0 && (reinterpret_cast<uintptr_t>(workspace) & 15) == 0;
  a.N = static_cast<int>(p.N); a.C = static_cast<int>(p.C); a.H = static_cast<int>(p.H);
  a.W = static_cast<int>(p.W); a.K = static_cast<int>(p.K); a.R = static_cast<int>(p.R);
  a.S = static_cast<int>(p.S); a.sh = static_cast<int>(p.sh); a.sw = static_cast<int>(p.sw);
  a.ph = static_cast<int>(p.ph); a.pw = static_cast<int>(p.pw); a.P = static_cast<int>(p.P);
  a.Q = static_cast<int>(p.Q);
  a.npix = p.N * p.P * p.Q;
  a.rsc = static_cast<int>(p.R * p.S * p.C);
  a.slices = bwd_filter_slices(p);
  a.dy_vec = (p.K % 8 == 0 && is_aligned(dy, 16)) ? 1 : 0;
  a.x_vec = (p.C % 8 == 0 && is_aligned(x, 16)) ? 1 : 0;
  a.pix_per_slice = (a.npix + a.slices - 1) / a.slices;
  const bool async_path = a.dy_vec && a.x_vec;
  const int tile_m = async_path ? kTileMA : kTileM;
  const int tile_n = async_path ? kTileNA : kTileN;
  const dim3 grid(static_cast<unsigned>((p.K + tile_m - 1) / tile_m),
                  static_cast<unsigned>((a.rsc + tile_n - 1) / tile_n),
                  static_cast<unsigned>(a.slices));
  if (grid.y > 65535) return fail(TBN_ERR_UNSUPPORTED, "backward filter: R S C too large");
  tbn_status st;
  if (async_path) {
    static std::once_flag attr_once;
    static cudaError_t attr_err = cudaSuccess;
    std::call_once(attr_once, [] {
      attr_err = cudaFuncSetAttribute(bwd_filter_tc_kernel,
                                      cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      kStages * kStageBytes + 1024);
    });
    if (attr_err != cudaSuccess)
      return cuda_fail(attr_err, "cudaFuncSetAttribute(bwd_filter_tc_kernel)");
    a.err = device_error_word();
    bwd_filter_tc_kernel<<<grid, kBwdThreads, kStages * kStageBytes + 1024, s>>>(a);
    st = check_launch("bwd_filter_tc_kernel");
  } else {
    bwd_filter_kernel<<<grid, kBwdThreads, 0, s>>>(a);
    st = check_launch("bwd_filter_kernel");
  }
  if (st != TBN_OK) return st;
  const int64_t count = p.K * a.rsc;
  const int groups = a.slices >= 8 ? 8 : a.slices >= 4 ? 4 : a.slices >= 2 ? 2 : 1;
  const int64_t per = kBwdThreads / groups;
  const int64_t blocks = (count + per - 1) / per;
  if (blocks > 0x7fffffff) return fail(TBN_ERR_UNSUPPORTED, "backward filter: too many weights");
  bwd_filter_reduce_kernel<<<static_cast<unsigned>(blocks), kBwdThreads, 0, s>>>(
      a.part, a.slices, groups, count, dw);
  return check_launch("bwd_filter_reduce_kernel");
}

}  // namespace tbn
