// tbn_gemv.cu -- small-batch two-bit fully-connected layer (Section 3:
// fully-connected layers treated as convolutions), y[b,k] = alpha_k *
// sum_j x[b,j] W~[k,j] for B <= 8, bandwidth-bound on the 2-bit weight stream.
//
// Tensor-core formulation per warp: mma.m16n8k16 with A = 16 weight rows x 16
// codes decoded in registers to bf16 W~/2 (exact), B = 16 inputs x 8 batch
// columns (batch padded with zeros), fp32 accumulation; 2 * alpha in the
// epilogue.  The A fragment of lane (g = lane/4, t = lane%4) needs codes
// 2t, 2t+1 and 2t+8, 2t+9 of rows g and g+8 -- nibbles t and t+4 of each
// row's word for the K step -- so every lane of a quad reads the same
// 16-byte group of four words (one transaction, broadcast) and decodes its
// own nibbles.  A CTA is 8 warps: 2 row tiles x 4 K quarters (interleaved
// 64-code chunks), reduced through shared memory.
#include <cuda_bf16.h>

#include <cstdint>

#include "tbn_device.cuh"
#include "tbn_internal.h"

namespace tbn {
namespace {

constexpr int kRowTiles = 2;   // 16-row tiles per CTA
constexpr int kKSplit = 4;     // warps along K per row tile
constexpr int kThreads = 32 * kRowTiles * kKSplit;

__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint32_t (&a)[4],
                                               uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
      "{%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

template <int kB>
__global__ void __launch_bounds__(kThreads) gemv_kernel(const __nv_bfloat16* __restrict__ x,
                                                        int K_in, const uint32_t* __restrict__ codes,
                                                        const float* __restrict__ alpha, int K_out,
                                                        void* __restrict__ y, int y_bf16, int relu,
                                                        const void* __restrict__ residual) {
  __shared__ float s_part[kRowTiles][kKSplit][32][4];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int rt = warp / kKSplit, ks = warp % kKSplit;
  const int g = lane >> 2, t = lane & 3;
  const int row0 = (blockIdx.x * kRowTiles + rt) * 16;
  const int wpf = K_in / 16;
  const int rA = row0 + g, rB = row0 + g + 8;
  const uint4* wa = reinterpret_cast<const uint4*>(codes + static_cast<size_t>(rA < K_out ? rA : 0) * wpf);
  const uint4* wb = reinterpret_cast<const uint4*>(codes + static_cast<size_t>(rB < K_out ? rB : 0) * wpf);
  const bool va = rA < K_out, vb = rB < K_out;
  // batch column n = g of the B fragment
  const bool xb = g < kB;
  const uint32_t* xrow = reinterpret_cast<const uint32_t*>(x + static_cast<size_t>(xb ? g : 0) * K_in);

  float d[4] = {0.f, 0.f, 0.f, 0.f};
  const int nchunks = K_in / 64;  // 64 codes = 4 words = one uint4 per row
  for (int c = ks; c < nchunks; c += kKSplit) {
    const uint4 A4 = va ? __ldg(wa + c) : make_uint4(0u, 0u, 0u, 0u);
    const uint4 B4 = vb ? __ldg(wb + c) : make_uint4(0u, 0u, 0u, 0u);
    const uint32_t wA[4] = {A4.x, A4.y, A4.z, A4.w};
    const uint32_t wB[4] = {B4.x, B4.y, B4.z, B4.w};
#pragma unroll
    for (int s = 0; s < 4; ++s) {
      const int k0 = c * 64 + s * 16;
      uint32_t a[4];
      a[0] = nibble_to_bf16x2((wA[s] >> (4 * t)) & 0xFu);        // row g,   k 2t..2t+1
      a[1] = nibble_to_bf16x2((wB[s] >> (4 * t)) & 0xFu);        // row g+8, k 2t..2t+1
      a[2] = nibble_to_bf16x2((wA[s] >> (4 * t + 16)) & 0xFu);   // row g,   k 2t+8..
      a[3] = nibble_to_bf16x2((wB[s] >> (4 * t + 16)) & 0xFu);   // row g+8, k 2t+8..
      const uint32_t b0 = xb ? __ldg(xrow + (k0 >> 1) + t) : 0u;
      const uint32_t b1 = xb ? __ldg(xrow + (k0 >> 1) + t + 4) : 0u;
      mma_bf16_16816(d, a, b0, b1);
    }
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) s_part[rt][ks][lane][i] = d[i];
  __syncthreads();
  if (ks != 0) return;
  float sum[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    sum[i] = s_part[rt][0][lane][i];
#pragma unroll
    for (int w = 1; w < kKSplit; ++w) sum[i] += s_part[rt][w][lane][i];
  }
  // d[0]: (row g, batch 2t)  d[1]: (row g, batch 2t+1)  d[2], d[3]: row g+8
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int row = (i < 2) ? rA : rB;
    const int b = 2 * t + (i & 1);
    if (row >= K_out || b >= kB) continue;
    float v = 2.0f * alpha[row] * sum[i];
    const size_t o = static_cast<size_t>(b) * K_out + row;
    if (y_bf16) {
      if (residual) v += __bfloat162float(static_cast<const __nv_bfloat16*>(residual)[o]);
      if (relu) v = fmaxf(v, 0.0f);
      static_cast<__nv_bfloat16*>(y)[o] = __float2bfloat16_rn(v);
    } else {
      if (residual) v += static_cast<const float*>(residual)[o];
      if (relu) v = fmaxf(v, 0.0f);
      static_cast<float*>(y)[o] = v;
    }
  }
}

template <int kB>
tbn_status launch_b(const void* x, int64_t K_in, const uint32_t* codes, const float* alpha,
                    int64_t K_out, void* y, tbn_dtype ydt, int relu, const void* residual,
                    cudaStream_t s) {
  const int64_t blocks = (K_out + 16 * kRowTiles - 1) / (16 * kRowTiles);
  gemv_kernel<kB><<<(unsigned)blocks, kThreads, 0, s>>>(
      static_cast<const __nv_bfloat16*>(x), (int)K_in, codes, alpha, (int)K_out, y,
      ydt == TBN_BF16 ? 1 : 0, relu, residual);
  return check_launch("gemv_kernel");
}

}  // namespace

const char* gemv_unsupported_reason(const void* x, tbn_dtype xdt, int64_t B, int64_t K_in,
                                    const uint32_t* codes) {
  if (xdt != TBN_BF16) return "GEMV needs bf16 activations";
  if (B < 1 || B > 8) return "GEMV needs 1 <= B <= 8";
  if (K_in % 64 != 0) return "GEMV needs K_in % 64 == 0";
  if (K_in >= (1ll << 30)) return "GEMV: K_in too large";
  if (!is_aligned(x, 16) || !is_aligned(codes, 16)) return "GEMV needs 16-byte aligned x and codes";
  return "";
}

tbn_status launch_gemv(const void* x, int64_t B, int64_t K_in, const uint32_t* codes,
                       const float* alpha, int64_t K_out, void* y, tbn_dtype ydt, int relu,
                       const void* residual, cudaStream_t s) {
  switch (B) {
    case 1: return launch_b<1>(x, K_in, codes, alpha, K_out, y, ydt, relu, residual, s);
    case 2: return launch_b<2>(x, K_in, codes, alpha, K_out, y, ydt, relu, residual, s);
    case 3: return launch_b<3>(x, K_in, codes, alpha, K_out, y, ydt, relu, residual, s);
    case 4: return launch_b<4>(x, K_in, codes, alpha, K_out, y, ydt, relu, residual, s);
    case 5: return launch_b<5>(x, K_in, codes, alpha, K_out, y, ydt, relu, residual, s);
    case 6: return launch_b<6>(x, K_in, codes, alpha, K_out, y, ydt, relu, residual, s);
    case 7: return launch_b<7>(x, K_in, codes, alpha, K_out, y, ydt, relu, residual, s);
    default: return launch_b<8>(x, K_in, codes, alpha, K_out, y, ydt, relu, residual, s);
  }
}

}  // namespace tbn
