// tbn_quant_core.cuh -- the per-word arithmetic of the quantizer (Eq. 3
// fields, Eq. 5 sums with exact two-float accumulation, alpha), shared by
// the quantize kernel and the fused quantize-and-convolve prologue of the
// implicit GEMM, so that both produce bitwise the same codes and alpha.
#pragma once

#include <cstdint>

#include "tbn_device.cuh"

namespace tbn {
namespace {

// ---- exact two-float accumulation (fp32 adds only) -----------------------
struct Sum2 {
  float hi, lo;
};

__device__ __forceinline__ void add2(Sum2& s, float x) {
  // TwoSum: hi + lo gains x with the rounding error of the add kept in lo
  const float t = __fadd_rn(s.hi, x);
  const float bp = __fsub_rn(t, s.hi);
  const float e = __fadd_rn(__fsub_rn(s.hi, __fsub_rn(t, bp)), __fsub_rn(x, bp));
  s.hi = t;
  s.lo = __fadd_rn(s.lo, e);
}

__device__ __forceinline__ void merge2(Sum2& s, const Sum2& o) {
  add2(s, o.hi);
  s.lo = __fadd_rn(s.lo, o.lo);
}

__device__ __forceinline__ Sum2 warp_sum2(Sum2 s) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    Sum2 t;
    t.hi = __shfl_xor_sync(0xffffffffu, s.hi, o);
    t.lo = __shfl_xor_sync(0xffffffffu, s.lo, o);
    merge2(s, t);
  }
  return s;
}

__device__ __forceinline__ int warp_sum(int v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Eq. 5 with |B1| + 4|B2| = n + 3|B2|: (hi + lo) / den with one final
// rounding, from an fp32 quotient and its exact remainder (den < 2^24 is
// exact in fp32; longer filters take the fp64 division).
__device__ __forceinline__ float alpha_of(const Sum2& s, int cnt2, int n) {
  const int64_t den_i = static_cast<int64_t>(n) + 3 * static_cast<int64_t>(cnt2);
  if (den_i >= (int64_t(1) << 24))
    return static_cast<float>((static_cast<double>(s.hi) + static_cast<double>(s.lo)) /
                              static_cast<double>(den_i));
  const float den = static_cast<float>(den_i);
  const float q = __fdiv_rn(s.hi, den);
  const float r = __fadd_rn(__fmaf_rn(-q, den, s.hi), s.lo);   // exact remainder + lo
  return __fadd_rn(q, __fdiv_rn(r, den));
}

// fp64 alpha of one filter, used only when a word sum overflowed fp32.
__device__ __noinline__ float alpha_fp64_row(const float* __restrict__ row, int n) {
  double num = 0.0;
  int64_t cnt2 = 0;
  for (int i = 0; i < n; ++i) {
    const double a = fabs(static_cast<double>(row[i]));
    if (a > 1.0) {
      num += 2.0 * a;
      ++cnt2;
    } else {
      num += a;
    }
  }
  return static_cast<float>(num / (static_cast<double>(n) + 3.0 * static_cast<double>(cnt2)));
}

// Sixteen weights -> one packed word, the fp32 pairwise sum of |W~|*|W| over
// them and the number of magnitude-two codes.  Eq. 3: s = [W <= 0] (so
// -1 <= W <= 0 and W < -1 are negative, -0.0 included), m = [|W| > 1].
__device__ __forceinline__ void encode16(const float (&v)[16], int nvalid, uint32_t& word,
                                         float& sum, int& cnt2) {
  float c[16];
  uint32_t w = 0;
  int n2 = 0;
#pragma unroll
  for (int e = 0; e < 16; ++e) {
    const float a = fabsf(v[e]);
    const uint32_t m = a > 1.0f ? 1u : 0u;
    const uint32_t s = v[e] <= 0.0f ? 1u : 0u;
    const bool valid = e < nvalid;
    w |= valid ? ((m << code_mag_bit(e)) | (s << (code_mag_bit(e) + 8))) : 0u;
    n2 += (valid && m) ? 1 : 0;
    c[e] = valid ? (m ? 2.0f * a : a) : 0.0f;
  }
#pragma unroll
  for (int e = 0; e < 8; ++e) c[e] += c[e + 8];
#pragma unroll
  for (int e = 0; e < 4; ++e) c[e] += c[e + 4];
  c[0] += c[2];
  c[1] += c[3];
  sum = c[0] + c[1];
  word = w;
  cnt2 = n2;
}

__device__ __forceinline__ bool finite_sum(float s) { return s <= 3.4028234663852886e38f; }

__device__ __forceinline__ void load16(const float* __restrict__ row, int n, int j, bool vec,
                                       float (&v)[16], int& nvalid) {
  const int base = 16 * j;
  nvalid = min(16, n - base);
  if (vec && nvalid == 16) {
    const float4* p = reinterpret_cast<const float4*>(row + base);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float4 t = __ldcs(p + q);
      v[4 * q + 0] = t.x;
      v[4 * q + 1] = t.y;
      v[4 * q + 2] = t.z;
      v[4 * q + 3] = t.w;
    }
  } else {
#pragma unroll
    for (int e = 0; e < 16; ++e) v[e] = (e < nvalid) ? __ldcs(row + base + e) : 0.0f;
  }
}

}  // namespace
}  // namespace tbn
