// tbn_gemv_f8.cu -- batch-1 two-bit fully-connected layer on the tcgen05
// tensor cores in fp8 (Section 3: a fully-connected layer is a convolution
// whose filters span the whole input): y[k] = alpha_k sum_j x[j] W~[k, j].
//
// W~/2 in {+-0.5, +-1} is exact in e4m3, and so is x after an exact split:
// with one power-of-two scale 2^E for the whole vector (max |x| 2^E in
// [128, 256)), x 2^E = t1 + t2 / 16 + t3 / 256 + r with t1, t2, t3 e4m3
// (round to nearest, subnormals kept) and |r| <= 2^-18 in scaled units, i.e.
// 2^-25 max |x| per element: over K_in <= 16384 inputs that is at most
// 2^-11 max|x| <= 2^-11 sum|x|, inside the 2e-3 alpha sum|x| bound.  The
// three terms are the first three columns of the MMA's B operand (N = 16,
// the other columns zero), so one fp32 accumulator column per term; the
// epilogue forms (d0 + d1 / 16 + d2 / 256) 2^-E.  The tensor core's fp8
// accumulation was checked exact on sums spanning 17 binades.
//
// Why fp8: the two-bit stream needs about 89 weights per clock per SM at the
// copy peak.  Decoding to bf16 costs one instruction per weight (a mask and
// a multiply-add per pair); decoding to e4m3 costs half that (a mask and a
// multiply-add per four weights), from the "e4m3-planar" words that
// tbn_linear_prepare_f8 writes once per weight matrix: code 4j + b of a
// word keeps its magnitude bit at bit 8b + j and its sign bit at 8b + 4 + j,
// so (w & (0x11111111 << j)) * 2^(3-j) + 0x30303030 is the four e4m3 bytes
// of codes 4j .. 4j + 3 (0x30 = 0.5, m -> 0x38 = 1.0, s -> sign).  The
// prepared words are also blocked: the 128 rows x 32 words of one (tile,
// stage) unit are 16 contiguous KiB, row r's 16-byte chunk c at chunk
// position c ^ (r % 8) (the 128-byte swizzle, so the decoders' row reads hit
// distinct banks); one 1-D bulk copy fetches a unit.  The
// tensor core is far from the limit: a kind::f8f6f4 MMA with M = 128,
// N = 16, K = 32 issues every 9 cycles (450 weights per clock).
//
// Work split: the (128-row tile, 512-code stage) units of the layer,
// tile-major, are cut into one contiguous range per CTA.  When the tiles
// fill at least 4/5 of the SMs each CTA takes whole tiles and its epilogue
// writes y.  Otherwise (stream-K) a CTA's range covers parts of one or more
// tiles ("segments"); each segment's fp32 partial sums go to a workspace
// slot, and gemv_f8_reduce_kernel adds a tile's slots in CTA order
// (bitwise reproducible) and applies 2 alpha, the residual and ReLU.
// Every CTA splits x itself (all of it; x is L2-resident after the first
// reads) while its first code stages are in flight.
//
// Per CTA: a producer warp streams the code blocks through a shared-memory
// ring with 1-D bulk copies; sixteen decoder warps (thread = tensor-memory
// lane = weight row, four warps per lane quarter, each a quarter of a
// stage's 32 words) turn them into e4m3 W~/2 in a
// 3-stage tensor-memory ring (128 columns per stage); one MMA warp issues
// the stage's 16 MMAs (A from tensor memory, B = the x terms, resident in
// shared memory for the whole K range); four epilogue warps read a
// segment's accumulator (double-buffered) and write its partial sums.
// Every wait is bounded; on expiry the kernel records a timeout in the
// device error word, stops, drains what it started and returns.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_fp8.h>

#include <algorithm>
#include <cstdint>
#include <cstring>
#include <mutex>

#include "tbn_device.cuh"
#include "tbn_internal.h"

namespace tbn {
namespace {

constexpr int kRows = 128;                 // MMA M: weight rows per tile
constexpr int kStageCodes = 512;           // codes per stage (32 words per row)
constexpr int kStageWords = kStageCodes / 16;
constexpr int kCodeStageBytes = kRows * kStageWords * 4;   // 16 KiB
constexpr int kMaxCodeStages = 12;        // shared-memory code ring (as deep as fits)
constexpr int kAStages = 3;                // tensor-memory operand ring
constexpr int kACols = kStageCodes / 4;    // 128 columns of 4 e4m3 per stage
constexpr int kDCols = 16;                 // MMA N
constexpr int kTmemCols = 512;             // D: 2 x 16 at 0, A ring at 128
constexpr int kAColBase = 128;
constexpr int kBStageBytes = 4 * 1024;     // x terms of one stage: 4 atoms of 8 rows x 128 B
constexpr int kMaxStagesK = 32;            // K_in <= 16384 (x terms resident)
constexpr int kDecWarps = 16;           // four per tensor-memory lane quarter
constexpr int kEpiWarps = 4;
constexpr int kFirstDecWarp = 2;
constexpr int kFirstEpiWarp = kFirstDecWarp + kDecWarps;
constexpr int kThreads = 32 * (kFirstEpiWarp + kEpiWarps);   // 704
constexpr uint64_t kWaitLimitNs = 1000000000ull;
constexpr int kSmemLimit = 232448;

static_assert(2 * kDCols <= kAColBase && kAColBase + kAStages * kACols <= kTmemCols, "TMEM");
// the x split's per-thread load batches cover K_in = 512 kMaxStagesK
static_assert(kMaxStagesK * kStageCodes / 8 <= 5 * (kThreads - 32) &&
              kMaxStagesK * kStageCodes / 4 <= 10 * (kThreads - 32), "x split batches");

struct F8Args {
  const __nv_bfloat16* x;   // [K_in]
  float* partial;           // [tiles][maxc][128] (split tiles)
  uint32_t* err;
  int K_out, K_in;
  int tiles, nks;           // 128-row tiles, 512-code stages per tile
  int units_per_cta;        // L: CTA b takes units [b L, (b + 1) L)
  int total_units;          // tiles * nks
  int maxc;                 // partial slots per tile
  int cstages;              // code ring depth
  const uint32_t* prepared; // blocked e4m3-planar codes [tiles][nks][128][32]
  int direct;               // every tile in one CTA: the epilogue writes y
  const float* alpha;
  void* y;
  const void* residual;
  int relu, y_bf16;
};

struct F8Smem {
  uint64_t full_c[kMaxCodeStages], empty_c[kMaxCodeStages];
  uint64_t full_a[kAStages], empty_a[kAStages];
  uint64_t acc_full[2], acc_empty[2];
  uint64_t drain;
  uint32_t tmem_base;
  int abort;
  uint32_t red[32];         // x split: per-warp maxima
  int E;                    // the x terms are x 2^E
};

// Shared-memory descriptor, K-major, 128-byte swizzle, with an explicit
// stride byte offset (distance to the next 8-row group).
__device__ __forceinline__ uint64_t desc_sw128(uint32_t saddr, uint32_t sbo) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
  d |= static_cast<uint64_t>(1u) << 16;
  d |= static_cast<uint64_t>((sbo >> 4) & 0x3FFFu) << 32;
  d |= static_cast<uint64_t>(1u) << 46;
  d |= static_cast<uint64_t>(2u) << 61;
  return d;
}

// Instruction descriptor, kind::f8f6f4: A and B E4M3 (format 0), D fp32,
// both K-major, N >> 3 at [17, 23), M >> 4 at [24, 29).
__host__ __device__ constexpr uint32_t idesc_e4m3_f32(uint32_t M, uint32_t N) {
  return (1u << 4) | ((N >> 3) << 17) | ((M >> 4) << 24);
}

__device__ __forceinline__ void mma_f8_ts(uint32_t d, uint32_t a, uint64_t bdesc, uint32_t idesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d),
      "r"(a), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// ---------------------------------------------------------------- prepare
// Byte-planar codes [K_out][K_in / 16] -> blocked e4m3-planar words
// [tiles][nks][128 rows][32 words]: byte-planar code l = 2p + h (m at bit
// 16h + p, s at 16h + 8 + p) becomes code l = 4j + b (m at bit 8b + j, s at
// 8b + 4 + j); word w of row r of a unit sits at chunk ((w / 4) ^ (r % 8)),
// position w % 4.  Rows past K_out are zero.
__global__ void __launch_bounds__(256) prepare_f8_kernel(const uint32_t* __restrict__ in,
                                                         int64_t K_out, int wpf, int64_t total,
                                                         uint32_t* __restrict__ out) {
  const int nks = wpf / kStageWords;
  for (int64_t o = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; o < total;
       o += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int wp = static_cast<int>(o % kStageWords);
    const int rr = static_cast<int>((o / kStageWords) % kRows);
    const int64_t unit = o / (kStageWords * kRows);
    const int ks = static_cast<int>(unit % nks);
    const int64_t t = unit / nks;
    const int w = (((wp >> 2) ^ (rr & 7)) << 2) | (wp & 3);   // logical word of the stage
    const int64_t row = t * kRows + rr;
    uint32_t res = 0;
    if (row < K_out) {
      const uint32_t v = in[row * wpf + ks * kStageWords + w];
#pragma unroll
      for (int l = 0; l < 16; ++l) {
        const int src = code_mag_bit(l);
        const int dst = 8 * (l & 3) + (l >> 2);
        res |= ((v >> src) & 1u) << dst;
        res |= ((v >> (src + 8)) & 1u) << (dst + 4);
      }
    }
    out[o] = res;
  }
}

// ---------------------------------------------------------------- x split
// Two values rounded to e4m3 (nearest, subnormals kept): the two bytes (low
// = first), and the rounded values back in fp32.
__device__ __forceinline__ float2 e4m3_round2(float2 v, uint32_t& bytes) {
  const __nv_fp8x2_storage_t b = __nv_cvt_float2_to_fp8x2(v, __NV_SATFINITE, __NV_E4M3);
  bytes = static_cast<uint32_t>(b);
  const __half2_raw hr = __nv_cvt_fp8x2_to_halfraw2(b, __NV_E4M3);
  return __half22float2(__half2(hr));
}

// ---------------------------------------------------------------- main kernel
// The unit sequence of CTA b: units [u0, u1) of the tile-major (tile, stage)
// order; segments are its runs of one tile.
struct UnitRange {
  int u0, u1;
};

__device__ __forceinline__ UnitRange cta_units(const F8Args& a) {
  UnitRange r;
  r.u0 = blockIdx.x * a.units_per_cta;
  r.u1 = min(a.total_units, r.u0 + a.units_per_cta);
  return r;
}

__global__ void __launch_bounds__(kThreads, 1) gemv_f8_kernel(const __grid_constant__ F8Args a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_addr(smem_raw) & 1023u)) & 1023u);
  const int CS = a.cstages;
  uint8_t* cring = smem;                                            // CS x 16 KiB
  uint8_t* bres = cring + CS * kCodeStageBytes;                     // nks x 4 KiB x terms
  uint8_t* bzero = bres + static_cast<size_t>(a.nks) * kBStageBytes;   // 1 KiB of zeros
  F8Smem* sh = reinterpret_cast<F8Smem*>(bzero + 1024);
  volatile int* abort_flag = &sh->abort;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const UnitRange ur = cta_units(a);

  if (threadIdx.x == 0) {
    for (int i = 0; i < CS; ++i) {
      mbar_init(&sh->full_c[i], 1);
      mbar_init(&sh->empty_c[i], kDecWarps);
    }
    for (int i = 0; i < kAStages; ++i) {
      mbar_init(&sh->full_a[i], kDecWarps);
      mbar_init(&sh->empty_a[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sh->acc_full[i], 1);
      mbar_init(&sh->acc_empty[i], kEpiWarps);
    }
    mbar_init(&sh->drain, 1);
    sh->abort = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(&sh->tmem_base, kTmemCols);
    tmem_relinquish();
  }
  // zero the x-term region (rows 3..7 of every atom stay zero) and the zero atom
  {
    uint4* z = reinterpret_cast<uint4*>(bres);
    const int n16 = (a.nks * kBStageBytes + 1024) / 16;
    for (int i = threadIdx.x; i < n16; i += kThreads) z[i] = make_uint4(0u, 0u, 0u, 0u);
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  // the CTA allocates all 512 columns, so the allocation starts at column 0
  if (sh->tmem_base != 0u) {
    if (threadIdx.x == 0) {
      raise_device_error(a.err, TBN_DEVERR_BAD_LAUNCH);
      sh->abort = 1;
    }
  }
  __syncthreads();
  if (*abort_flag) {
    if (warp == 1) tmem_dealloc(sh->tmem_base, kTmemCols);
    return;
  }
  constexpr uint32_t tmem = 0;

  if (warp == 0) {
    // ================= producer: code boxes =================
    int g = 0;
    bool ok = true;
    for (int u = ur.u0; u < ur.u1 && ok; ++u, ++g) {
      const int s = g % CS;
      if (g >= CS)
        ok = mbar_wait(&sh->empty_c[s], static_cast<uint32_t>((g / CS) - 1) & 1u, abort_flag,
                       a.err, kWaitLimitNs);
      if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
      if (elect_one()) {
        // unit u = (tile, stage) is the u-th 16 KiB block of the prepared words
        mbar_arrive_expect_tx(&sh->full_c[s], kCodeStageBytes);
        bulk_load_1d(cring + s * kCodeStageBytes,
                     a.prepared + static_cast<size_t>(u) * (kRows * kStageWords), kCodeStageBytes,
                     &sh->full_c[s]);
      }
      __syncwarp();
    }
    // every copy issued must land before the CTA may exit
    for (int i = g > CS ? g - CS : 0; i < g; ++i)
      mbar_wait(&sh->full_c[i % CS], static_cast<uint32_t>(i / CS) & 1u, nullptr, a.err,
                kWaitLimitNs);
  } else {
    // The exact three-term split of x (which may come from the previous
    // kernel), done by every CTA for the whole vector while its first code
    // stages are in flight, straight into the resident B region: input k of
    // term r goes to atom (k / 512, (k % 512) / 128), row r, 16-byte chunk
    // ((k % 128) / 16) ^ r, byte k % 16.  E from max |x| (the bit pattern of
    // a finite bf16 |x| orders like |x|).  All warps but the producer take
    // part, with every thread's loads in flight at once.
    grid_dependency_wait();
    grid_dependents_launch();
    const int nt = kThreads - 32, tid = threadIdx.x - 32;
    {
      // max |x|: at most 16384 / 8 / 416 < 5 loads per thread, all in flight
      const uint4* x4 = reinterpret_cast<const uint4*>(a.x);
      uint4 xv[5];
#pragma unroll
      for (int k = 0; k < 5; ++k) {
        const int i = tid + k * nt;
        xv[k] = i < a.K_in / 8 ? __ldg(x4 + i) : make_uint4(0u, 0u, 0u, 0u);
      }
      uint32_t mx = 0;
#pragma unroll
      for (int k = 0; k < 5; ++k) {
        const uint4 v = xv[k];
        mx = max(mx, max(max(v.x & 0x7FFF7FFFu, v.y & 0x7FFF7FFFu),
                         max(v.z & 0x7FFF7FFFu, v.w & 0x7FFF7FFFu)) >> 16);
        mx = max(mx, max(max(v.x & 0x7FFFu, v.y & 0x7FFFu), max(v.z & 0x7FFFu, v.w & 0x7FFFu)));
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) mx = max(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      if (lane == 0) sh->red[warp] = mx;
      named_barrier_sync(1, nt);
      if (warp == 1) {
        uint32_t v = lane >= 1 && lane < kThreads / 32 ? sh->red[lane] : 0u;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) v = max(v, __shfl_xor_sync(0xffffffffu, v, o));
        if (lane == 0) {
          const float mf = __uint_as_float(v << 16);
          int ex = 0;
          if (mf > 0.0f) frexpf(mf, &ex);   // mf in [2^(ex-1), 2^ex)
          sh->E = mf > 0.0f ? 8 - ex : 0;   // max |x| 2^E in [128, 256)
        }
      }
      named_barrier_sync(1, nt);
      const int E = sh->E;
      // 2^E as two normal fp32 factors (|E| <= 140): x 2^E is exact for every
      // x that stays normal, and an x that does not is below 2^-25 max |x|
      const int E1 = E / 2, E2 = E - E / 2;
      const float sc1 = __int_as_float((127 + E1) << 23), sc2 = __int_as_float((127 + E2) << 23);
      // the terms: groups of four consecutive inputs (one 32-bit word of each
      // term), at most 16384 / 4 / 416 < 10 per thread, loads all in flight
      const uint2* x2 = reinterpret_cast<const uint2*>(a.x);
      uint2 xq[10];
#pragma unroll
      for (int k = 0; k < 10; ++k) {
        const int i = tid + k * nt;
        xq[k] = i < a.K_in / 4 ? __ldg(x2 + i) : make_uint2(0u, 0u);
      }
#pragma unroll
      for (int k = 0; k < 10; ++k) {
        const int i = tid + k * nt;
        if (i >= a.K_in / 4) break;
        uint32_t w1 = 0, w2 = 0, w3 = 0;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const uint32_t xw = h ? xq[k].y : xq[k].x;
          const float2 v = make_float2(__uint_as_float(xw << 16) * sc1 * sc2,
                                       __uint_as_float(xw & 0xFFFF0000u) * sc1 * sc2);
          uint32_t b1, b2, b3;
          const float2 t1 = e4m3_round2(v, b1);
          const float2 r1 = make_float2(v.x - t1.x, v.y - t1.y);
          const float2 t2 = e4m3_round2(make_float2(r1.x * 16.0f, r1.y * 16.0f), b2);
          const float2 r2 = make_float2(r1.x - t2.x * 0.0625f, r1.y - t2.y * 0.0625f);
          e4m3_round2(make_float2(r2.x * 256.0f, r2.y * 256.0f), b3);
          w1 |= b1 << (16 * h);
          w2 |= b2 << (16 * h);
          w3 |= b3 << (16 * h);
        }
        const int kk = 4 * i;
        const int ks = kk / kStageCodes, c = (kk % kStageCodes) / 128, q = (kk % 128) / 16, b = kk % 16;
        uint8_t* at = bres + ks * kBStageBytes + c * 1024 + b;
        *reinterpret_cast<uint32_t*>(at + 0 * 128 + ((q ^ 0) << 4)) = w1;
        *reinterpret_cast<uint32_t*>(at + 1 * 128 + ((q ^ 1) << 4)) = w2;
        *reinterpret_cast<uint32_t*>(at + 2 * 128 + ((q ^ 2) << 4)) = w3;
      }
    }
    fence_proxy_async_smem();   // generic writes -> visible to tcgen05.mma
    named_barrier_sync(1, nt);

    if (warp == 1) {
      // ================= MMA issuer =================
      const uint32_t idesc = idesc_e4m3_f32(kRows, kDCols);
      const uint32_t zero_s = smem_addr(bzero);
      int g = 0, seg = 0, issued = 0;
      bool ok = true;
      for (int u = ur.u0; u < ur.u1 && ok;) {
        const int t = u / a.nks;
        const int uend = min(ur.u1, (t + 1) * a.nks);
        const int useg = u;   // the segment's first unit starts a fresh accumulation
        const int ds = seg & 1;
        // the epilogue must have read this accumulator slot's previous segment
        if (seg >= 2)
          ok = mbar_wait(&sh->acc_empty[ds], static_cast<uint32_t>((seg >> 1) - 1) & 1u, abort_flag,
                         a.err, kWaitLimitNs);
        if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
        tc_fence_after_sync();
        for (; u < uend; ++u, ++g) {
          const int ks = u - t * a.nks;
          const int s = g % kAStages;
          ok = mbar_wait(&sh->full_a[s], static_cast<uint32_t>(g / kAStages) & 1u, abort_flag, a.err,
                         kWaitLimitNs);
          if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
          tc_fence_after_sync();
          if (elect_one()) {
            const uint32_t acol = tmem + kAColBase + static_cast<uint32_t>(s * kACols);
#pragma unroll
            for (int kk = 0; kk < kStageCodes / 32; ++kk) {
              const uint32_t atom = smem_addr(bres + ks * kBStageBytes + (kk >> 2) * 1024);
              const uint64_t bdesc = desc_sw128(atom + 32u * (kk & 3), zero_s - atom);
              mma_f8_ts(tmem + static_cast<uint32_t>(ds * kDCols), acol + 8u * kk, bdesc, idesc,
                        (u == useg && kk == 0) ? 0u : 1u);
            }
            tc_commit(&sh->empty_a[s]);
          }
          __syncwarp();
          ++issued;
        }
        if (!ok) break;
        if (elect_one()) tc_commit(&sh->acc_full[ds]);
        __syncwarp();
        ++seg;
      }
      if (!ok && issued > 0) {
        if (elect_one()) tc_commit(&sh->drain);
        __syncwarp();
        mbar_wait(&sh->drain, 0u, nullptr, a.err, kWaitLimitNs);
      }
    } else if (warp >= kFirstDecWarp && warp < kFirstDecWarp + kDecWarps) {
      // ================= decoders =================
      const int sub = warp & 3;
      const int quarter = (warp - kFirstDecWarp) >> 2;  // words [8 quarter, 8 quarter + 8) of a stage
      const int m = sub * 32 + lane;                   // tile row = tensor-memory lane
      const uint32_t lane_off = static_cast<uint32_t>(sub * 32) << 16;
      // opaque multipliers 2^(3-j): keep the multiply-add on the FMA pipe
      uint32_t mul[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) asm("mov.b32 %0, %1;" : "=r"(mul[j]) : "r"(1u << (3 - j)));
      // unit gg's 8 words of this row, decoded: wait for the code stage,
      // two 16-byte chunks (2 quarter, 2 quarter + 1 of row m), release it
      auto fetch = [&](int gg, uint32_t (&v)[32]) -> bool {
        const int sc = gg % CS;
        const bool r = mbar_wait(&sh->full_c[sc], static_cast<uint32_t>(gg / CS) & 1u, abort_flag,
                                 a.err, kWaitLimitNs);
        if (!__all_sync(0xffffffffu, r)) return false;
        const uint8_t* row = cring + sc * kCodeStageBytes + m * 128;
        uint4 wv[2];
#pragma unroll
        for (int c = 0; c < 2; ++c)
          wv[c] = *reinterpret_cast<const uint4*>(row + (((2 * quarter + c) ^ (m & 7)) << 4));
        __syncwarp();
        if (lane == 0) mbar_arrive(&sh->empty_c[sc]);
#pragma unroll
        for (int c = 0; c < 2; ++c) {
          const uint32_t w4[4] = {wv[c].x, wv[c].y, wv[c].z, wv[c].w};
#pragma unroll
          for (int q = 0; q < 4; ++q)
#pragma unroll
            for (int j = 0; j < 4; ++j)
              v[16 * c + 4 * q + j] = (w4[q] & (0x11111111u << j)) * mul[j] + 0x30303030u;
        }
        return true;
      };
      // unit gg's 32 columns into its tensor-memory slot, then publish it
      auto put = [&](int gg, const uint32_t (&v)[32]) -> bool {
        const int sa = gg % kAStages;
        if (gg >= kAStages) {
          const bool r = mbar_wait(&sh->empty_a[sa], static_cast<uint32_t>((gg / kAStages) - 1) & 1u,
                                   abort_flag, a.err, kWaitLimitNs);
          if (!__all_sync(0xffffffffu, r)) return false;
        }
        tc_fence_after_sync();
        tmem_st_32x32b_x32(tmem + lane_off + kAColBase + static_cast<uint32_t>(sa * kACols + 32 * quarter), v);
        tmem_wait_st();
        tc_fence_before_sync();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sh->full_a[sa]);
        return true;
      };
      const int n = ur.u1 - ur.u0;
      uint32_t v[32];
      for (int g = 0; g < n; ++g)
        if (!fetch(g, v) || !put(g, v)) break;
    } else if (warp >= kFirstEpiWarp) {
      // ================= epilogue: a segment's partial sums =================
      const int sub = warp & 3;
      const int m = sub * 32 + lane;
      const uint32_t lane_off = static_cast<uint32_t>(sub * 32) << 16;
      const float unscale = ldexpf(1.0f, -sh->E);
      int seg = 0;
      bool ok = true;
      for (int u = ur.u0; u < ur.u1; ++seg) {
        const int t = u / a.nks;
        const int uend = min(ur.u1, (t + 1) * a.nks);
        const int ds = seg & 1;
        if (ok)
          ok = mbar_wait(&sh->acc_full[ds], static_cast<uint32_t>(seg >> 1) & 1u, abort_flag, a.err,
                         kWaitLimitNs);
        if (!__all_sync(0xffffffffu, ok)) break;
        tc_fence_after_sync();
        uint32_t d[32];
        tmem_ld_32x32b_x32(tmem + lane_off + static_cast<uint32_t>(ds * kDCols), d);
        tmem_wait_ld();
        tc_fence_before_sync();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sh->acc_empty[ds]);
        const float p = (__uint_as_float(d[0]) + __uint_as_float(d[1]) * 0.0625f +
                         __uint_as_float(d[2]) * 0.00390625f) * unscale;
        if (a.direct) {
          // the whole tile was this segment: y = 2 alpha p (+ residual), ReLU
          const int k = t * kRows + m;
          if (k < a.K_out) {
            float yv = 2.0f * __ldg(a.alpha + k) * p;
            if (a.y_bf16) {
              if (a.residual) yv += __bfloat162float(static_cast<const __nv_bfloat16*>(a.residual)[k]);
              if (a.relu) yv = fmaxf(yv, 0.0f);
              static_cast<__nv_bfloat16*>(a.y)[k] = __float2bfloat16_rn(yv);
            } else {
              if (a.residual) yv += static_cast<const float*>(a.residual)[k];
              if (a.relu) yv = fmaxf(yv, 0.0f);
              static_cast<float*>(a.y)[k] = yv;
            }
          }
        } else {
          // slot of this CTA among the CTAs that cover tile t
          const int first = (t * a.nks) / a.units_per_cta;
          a.partial[(static_cast<size_t>(t) * a.maxc + (blockIdx.x - first)) * kRows + m] = p;
        }
        u = uend;
      }
    }
  }
  tc_fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after_sync();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// y[k] = 2 alpha[k] (sum of tile k / 128's partial slots in CTA order)
// (+ residual), ReLU, rounded to y's dtype.
__global__ void __launch_bounds__(256) gemv_f8_reduce_kernel(const float* __restrict__ partial,
                                                             const float* __restrict__ alpha,
                                                             const void* residual, int relu,
                                                             void* y, int y_bf16, int K_out, int nks,
                                                             int units_per_cta, int maxc) {
  grid_dependency_wait();   // the partial sums come from the previous kernel
  const int k = blockIdx.x * blockDim.x + threadIdx.x;
  if (k >= K_out) return;
  const int t = k / kRows, m = k - t * kRows;
  const int first = (t * nks) / units_per_cta, last = ((t + 1) * nks - 1) / units_per_cta;
  float acc = 0.0f;
  for (int c = 0; c <= last - first; ++c) acc += partial[(static_cast<size_t>(t) * maxc + c) * kRows + m];
  float v = 2.0f * alpha[k] * acc;
  if (y_bf16) {
    if (residual) v += __bfloat162float(static_cast<const __nv_bfloat16*>(residual)[k]);
    if (relu) v = fmaxf(v, 0.0f);
    static_cast<__nv_bfloat16*>(y)[k] = __float2bfloat16_rn(v);
  } else {
    if (residual) v += static_cast<const float*>(residual)[k];
    if (relu) v = fmaxf(v, 0.0f);
    static_cast<float*>(y)[k] = v;
  }
}

// ---------------------------------------------------------------- host side
struct F8Plan {
  int tiles, nks, grid, units_per_cta, total_units, maxc, cstages, direct;
  size_t smem, bytes;
};

F8Plan plan_f8(int64_t K_in, int64_t K_out, int sms) {
  F8Plan p{};
  p.tiles = static_cast<int>((K_out + kRows - 1) / kRows);
  p.nks = static_cast<int>(K_in / kStageCodes);
  p.total_units = p.tiles * p.nks;
  if (5 * p.tiles >= 4 * sms) {
    // the tiles nearly fill the SMs: whole tiles per CTA, no partial sums
    p.units_per_cta = p.nks * ((p.tiles + sms - 1) / sms);
  } else {
    // stream-K: equal ranges of (tile, stage) units, split tiles reduced after
    const int grid0 = std::min(sms, p.total_units);
    p.units_per_cta = (p.total_units + grid0 - 1) / grid0;
  }
  p.grid = (p.total_units + p.units_per_cta - 1) / p.units_per_cta;
  p.maxc = 0;
  for (int t = 0; t < p.tiles; ++t) {
    const int first = (t * p.nks) / p.units_per_cta;
    const int last = ((t + 1) * p.nks - 1) / p.units_per_cta;
    p.maxc = std::max(p.maxc, last - first + 1);
  }
  // the code ring takes what the resident x terms leave of the shared memory
  const size_t fixed = 1024 + static_cast<size_t>(p.nks) * kBStageBytes + 1024 +
                       ((sizeof(F8Smem) + 15) / 16) * 16;
  p.cstages = static_cast<int>(std::min<size_t>(kMaxCodeStages,
                                                (kSmemLimit - fixed) / kCodeStageBytes));
  p.smem = fixed + static_cast<size_t>(p.cstages) * kCodeStageBytes;
  p.direct = p.maxc == 1 ? 1 : 0;
  // workspace: the partial sums of split tiles
  p.bytes = std::max<size_t>(256, p.direct ? 0 : static_cast<size_t>(p.tiles) * p.maxc * kRows * 4);
  return p;
}

}  // namespace

const char* gemv_f8_unsupported_reason(int64_t B, int64_t K_in, int64_t K_out) {
  if (B != 1) return "fp8 GEMV: batch 1 only";
  if (K_in % kStageCodes != 0 || K_in / kStageCodes > kMaxStagesK)
    return "fp8 GEMV: K_in must be a multiple of 512, at most 16384";
  if (K_out < 1 || K_out > (int64_t(1) << 24)) return "fp8 GEMV: K_out out of range";
  return "";
}

size_t gemv_f8_workspace_bytes(int64_t K_in, int64_t K_out) {
  if (K_in % kStageCodes != 0 || K_in / kStageCodes > kMaxStagesK || K_out < 1) return 0;
  return plan_f8(K_in, K_out, device_sm_count()).bytes;
}

int64_t gemv_f8_prepared_words(int64_t K_out, int64_t K_in) {
  return (K_out + kRows - 1) / kRows * kRows * (K_in / 16);
}

tbn_status launch_prepare_f8(const uint32_t* codes, int64_t K_out, int64_t K_in, uint32_t* out,
                             cudaStream_t s) {
  const int64_t total = gemv_f8_prepared_words(K_out, K_in);
  const int64_t blocks = std::min<int64_t>((total + 255) / 256, int64_t(device_sm_count()) * 16);
  prepare_f8_kernel<<<static_cast<unsigned>(std::max<int64_t>(blocks, 1)), 256, 0, s>>>(
      codes, K_out, static_cast<int>(K_in / 16), total, out);
  return check_launch("prepare_f8_kernel");
}

tbn_status launch_gemv_f8(const void* x, int64_t K_in, const uint32_t* prepared, const float* alpha,
                          int64_t K_out, void* y, tbn_dtype ydt, const void* residual, int relu,
                          void* workspace, size_t workspace_bytes, cudaStream_t s) {
  const F8Plan p = plan_f8(K_in, K_out, device_sm_count());
  if (workspace_bytes < p.bytes) return fail(TBN_ERR_INVALID_ARG, "fp8 GEMV: workspace too small");
  float* partial = static_cast<float*>(workspace);
  // 1. the tensor-core pass (it splits x itself)
  {
    static std::once_flag once;
    static cudaError_t attr_err = cudaSuccess;
    std::call_once(once, [&] {
      attr_err = cudaFuncSetAttribute(gemv_f8_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      kSmemLimit);
      if (attr_err == cudaSuccess)
        attr_err = cudaFuncSetAttribute(gemv_f8_kernel, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
    });
    if (attr_err != cudaSuccess) return cuda_fail(attr_err, "cudaFuncSetAttribute(gemv_f8_kernel)");
    if (p.smem > static_cast<size_t>(kSmemLimit)) return fail(TBN_ERR_UNSUPPORTED, "fp8 GEMV: shared memory");
    F8Args a{};
    a.x = static_cast<const __nv_bfloat16*>(x);
    a.partial = partial;
    a.direct = p.direct;
    a.alpha = alpha;
    a.y = y;
    a.residual = residual;
    a.relu = relu;
    a.y_bf16 = ydt == TBN_BF16 ? 1 : 0;
    a.err = device_error_word();
    a.K_out = static_cast<int>(K_out);
    a.K_in = static_cast<int>(K_in);
    a.tiles = p.tiles;
    a.nks = p.nks;
    a.units_per_cta = p.units_per_cta;
    a.total_units = p.total_units;
    a.maxc = p.maxc;
    a.cstages = p.cstages;
    a.prepared = prepared;
    if (p.cstages < 2) return fail(TBN_ERR_UNSUPPORTED, "fp8 GEMV: shared memory");
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(static_cast<unsigned>(p.grid));
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = p.smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const cudaError_t le = cudaLaunchKernelEx(&cfg, gemv_f8_kernel, a);
    if (le != cudaSuccess) return cuda_fail(le, "cudaLaunchKernelEx(gemv_f8_kernel)");
  }
  // 2. split tiles: the ordered sum of the partial slots and the epilogue
  if (!p.direct) {
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(static_cast<unsigned>((K_out + 255) / 256));
    cfg.blockDim = dim3(256);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const cudaError_t le = cudaLaunchKernelEx(&cfg, gemv_f8_reduce_kernel, (const float*)partial, alpha,
                                              residual, relu, y, ydt == TBN_BF16 ? 1 : 0, (int)K_out,
                                              p.nks, p.units_per_cta, p.maxc);
    if (le != cudaSuccess) return cuda_fail(le, "cudaLaunchKernelEx(gemv_f8_reduce_kernel)");
  }
  return check_launch("gemv_f8");
}

}  // namespace tbn
