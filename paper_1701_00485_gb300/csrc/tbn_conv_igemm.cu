// tbn_conv_igemm.cu -- two-bit convolution (Eq. 1, Section 2) as an
// implicit GEMM on the sm_100-family tensor cores (tcgen05), NHWC bf16.
//
// GEMM view of one CTA tile:  D[128 filters x T pixels] = A[128 x K] * B[K x T]
// with K = R*S*C walked in blocks of one filter tap (r, s) x 64 channels.
//
//   A (filters)     the 2-bit codes, decoded in registers to bf16 W~/2 in
//                   {+-0.5, +-1} (exact) and written straight into tensor
//                   memory (tcgen05.st) by four "expander" warps: thread i
//                   owns filter row i = TMEM lane i.  The decoded weights
//                   never touch shared memory, so shared-memory bandwidth is
//                   left to the activation operand.
//   B (activations) a box of NHWC pixels x 64 channels loaded by TMA with the
//                   128-byte swizzle; the box is the tile's output pixels
//                   shifted by the tap (zero fill supplies the padding,
//                   element strides supply the convolution stride).
//   D               fp32 in tensor memory; epilogue multiplies row i by
//                   2 * alpha_i (Eq. 1 applies alpha to the whole filter, and
//                   the factor 2 undoes the W~/2 encoding -- both exact
//                   power-of-two / per-row scalings), adds the optional
//                   residual, applies ReLU, and stores NHWC.
//
// Warp roles (192 threads, one CTA per SM):
//   warp 0     TMA producer for the activation ring (one elected lane)
//   warp 1     TMEM allocator + MMA issuer (one elected lane)
//   warps 2-5  expanders during the main loop, epilogue afterwards
// All waits are bounded (see tbn_device.cuh); on a timeout the CTA records
// the error, drains its own in-flight copies and MMAs, frees TMEM, returns.
#include <cuda.h>
#include <cuda_bf16.h>

#include <algorithm>
#include <cstdint>
#include <cstring>
#include <mutex>

#include "tbn_device.cuh"
#include "tbn_internal.h"

namespace tbn {
namespace {

constexpr int kBM = 128;            // filters per tile = TMEM lanes
constexpr int kBKC = 64;            // channels per K block (128-byte rows)
constexpr int kMaxTileN = 256;      // pixels per tile (MMA N) upper bound
constexpr int kStagesB = 6;         // activation ring depth (shared memory)
constexpr int kStagesA = 8;         // weight ring depth (tensor memory)
constexpr int kAColsPerStage = kBKC / 2;   // 64 bf16 = 32 columns of 32 bits
constexpr int kAccCols = 256;
constexpr int kTmemCols = 512;      // accumulator [0,256) + weight ring [256,512)
constexpr int kThreads = 192;
constexpr int kStageBytes = kMaxTileN * kBKC * 2;   // 32 KiB
constexpr uint64_t kWaitLimitNs = 1000000000ull;    // 1 s

static_assert(kAccCols + kStagesA * kAColsPerStage <= kTmemCols, "TMEM budget");
static_assert(kMaxTileN * kBM * 4 <= kStagesB * kStageBytes, "epilogue staging fits the ring");

struct IgArgs {
  int N, C, H, W, K, R, S, sh, sw, ph, pw, P, Q;
  int bw, bh, bn;          // output pixels per tile along q, p, image
  int tile_n;              // MMA N: bw*bh*bn rounded up to 16
  int tiles_q, tiles_p, tiles_k;
  int cblocks, kblocks, wpf;
  const uint32_t* codes;
  const float* alpha;
  void* y;
  const void* residual;
  int relu, y_bf16;
  uint32_t* err;
};

struct SmemCtl {
  uint64_t b_full[kStagesB];
  uint64_t b_empty[kStagesB];
  uint64_t a_full[kStagesA];
  uint64_t a_empty[kStagesA];
  uint64_t acc_full;
  uint32_t tmem_base;
  int abort;
};

constexpr size_t kSmemBytes = 1024 /*align slack*/ + kStagesB * kStageBytes + sizeof(SmemCtl);

__device__ __forceinline__ void named_barrier_sync(int id, int nthreads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

__global__ void __launch_bounds__(kThreads, 1)
    conv_igemm_kernel(const __grid_constant__ CUtensorMap tmap_x, const __grid_constant__ IgArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* ring = smem;  // kStagesB x 32 KiB, 1024-aligned
  SmemCtl* ctl = reinterpret_cast<SmemCtl*>(smem + kStagesB * kStageBytes);
  volatile int* abort_flag = &ctl->abort;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  // ---- tile coordinates (filter tile fastest: neighbouring CTAs share the
  // activation tile through L2)
  const int lin = blockIdx.x;
  const int ktile = lin % a.tiles_k;
  const int ptile = lin / a.tiles_k;
  const int qt = ptile % a.tiles_q;
  const int pt = (ptile / a.tiles_q) % a.tiles_p;
  const int nt = ptile / (a.tiles_q * a.tiles_p);
  const int q0 = qt * a.bw, p0 = pt * a.bh, n0 = nt * a.bn;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kStagesB; ++i) {
      mbar_init(&ctl->b_full[i], 1);
      mbar_init(&ctl->b_empty[i], 1);
    }
    for (int i = 0; i < kStagesA; ++i) {
      mbar_init(&ctl->a_full[i], 128);
      mbar_init(&ctl->a_empty[i], 1);
    }
    mbar_init(&ctl->acc_full, 1);
    ctl->abort = 0;
    fence_mbar_init();
    prefetch_tmap(&tmap_x);
  }
  if (warp == 1) {
    tmem_alloc(&ctl->tmem_base, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = ctl->tmem_base;
  const uint32_t acc_tmem = tmem;                 // columns [0, tile_n)
  const uint32_t a_tmem0 = tmem + kAccCols;       // weight ring
  const int KB = a.kblocks;

  if (warp == 0) {
    // ================= TMA producer =================
    if (lane == 0) {
      const uint32_t box_bytes = static_cast<uint32_t>(a.bw * a.bh * a.bn * kBKC * 2);
      int issued = 0;
      for (int kb = 0; kb < KB; ++kb) {
        const int sb = kb % kStagesB;
        const uint32_t it = static_cast<uint32_t>(kb / kStagesB);
        if (!mbar_wait(&ctl->b_empty[sb], (it & 1u) ^ 1u, abort_flag, a.err, kWaitLimitNs)) break;
        const int tap = kb / a.cblocks, cb = kb % a.cblocks;
        const int r = tap / a.S, s = tap % a.S;
        mbar_arrive_expect_tx(&ctl->b_full[sb], box_bytes);
        tma_load_4d(ring + sb * kStageBytes, &tmap_x, &ctl->b_full[sb], cb * kBKC,
                    q0 * a.sw - a.pw + s, p0 * a.sh - a.ph + r, n0);
        ++issued;
      }
      // drain: every issued copy must land before the CTA may exit
      for (int i = issued > kStagesB ? issued - kStagesB : 0; i < issued; ++i)
        mbar_wait(&ctl->b_full[i % kStagesB], static_cast<uint32_t>(i / kStagesB) & 1u, nullptr,
                  a.err, kWaitLimitNs);
    }
  } else if (warp == 1) {
    // ================= MMA issuer =================
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16_f32(kBM, static_cast<uint32_t>(a.tile_n));
      int issued = 0;
      for (int kb = 0; kb < KB; ++kb) {
        const int sb = kb % kStagesB, sa = kb % kStagesA;
        if (!mbar_wait(&ctl->a_full[sa], static_cast<uint32_t>(kb / kStagesA) & 1u, abort_flag,
                       a.err, kWaitLimitNs))
          break;
        if (!mbar_wait(&ctl->b_full[sb], static_cast<uint32_t>(kb / kStagesB) & 1u, abort_flag,
                       a.err, kWaitLimitNs))
          break;
        tc_fence_after_sync();
        const uint64_t bdesc = smem_desc_sw128_kmajor(smem_addr(ring + sb * kStageBytes));
        const uint32_t a_col = a_tmem0 + static_cast<uint32_t>(sa * kAColsPerStage);
#pragma unroll
        for (int kk = 0; kk < kBKC / 16; ++kk) {
          // K step kk: 16 channels = 8 TMEM columns of A, 32 bytes of B rows
          tc_mma_ts(acc_tmem, a_col + 8u * kk, bdesc + static_cast<uint64_t>(2 * kk), idesc,
                    (kb | kk) != 0 ? 1u : 0u);
        }
        tc_commit(&ctl->a_empty[sa]);
        tc_commit(&ctl->b_empty[sb]);
        ++issued;
      }
      // accumulator complete (also drains in-flight MMAs after an abort)
      tc_commit(&ctl->acc_full);
      if (*abort_flag && issued > 0)
        mbar_wait(&ctl->acc_full, 0u, nullptr, a.err, kWaitLimitNs);
    }
  } else {
    // ================= expanders, then epilogue =================
    const int sub = warp & 3;             // TMEM sub-partition this warp may access
    const int m = sub * 32 + lane;        // filter row within the tile
    const int k = ktile * kBM + m;
    const bool kvalid = k < a.K;
    const uint32_t lane_off = static_cast<uint32_t>(sub * 32) << 16;
    const uint4* crow = reinterpret_cast<const uint4*>(a.codes + static_cast<size_t>(kvalid ? k : 0) * a.wpf);
    const int cw = a.C / 64;  // uint4 (64 codes) per tap

    auto load_codes = [&](int kb) -> uint4 {
      if (!kvalid || kb >= KB) return make_uint4(0u, 0u, 0u, 0u);
      const int tap = kb / a.cblocks, cb = kb % a.cblocks;
      return __ldg(crow + tap * cw + cb);
    };
    uint4 pf0 = load_codes(0), pf1 = load_codes(1);
    bool ok = true;
    for (int kb = 0; kb < KB; ++kb) {
      const uint4 cur = pf0;
      pf0 = pf1;
      pf1 = load_codes(kb + 2);
      const int sa = kb % kStagesA;
      if (!mbar_wait(&ctl->a_empty[sa], (static_cast<uint32_t>(kb / kStagesA) & 1u) ^ 1u,
                     abort_flag, a.err, kWaitLimitNs)) {
        ok = false;
      }
      ok = __all_sync(0xffffffffu, ok);
      if (!ok) break;
      tc_fence_after_sync();
      uint32_t v[32];
      word_to_bf16x2(cur.x, v + 0);
      word_to_bf16x2(cur.y, v + 8);
      word_to_bf16x2(cur.z, v + 16);
      word_to_bf16x2(cur.w, v + 24);
      tmem_st_32x32b_x32(a_tmem0 + lane_off + static_cast<uint32_t>(sa * kAColsPerStage), v);
      tmem_wait_st();
      tc_fence_before_sync();
      mbar_arrive(&ctl->a_full[sa]);
    }

    // ---- epilogue
    bool acc_ok = ok && mbar_wait(&ctl->acc_full, 0u, abort_flag, a.err, kWaitLimitNs);
    acc_ok = __all_sync(0xffffffffu, acc_ok);
    // all four epilogue warps must agree before touching the staging buffer
    __shared__ int s_epi_ok;
    if (threadIdx.x == 64) s_epi_ok = 1;
    named_barrier_sync(1, 128);
    if (!acc_ok && lane == 0) atomicAnd(&s_epi_ok, 0);
    named_barrier_sync(1, 128);
    if (s_epi_ok && !*abort_flag) {
      tc_fence_after_sync();
      float* stage = reinterpret_cast<float*>(ring);  // [tile_n][128] fp32
      const float a2 = kvalid ? 2.0f * a.alpha[k] : 0.0f;
      // columns beyond tile_n (up to the next multiple of 32) hold garbage
      // and land in staging rows that the copy-out never reads
      for (int j = 0; j < (a.tile_n + 31) / 32; ++j) {
        uint32_t v[32];
        tmem_ld_32x32b_x32(acc_tmem + lane_off + static_cast<uint32_t>(32 * j), v);
        tmem_wait_ld();
#pragma unroll
        for (int i = 0; i < 32; ++i) stage[(32 * j + i) * kBM + m] = a2 * __uint_as_float(v[i]);
      }
      named_barrier_sync(1, 128);
      // copy-out: 16 threads per pixel row, 8 filters (one 16-byte bf16 vector) each
      const int e = threadIdx.x - 64;
      const int c8 = (e & 15) * 8;
      const int npix_tile = a.bw * a.bh * a.bn;
      const int kbase = ktile * kBM + c8;
      const bool vec_ok = (a.K % 8) == 0 && kbase + 8 <= a.K;
      for (int pr = e >> 4; pr < npix_tile; pr += 8) {
        const int wi = pr % a.bw, hi = (pr / a.bw) % a.bh, ni = pr / (a.bw * a.bh);
        const int q = q0 + wi, p = p0 + hi, n = n0 + ni;
        if (q >= a.Q || p >= a.P || n >= a.N || kbase >= a.K) continue;
        const size_t o = ((static_cast<size_t>(n) * a.P + p) * a.Q + q) * a.K + kbase;
        const float4 lo = *reinterpret_cast<const float4*>(&stage[pr * kBM + c8]);
        const float4 hi4 = *reinterpret_cast<const float4*>(&stage[pr * kBM + c8 + 4]);
        float v[8] = {lo.x, lo.y, lo.z, lo.w, hi4.x, hi4.y, hi4.z, hi4.w};
        if (vec_ok) {
          if (a.y_bf16) {
            if (a.residual) {
              const uint4 rr = *reinterpret_cast<const uint4*>(
                  static_cast<const __nv_bfloat16*>(a.residual) + o);
              const __nv_bfloat16* rb = reinterpret_cast<const __nv_bfloat16*>(&rr);
#pragma unroll
              for (int i = 0; i < 8; ++i) v[i] += __bfloat162float(rb[i]);
            }
            uint4 out;
            __nv_bfloat16* ob = reinterpret_cast<__nv_bfloat16*>(&out);
#pragma unroll
            for (int i = 0; i < 8; ++i) ob[i] = __float2bfloat16_rn(a.relu ? fmaxf(v[i], 0.0f) : v[i]);
            *reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(a.y) + o) = out;
          } else {
            if (a.residual) {
              const float4* rp = reinterpret_cast<const float4*>(static_cast<const float*>(a.residual) + o);
              const float4 r0 = rp[0], r1 = rp[1];
              v[0] += r0.x; v[1] += r0.y; v[2] += r0.z; v[3] += r0.w;
              v[4] += r1.x; v[5] += r1.y; v[6] += r1.z; v[7] += r1.w;
            }
            if (a.relu) {
#pragma unroll
              for (int i = 0; i < 8; ++i) v[i] = fmaxf(v[i], 0.0f);
            }
            float4* yp = reinterpret_cast<float4*>(static_cast<float*>(a.y) + o);
            yp[0] = make_float4(v[0], v[1], v[2], v[3]);
            yp[1] = make_float4(v[4], v[5], v[6], v[7]);
          }
        } else {
          for (int i = 0; i < 8 && kbase + i < a.K; ++i) {
            float t = v[i];
            if (a.y_bf16) {
              if (a.residual) t += __bfloat162float(static_cast<const __nv_bfloat16*>(a.residual)[o + i]);
              if (a.relu) t = fmaxf(t, 0.0f);
              static_cast<__nv_bfloat16*>(a.y)[o + i] = __float2bfloat16_rn(t);
            } else {
              if (a.residual) t += static_cast<const float*>(a.residual)[o + i];
              if (a.relu) t = fmaxf(t, 0.0f);
              static_cast<float*>(a.y)[o + i] = t;
            }
          }
        }
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

// ---------------------------------------------------------------- host side
using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                   const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                   const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

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

struct TilePlan {
  int bw, bh, bn, T, tile_n, tiles_q, tiles_p, tiles_n;
};

int ceil_div(int64_t a, int64_t b) { return static_cast<int>((a + b - 1) / b); }

// Output pixels per tile: whole rows of the output (so one TMA box per tap
// covers the tile), balanced so the last tile along each axis is not a
// sliver, at most 256 pixels.
TilePlan plan_tiles(const ConvProblem& p) {
  TilePlan t{};
  const int bw_max = std::min<int64_t>(p.Q, kMaxTileN / p.sw);
  t.tiles_q = ceil_div(p.Q, bw_max);
  t.bw = ceil_div(p.Q, t.tiles_q);
  if (t.tiles_q > 1) {
    t.bh = 1;
    t.bn = 1;
  } else {
    const int bh_max = static_cast<int>(std::min<int64_t>({p.P, kMaxTileN / t.bw, kMaxTileN / p.sh}));
    const int tp = ceil_div(p.P, bh_max);
    t.bh = ceil_div(p.P, tp);
    if (tp > 1) {
      t.bn = 1;
    } else {
      const int bn_max = static_cast<int>(std::min<int64_t>(p.N, kMaxTileN / (t.bw * t.bh)));
      t.bn = ceil_div(p.N, ceil_div(p.N, bn_max));
    }
  }
  t.tiles_p = ceil_div(p.P, t.bh);
  t.tiles_n = ceil_div(p.N, t.bn);
  t.T = t.bw * t.bh * t.bn;
  t.tile_n = ((t.T + 15) / 16) * 16;
  return t;
}

}  // namespace

const char* conv_igemm_unsupported_reason(const ConvProblem& p) {
  if (p.layout != TBN_NHWC) return "implicit GEMM needs NHWC";
  if (p.xdt != TBN_BF16) return "implicit GEMM needs bf16 activations";
  if (p.C % kBKC != 0) return "implicit GEMM needs C % 64 == 0";
  if (!is_aligned(p.x, 16)) return "implicit GEMM needs 16-byte aligned x";
  if (!is_aligned(p.codes, 16)) return "implicit GEMM needs 16-byte aligned codes";
  if (p.sh < 1 || p.sh > 2 || p.sw < 1 || p.sw > 2) return "implicit GEMM supports stride 1 or 2";
  if (p.residual && !is_aligned(p.residual, 16)) return "implicit GEMM needs 16-byte aligned residual";
  if (!is_aligned(p.y, 16)) return "implicit GEMM needs 16-byte aligned y";
  if (p.N > (1 << 30) || p.H > (1 << 30) || p.W > (1 << 30)) return "dimension too large";
  if (p.ph > p.R || p.pw > p.S) return "implicit GEMM needs pad <= kernel extent";
  int dev = 0, major = 0, minor = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return "no CUDA device";
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
  if (major != 10 || minor != 3) return "implicit GEMM kernel is built for sm_103a only";
  if (get_encode_tiled() == nullptr) return "cuTensorMapEncodeTiled unavailable";
  return "";
}

tbn_status launch_conv_igemm(const ConvProblem& p, cudaStream_t s) {
  const TilePlan t = plan_tiles(p);
  IgArgs a{};
  a.N = (int)p.N; a.C = (int)p.C; a.H = (int)p.H; a.W = (int)p.W; a.K = (int)p.K;
  a.R = (int)p.R; a.S = (int)p.S; a.sh = (int)p.sh; a.sw = (int)p.sw;
  a.ph = (int)p.ph; a.pw = (int)p.pw; a.P = (int)p.P; a.Q = (int)p.Q;
  a.bw = t.bw; a.bh = t.bh; a.bn = t.bn; a.tile_n = t.tile_n;
  a.tiles_q = t.tiles_q; a.tiles_p = t.tiles_p;
  a.tiles_k = ceil_div(p.K, kBM);
  a.cblocks = (int)(p.C / kBKC);
  a.kblocks = (int)(p.R * p.S) * a.cblocks;
  a.wpf = (int)((p.C * p.R * p.S + 15) / 16);
  a.codes = p.codes; a.alpha = p.alpha; a.y = p.y; a.residual = p.residual;
  a.relu = p.relu; a.y_bf16 = p.ydt == TBN_BF16 ? 1 : 0;
  a.err = device_error_word();

  const int64_t grid = static_cast<int64_t>(t.tiles_q) * t.tiles_p * t.tiles_n * a.tiles_k;
  if (grid > 0x7fffffffLL) return fail(TBN_ERR_UNSUPPORTED, "implicit GEMM: grid too large");

  CUtensorMap tmap;
  std::memset(&tmap, 0, sizeof(tmap));
  const cuuint64_t gdim[4] = {(cuuint64_t)p.C, (cuuint64_t)p.W, (cuuint64_t)p.H, (cuuint64_t)p.N};
  const cuuint64_t gstride[3] = {(cuuint64_t)(p.C * 2), (cuuint64_t)(p.W * p.C * 2),
                                 (cuuint64_t)(p.H * p.W * p.C * 2)};
  const cuuint32_t box[4] = {(cuuint32_t)kBKC, (cuuint32_t)(t.bw * p.sw), (cuuint32_t)(t.bh * p.sh),
                             (cuuint32_t)t.bn};
  const cuuint32_t estr[4] = {1u, (cuuint32_t)p.sw, (cuuint32_t)p.sh, 1u};
  if (box[1] > 256 || box[2] > 256 || box[3] > 256)
    return fail(TBN_ERR_UNSUPPORTED, "implicit GEMM: TMA box too large");
  const CUresult cr = get_encode_tiled()(&tmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4,
                                         const_cast<void*>(p.x), gdim, gstride, box, estr,
                                         CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                                         CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                                         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (cr != CUDA_SUCCESS) return fail(TBN_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", (int)cr);

  static bool attr_done[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64 || !attr_done[dev]) {
    const cudaError_t e = cudaFuncSetAttribute(conv_igemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               (int)kSmemBytes);
    if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(conv_igemm_kernel)");
    if (dev >= 0 && dev < 64) attr_done[dev] = true;
  }
  conv_igemm_kernel<<<(unsigned)grid, kThreads, kSmemBytes, s>>>(tmap, a);
  return check_launch("conv_igemm_kernel");
}

}  // namespace tbn
