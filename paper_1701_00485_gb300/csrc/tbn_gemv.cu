// tbn_gemv.cu -- small-batch two-bit fully-connected layer (Section 3: a
// fully-connected layer is a convolution whose filters span the whole
// input), y[b, k] = alpha_k * sum_j x[b, j] W~[k, j] for 1 <= B <= 8.
//
// The packed weight stream (K_in / 4 bytes per output) dominates the
// traffic, so the kernel is organised to keep HBM busy and to spend as few
// issue slots as possible per weight:
//
// * Persistent CTAs, at most one per SM.  The K_out / 16 row tiles are cut
//   into bands of n_t consecutive tiles (n_t <= 16, balanced to within one
//   tile across the grid); a CTA processes `rounds` bands.
// * One producer warp streams a band through an mbarrier ring with TMA.  A
//   stage holds 512 input positions: a [16 n_t rows x 32 words] box of
//   packed codes with the 128-byte swizzle, and the matching inputs of all
//   B batch rows laid out [64 chunks][B][8 bf16], so the eight batch rows
//   of one 8-wide chunk are one contiguous 128-byte ldmatrix read.
// * Sixteen consumer warps: P = 16 / n_t warps per tile split the tile's
//   stages (ring iteration i of the CTA goes to warp i % P of each tile) and
//   their partial sums are added in a fixed order.  The ring depth is a
//   multiple of P, so the previous use of the slot a warp waits on was that
//   warp's own: a slot is never more than one phase ahead of its waiter,
//   which is what a parity wait on an mbarrier can tell apart.  Per K step of 16 a warp runs
//   one mma.m16n8k16: A = 16 rows x 16 codes decoded in registers to bf16
//   W~/2, B = 16 inputs x 8 batch columns (lanes past B read batch row
//   n mod B, which only fills mma columns that are dropped), fp32
//   accumulation.  Lane (g, t) of the A fragment holds pairs t and
//   t + 4 of the K step's word of rows g and g + 8; with the byte-planar
//   packing a pair is one mask and one multiply-add.  2 alpha is applied
//   in the epilogue (W~/2 is exact in bf16).
//
// Every mbarrier wait is bounded; on expiry the kernel records a timeout in
// the device error word, stops issuing, drains the copies it started and
// returns.
//
// The kernel is launched as a programmatic dependent of the previous kernel
// on the stream: the first ring's worth of code boxes is requested before
// griddepcontrol.wait, the inputs (and the residual) only after it, so in a
// chain of layers the weight stream of one starts while the previous one
// finishes.  Codes and alpha must therefore not be the output of the
// immediately preceding call when that call is one of this library's
// kernels that let their dependents start early.
#include <cuda.h>
#include <cuda_bf16.h>

#include <cstdint>
#include <mutex>
#include <utility>

#include "tbn_device.cuh"
#include "tbn_internal.h"

namespace tbn {
namespace {

constexpr int kConsumerWarps = 16;
constexpr int kThreads = 32 * (kConsumerWarps + 1);
constexpr int kProducerWarp = kConsumerWarps;
constexpr int kCodesPerStage = 512;           // 32 packed words per row
constexpr int kWordsPerStage = kCodesPerStage / 16;
constexpr int kMaxTilesPerBand = 16;          // TMA box height 256 rows
constexpr int kMaxStages = 16;
constexpr int kSmemBudget = 200 * 1024;
constexpr uint64_t kWaitLimitNs = 1000000000ull;

struct GemvArgs {
  const float* alpha;
  void* y;
  const void* residual;
  uint32_t* err;
  int K_out, K_in, B;
  int T;           // row tiles = ceil(K_out / 16)
  int n_t;         // tiles per band
  int rounds;      // bands per CTA
  int nks;         // stages per band = ceil(K_in / 512)
  int P;           // consumer warps per tile (K split), n_t * P <= 16
  int stages;      // ring depth
  uint32_t w_bytes;      // packed-code bytes per stage = n_t * 2048
  uint32_t stage_bytes;  // w_bytes + B * 1024
  int y_bf16, relu;
};

__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], uint32_t a0, uint32_t a1,
                                               uint32_t a2, uint32_t a3, uint32_t b0,
                                               uint32_t b1) {
  // no side effects beyond its registers: the compiler may schedule it freely
  asm(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
      "{%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// ldmatrix.x4 at addr + kOff (kOff folded into the instruction).
template <int kOff>
__device__ __forceinline__ void ldmatrix_x4(uint32_t (&r)[4], uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4+%5];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr), "n"(kOff)
               : "memory");
}

template <int kOff>
__device__ __forceinline__ uint4 lds128(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4+%5];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "r"(addr), "n"(kOff)
               : "memory");
  return v;
}

// Per-lane decode constants for pairs t and t + 4 (t = lane % 4): the
// pair's bits (at p, 8+p, 16+p, 24+p) are masked and moved to 7, 15, 23,
// 31 by a power-of-two multiply; adding 0x3F003F00 sets the remaining bf16
// bits of +-0.5 / +-1 (no carries: the bit sets are disjoint).
struct PairDecode {
  uint32_t mask_lo, mul_lo, mask_hi, mul_hi;
  __device__ __forceinline__ explicit PairDecode(int t)
      : mask_lo(0x01010101u << t), mask_hi(0x10101010u << t) {
    // The multipliers pass through an opaque move so the compiler keeps the
    // multiply-add (FMA pipe) instead of rewriting it as shift + OR on the
    // integer ALU pipe, which the masks already load.
    asm("mov.b32 %0, %1;" : "=r"(mul_lo) : "r"(1u << (7 - t)));
    asm("mov.b32 %0, %1;" : "=r"(mul_hi) : "r"(1u << (3 - t)));
  }
  __device__ __forceinline__ uint32_t lo(uint32_t w) const {
    return (w & mask_lo) * mul_lo + 0x3F003F00u;
  }
  __device__ __forceinline__ uint32_t hi(uint32_t w) const {
    return (w & mask_hi) * mul_hi + 0x3F003F00u;
  }
};

// A stage of a 16-row tile is 32 K steps of 16, accumulated into two
// independent chains (K step i goes to chain i % 2) so consecutive mma
// instructions do not wait on each other.
//   w_lane: shared address of the tile's row g with this lane's swizzle
//   phase folded in, (row address) | (g << 4).  Rows are 128-byte swizzled
//   (chunk j of row r stored at j ^ (r & 7)), so chunk j of row g is at
//   w_lane ^ (j << 4) and row g + 8 is 1024 bytes further.
//   x_lane: this lane's ldmatrix row address for chunk 0: matrix m =
//   lane / 8 (chunk offset), batch row n = lane % 8.  Lanes with n >= B
//   read row n % B; that only fills mma columns n >= B, which are dropped.
// Operands of one 4-K-step chunk: words 4J .. 4J + 3 of rows g and g + 8
// and the x fragments of chunks 8J .. 8J + 7.
struct ChunkRegs {
  uint4 wa, wb;
  uint32_t b0[4], b1[4];
};

template <int kB, int J>
__device__ __forceinline__ void load_chunk(ChunkRegs& r, uint32_t w_lane, uint32_t x_lane) {
  const uint32_t aw = w_lane ^ static_cast<uint32_t>(J << 4);
  r.wa = lds128<0>(aw);
  r.wb = lds128<1024>(aw);
  ldmatrix_x4<(8 * J) * kB * 16>(r.b0, x_lane);
  ldmatrix_x4<(8 * J + 4) * kB * 16>(r.b1, x_lane);
}

__device__ __forceinline__ void mma_chunk(float (&d)[2][4], const ChunkRegs& r,
                                          const PairDecode& dec) {
  const uint4& wa = r.wa;
  const uint4& wb = r.wb;
  mma_bf16_16816(d[0], dec.lo(wa.x), dec.lo(wb.x), dec.hi(wa.x), dec.hi(wb.x), r.b0[0], r.b0[1]);
  mma_bf16_16816(d[1], dec.lo(wa.y), dec.lo(wb.y), dec.hi(wa.y), dec.hi(wb.y), r.b0[2], r.b0[3]);
  mma_bf16_16816(d[0], dec.lo(wa.z), dec.lo(wb.z), dec.hi(wa.z), dec.hi(wb.z), r.b1[0], r.b1[1]);
  mma_bf16_16816(d[1], dec.lo(wa.w), dec.lo(wb.w), dec.hi(wa.w), dec.hi(wb.w), r.b1[2], r.b1[3]);
}

// Chunk J: issue the loads of chunk J + 1, then the four mma of chunk J
// (the shared-memory loads keep program order, so this is the prefetch).
template <int kB, int J>
__device__ __forceinline__ void tile_chunk(float (&d)[2][4], uint32_t w_lane, uint32_t x_lane,
                                           const PairDecode& dec, ChunkRegs& cur) {
  if constexpr (J + 1 < 8) {
    ChunkRegs nxt;
    load_chunk<kB, J + 1>(nxt, w_lane, x_lane);
    mma_chunk(d, cur, dec);
    cur = nxt;
  } else {
    mma_chunk(d, cur, dec);
  }
}

template <int kB, int... J>
__device__ __forceinline__ void tile_stage_chunks(float (&d)[2][4], uint32_t w_lane,
                                                  uint32_t x_lane, const PairDecode& dec,
                                                  std::integer_sequence<int, J...>) {
  ChunkRegs cur;
  load_chunk<kB, 0>(cur, w_lane, x_lane);
  (tile_chunk<kB, J>(d, w_lane, x_lane, dec, cur), ...);
}

template <int kB>
__device__ __forceinline__ void tile_stage(float (&d)[2][4], uint32_t w_lane, uint32_t x_lane,
                                           const PairDecode& dec) {
  tile_stage_chunks<kB>(d, w_lane, x_lane, dec, std::make_integer_sequence<int, 8>{});
}

template <int kB>
__device__ __forceinline__ void store_out(const GemvArgs& a, int row, int n, float acc) {
  if (row >= a.K_out || n >= kB) return;
  float v = 2.0f * a.alpha[row] * acc;
  const size_t o = static_cast<size_t>(n) * a.K_out + row;
  if (a.y_bf16) {
    if (a.residual) v += __bfloat162float(static_cast<const __nv_bfloat16*>(a.residual)[o]);
    if (a.relu) v = fmaxf(v, 0.0f);
    static_cast<__nv_bfloat16*>(a.y)[o] = __float2bfloat16_rn(v);
  } else {
    if (a.residual) v += static_cast<const float*>(a.residual)[o];
    if (a.relu) v = fmaxf(v, 0.0f);
    static_cast<float*>(a.y)[o] = v;
  }
}

template <int kB>
__global__ void __launch_bounds__(kThreads, 1)
    gemv_tma_kernel(const __grid_constant__ CUtensorMap tmap_w,
                    const __grid_constant__ CUtensorMap tmap_x, const GemvArgs a) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ uint64_t full_bar[kMaxStages], empty_bar[kMaxStages];
  __shared__ float partial[kConsumerWarps][32][4];
  __shared__ volatile int abort_flag;

  // stage s at ring + s * stage_bytes; 1024-byte aligned for the swizzle
  const uint32_t raw = smem_addr(smem_raw);
  const uint32_t ring = (raw + 1023u) & ~1023u;
  uint8_t* ring_ptr = smem_raw + (ring - raw);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    abort_flag = 0;
    for (int s = 0; s < a.stages; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], static_cast<uint32_t>(a.n_t));   // one warp per tile per stage
    }
    fence_mbar_init();
  }
  __syncthreads();

  if (warp == kProducerWarp) {
    // ---------------------------------------------------------- producer
    const bool elected = elect_one();
    if (elected) {
      prefetch_tmap(&tmap_w);
      prefetch_tmap(&tmap_x);
    }
    // CTAs start their sweep over K at evenly spread offsets, so at any
    // moment the grid reads many different column ranges of the (row-pitch
    // strided) code matrix instead of one.  Consumers do not depend on the
    // order: a stage's data position only enters through these coordinates.
    const int k_start = static_cast<int>((static_cast<int64_t>(blockIdx.x) * a.nks) / gridDim.x);
    int it = 0;                      // stages issued so far
    int slot = 0;                    // it % stages
    uint32_t empty_parity = 1;       // parity of the release before use it / stages
    auto load_x = [&](int sl, int kc) {
      uint8_t* st = ring_ptr + static_cast<size_t>(sl) * a.stage_bytes;
      if (kB == 1) {
        // one batch row: the stage's inputs are 1 KB contiguous
        tma_load_2d(st + a.w_bytes, &tmap_x, &full_bar[sl], kc * kCodesPerStage, 0);
        tma_load_2d(st + a.w_bytes + 512, &tmap_x, &full_bar[sl], kc * kCodesPerStage + 256, 0);
      } else {
        tma_load_3d(st + a.w_bytes, &tmap_x, &full_bar[sl], 0, 0, kc * (kCodesPerStage / 8));
      }
    };
    // The first band's first stages: codes now, inputs after the wait.
    int deferred = 0;
    bool waited = false;
    auto finish_wait = [&]() {
      grid_dependency_wait();   // the inputs may come from the previous kernel
      grid_dependents_launch();
      if (elected)
        for (int i = 0; i < deferred; ++i) load_x(i, (k_start + i) % a.nks);
      __syncwarp();
      waited = true;
    };
    for (int r = 0; r < a.rounds; ++r) {
      const int band = blockIdx.x + r * gridDim.x;
      if (band * a.n_t >= a.T) break;
      int kc = k_start;
      for (int ks = 0; ks < a.nks; ++ks) {
        if (!waited && (r > 0 || it >= a.stages)) finish_wait();
        bool ok = true;
        if (it >= a.stages)
          ok = mbar_wait_sleep(&empty_bar[slot], empty_parity, &abort_flag, a.err, kWaitLimitNs);
        // one decision for the whole warp (lane 0's)
        if (!__shfl_sync(0xffffffffu, ok && !abort_flag, 0)) break;
        if (elected) {
          uint8_t* st = ring_ptr + static_cast<size_t>(slot) * a.stage_bytes;
          mbar_arrive_expect_tx(&full_bar[slot], a.stage_bytes);
          tma_load_2d(st, &tmap_w, &full_bar[slot], kc * kWordsPerStage, band * a.n_t * 16);
          if (waited) load_x(slot, kc);
        }
        if (!waited) ++deferred;
        __syncwarp();
        ++it;
        if (++kc == a.nks) kc = 0;
        if (++slot == a.stages) {
          slot = 0;
          empty_parity ^= 1u;
        }
      }
      if (__shfl_sync(0xffffffffu, abort_flag, 0)) break;
    }
    if (!waited) finish_wait();
    // On abort, wait (bounded) for the last copy issued into each slot so
    // no TMA write lands after the CTA has exited.
    if (elected && abort_flag) {
      for (int s = 0; s < a.stages && s < it; ++s) {
        const int last_use = (it - 1 - s) / a.stages;
        mbar_wait(&full_bar[s], static_cast<uint32_t>(last_use & 1), nullptr, a.err,
                  kWaitLimitNs);
      }
    }
    return;
  }

  // ------------------------------------------------------------ consumers
  grid_dependency_wait();   // the residual may come from the previous kernel
  const int g = lane >> 2, t = lane & 3;
  const PairDecode dec(t);
  // warp w works on tile w / P of the band, ring iterations i with
  // i % P == w % P (i = r * nks + ks for stage ks of round r)
  const int P = a.P;
  const int tau = warp / P, pi = warp % P;
  const bool active = tau < a.n_t;
  // per-lane shared-memory offsets inside a stage
  const uint32_t w_lane_off = static_cast<uint32_t>((tau * 16 + g) * 128 + (g << 4));
  const uint32_t x_lane_off =
      static_cast<uint32_t>(((lane >> 3) * kB + (lane & 7) % kB) * 16);

  for (int r = 0; r < a.rounds; ++r) {
    const int band = blockIdx.x + r * gridDim.x;
    if (band * a.n_t >= a.T) break;
    float c[2][4];
#pragma unroll
    for (int q = 0; q < 2; ++q)
#pragma unroll
      for (int i = 0; i < 4; ++i) c[q][i] = 0.0f;
    // this warp's first stage of the band and its ring slot / parity; the
    // slot then advances by P, which divides the ring depth
    const int band_it = r * a.nks;
    int ks = ((pi - band_it) % P + P) % P;
    int slot = (band_it + ks) % a.stages;
    uint32_t parity = static_cast<uint32_t>(((band_it + ks) / a.stages) & 1);
    for (; active && ks < a.nks; ks += P) {
      const bool ok_lane = mbar_wait_sleep(&full_bar[slot], parity, &abort_flag, a.err,
                                           kWaitLimitNs);
      // ldmatrix / mma need the whole warp: follow lane 0's outcome
      if (__shfl_sync(0xffffffffu, ok_lane, 0)) {
        const uint32_t st = ring + static_cast<uint32_t>(slot) * a.stage_bytes;
        tile_stage<kB>(c, st + w_lane_off, st + a.w_bytes + x_lane_off, dec);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty_bar[slot]);
      slot += P;   // slot % P == this warp's residue; wrap past the end
      if (slot >= a.stages) {
        slot -= a.stages;
        parity ^= 1u;
      }
    }
    float d[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) d[i] = c[0][i] + c[1][i];
    const int ra = band * a.n_t * 16 + tau * 16 + g;
    if (P == 1) {
      if (active && !abort_flag) {
        store_out<kB>(a, ra, 2 * t, d[0]);
        store_out<kB>(a, ra, 2 * t + 1, d[1]);
        store_out<kB>(a, ra + 8, 2 * t, d[2]);
        store_out<kB>(a, ra + 8, 2 * t + 1, d[3]);
      }
    } else {
      // fixed-order sum of the P partial tiles
#pragma unroll
      for (int i = 0; i < 4; ++i) partial[warp][lane][i] = d[i];
      named_barrier_sync(1, 32 * kConsumerWarps);
      if (active && pi == 0 && !abort_flag) {
        float sum[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          sum[i] = partial[warp][lane][i];
          for (int q = 1; q < P; ++q) sum[i] += partial[warp + q][lane][i];
        }
        store_out<kB>(a, ra, 2 * t, sum[0]);
        store_out<kB>(a, ra, 2 * t + 1, sum[1]);
        store_out<kB>(a, ra + 8, 2 * t, sum[2]);
        store_out<kB>(a, ra + 8, 2 * t + 1, sum[3]);
      }
      named_barrier_sync(1, 32 * kConsumerWarps);
    }
  }
}

struct GemvPlan {
  int T, n_t, rounds, grid, nks, P, stages;
  uint32_t w_bytes, stage_bytes;
  size_t smem;
};

GemvPlan plan_gemv(int64_t B, int64_t K_in, int64_t K_out, int sms) {
  GemvPlan p{};
  p.T = static_cast<int>((K_out + 15) / 16);
  p.rounds = (p.T + kMaxTilesPerBand * sms - 1) / (kMaxTilesPerBand * sms);
  p.n_t = (p.T + sms * p.rounds - 1) / (sms * p.rounds);
  p.grid = (p.T + p.n_t * p.rounds - 1) / (p.n_t * p.rounds);
  p.nks = static_cast<int>((K_in + kCodesPerStage - 1) / kCodesPerStage);
  p.P = kConsumerWarps / p.n_t;   // n_t <= 16
  if (p.P > p.nks) p.P = p.nks;
  p.w_bytes = static_cast<uint32_t>(p.n_t) * 16u * 128u;
  p.stage_bytes = p.w_bytes + static_cast<uint32_t>(B) * 1024u;
  p.stages = static_cast<int>(kSmemBudget / p.stage_bytes);
  if (p.stages > kMaxStages) p.stages = kMaxStages;
  p.stages -= p.stages % p.P;   // a multiple of P (see the consumer loop)
  p.smem = static_cast<size_t>(p.stages) * p.stage_bytes + 1024;
  return p;
}

}  // namespace

const char* gemv_unsupported_reason(const void* x, tbn_dtype xdt, int64_t B, int64_t K_in,
                                    const uint32_t* codes) {
  if (xdt != TBN_BF16) return "GEMV needs bf16 activations";
  if (B < 1 || B > 8) return "GEMV needs 1 <= B <= 8";
  if (K_in % 64 != 0) return "GEMV needs K_in % 64 == 0";
  if (K_in >= (1ll << 30)) return "GEMV: K_in too large";
  if (!is_aligned(x, 16) || !is_aligned(codes, 16)) return "GEMV needs 16-byte aligned x and codes";
  if (get_encode_tiled() == nullptr) return "cuTensorMapEncodeTiled unavailable";
  return "";
}

tbn_status launch_gemv(const void* x, int64_t B, int64_t K_in, const uint32_t* codes,
                       const float* alpha, int64_t K_out, void* y, tbn_dtype ydt, int relu,
                       const void* residual, cudaStream_t s) {
  if (K_out >= (1ll << 31) - 16) return fail(TBN_ERR_INVALID_ARG, "GEMV: K_out too large");
  const GemvPlan p = plan_gemv(B, K_in, K_out, device_sm_count());
  if (p.stages < 2 || p.stages < p.P)
    return fail(TBN_ERR_UNSUPPORTED, "GEMV: stage does not fit shared memory");

  alignas(64) CUtensorMap tmap_w, tmap_x;
  {
    const cuuint64_t gdim[2] = {static_cast<cuuint64_t>(K_in / 16), static_cast<cuuint64_t>(K_out)};
    const cuuint64_t gstride[1] = {static_cast<cuuint64_t>(K_in / 4)};
    const cuuint32_t box[2] = {kWordsPerStage, static_cast<cuuint32_t>(p.n_t * 16)};
    const cuuint32_t estr[2] = {1, 1};
    const CUresult cr = get_encode_tiled()(
        &tmap_w, CU_TENSOR_MAP_DATA_TYPE_UINT32, 2, const_cast<uint32_t*>(codes), gdim, gstride,
        box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (cr != CUDA_SUCCESS)
      return fail(TBN_ERR_CUDA, "cuTensorMapEncodeTiled(codes) failed (%d)", (int)cr);
  }
  if (B == 1) {
    const cuuint64_t gdim[2] = {static_cast<cuuint64_t>(K_in), 1};
    const cuuint64_t gstride[1] = {static_cast<cuuint64_t>(K_in * 2)};
    const cuuint32_t box[2] = {256, 1};
    const cuuint32_t estr[2] = {1, 1};
    const CUresult cr = get_encode_tiled()(
        &tmap_x, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(x), gdim, gstride, box,
        estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (cr != CUDA_SUCCESS)
      return fail(TBN_ERR_CUDA, "cuTensorMapEncodeTiled(x) failed (%d)", (int)cr);
  } else {
    // x [B][K_in] viewed as (8 elements, B rows, K_in / 8 chunks) so a box
    // lands in shared memory as [chunk][batch row][8 elements]
    const cuuint64_t gdim[3] = {8, static_cast<cuuint64_t>(B), static_cast<cuuint64_t>(K_in / 8)};
    const cuuint64_t gstride[2] = {static_cast<cuuint64_t>(K_in * 2), 16};
    const cuuint32_t box[3] = {8, static_cast<cuuint32_t>(B), kCodesPerStage / 8};
    const cuuint32_t estr[3] = {1, 1, 1};
    const CUresult cr = get_encode_tiled()(
        &tmap_x, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(x), gdim, gstride, box,
        estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
        CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (cr != CUDA_SUCCESS)
      return fail(TBN_ERR_CUDA, "cuTensorMapEncodeTiled(x) failed (%d)", (int)cr);
  }

  static std::once_flag attr_once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(attr_once, [] {
    const void* fns[8] = {(const void*)gemv_tma_kernel<1>, (const void*)gemv_tma_kernel<2>,
                          (const void*)gemv_tma_kernel<3>, (const void*)gemv_tma_kernel<4>,
                          (const void*)gemv_tma_kernel<5>, (const void*)gemv_tma_kernel<6>,
                          (const void*)gemv_tma_kernel<7>, (const void*)gemv_tma_kernel<8>};
    for (const void* f : fns) {
      const cudaError_t e =
          cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBudget + 1024);
      if (e != cudaSuccess && attr_err == cudaSuccess) attr_err = e;
    }
  });
  if (attr_err != cudaSuccess) return cuda_fail(attr_err, "cudaFuncSetAttribute(gemv)");

  GemvArgs a{};
  a.alpha = alpha;
  a.y = y;
  a.residual = residual;
  a.err = device_error_word();
  a.K_out = static_cast<int>(K_out);
  a.K_in = static_cast<int>(K_in);
  a.B = static_cast<int>(B);
  a.T = p.T;
  a.n_t = p.n_t;
  a.rounds = p.rounds;
  a.nks = p.nks;
  a.P = p.P;
  a.stages = p.stages;
  a.w_bytes = p.w_bytes;
  a.stage_bytes = p.stage_bytes;
  a.y_bf16 = ydt == TBN_BF16 ? 1 : 0;
  a.relu = relu;
  void (*kern)(CUtensorMap, CUtensorMap, GemvArgs) = nullptr;
  switch (B) {
    case 1: kern = gemv_tma_kernel<1>; break;
    case 2: kern = gemv_tma_kernel<2>; break;
    case 3: kern = gemv_tma_kernel<3>; break;
    case 4: kern = gemv_tma_kernel<4>; break;
    case 5: kern = gemv_tma_kernel<5>; break;
    case 6: kern = gemv_tma_kernel<6>; break;
    case 7: kern = gemv_tma_kernel<7>; break;
    default: kern = gemv_tma_kernel<8>; break;
  }
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
  const cudaError_t le = cudaLaunchKernelEx(&cfg, kern, tmap_w, tmap_x, a);
  if (le != cudaSuccess) return cuda_fail(le, "cudaLaunchKernelEx(gemv_tma_kernel)");
  return check_launch("gemv_tma_kernel");
}

}  // namespace tbn
