// tbn_conv_igemm.cuh -- the tcgen05 implicit-GEMM kernel of the two-bit
// convolution (Eq. 1, Section 2) and its launch, shared by the translation
// units that instantiate it (tbn_conv_igemm.cu: host dispatch and the
// gathering modes; tbn_conv_igemm_tma64.cu / _tma32.cu: the TMA modes with
// and without fused quantization), so that its variants compile in parallel.
//
//
// GEMM view of one tile:  D[128 filters x T pixels] = A[128 x n] * B[n x T]
// with T <= 256 output pixels and n = R*S*C in the codes' (r, s, c) order,
// 64 codes per K block (= pipeline stage: four MMAs of K = 16).
//
//   A (filters)     the 2-bit codes, decoded in registers to bf16 W~/2 in
//                   {+-0.5, +-1} (exact) and written straight into tensor
//                   memory (tcgen05.st) by eight "expander" warps: two per
//                   TMEM sub-partition, each decoding half of a K block's 64
//                   codes for the 32 filter rows (= TMEM lanes) it can reach,
//                   two K blocks per tcgen05.wait::st.  The decoded weights
//                   never touch shared memory, which is left to the
//                   activation operand.  Decoding costs integer-pipe issue
//                   slots per (filter, code), so a tile spans up to 256
//                   pixels to amortize it over as many MMA columns as the
//                   instruction allows.
//   B (activations) im2col rows per pixel, 128-byte rows (64 codes) with the
//                   128-byte swizzle.  When C % 64 == 0 a K block is one tap x
//                   64 channels and one TMA box load fetches it (the box is
//                   the tile's output pixels shifted by the tap; zero fill
//                   supplies the padding, element strides the conv stride).
//                   When C % 32 == 0 (e.g. 96 channels) a K block is two
//                   boxes of 32 channels, each from its own tap, into two
//                   64-byte-row halves of the stage with the 64-byte swizzle
//                   (a box past the filter's last code is loaded out of
//                   range and arrives zero-filled).  Otherwise gather warps
//                   assemble the rows from a per-K-block table of (tap,
//                   channel) offsets.
//   D               fp32 in tensor memory (256 columns).  Epilogue warps read
//                   lane = filter, column = pixel, multiply by 2 * alpha (Eq. 1
//                   applies alpha to the whole filter; the factor 2 undoes the
//                   W~/2 encoding -- exact scalings), add the optional
//                   residual, apply ReLU and the optional 2x2 max pool, round
//                   to bf16 into a shared-memory staging tile laid out as the
//                   NHWC output box, and one TMA bulk tensor store writes the
//                   box (clipped at the tensor's edges).  The accumulator is
//                   released as soon as it has been read, before the staging
//                   writes and the store complete.
//
// The kernel is persistent: each CTA walks tiles blockIdx.x, +gridDim.x, ...
// (filter tile fastest, so CTAs working at the same time share activation
// tiles in L2); producers and expanders run ahead into the next tile while
// the epilogue drains the accumulator.
//
// Warp roles (every role is a whole warp that waits on the barriers; where a
// single thread must issue -- TMA copies, MMAs, commits -- one elected lane
// does, with warp-uniform operands):
//   warps 0, 18.. TMA producers (TMA mode), taking K blocks in turn: one
//                 issuing thread delivers tiled boxes at a limited rate, so
//                 several keep the activation ring fuller
//   warp 1        TMEM allocator + MMA issuer
//   warps 2-9     expanders
//   warps 10-17   epilogue
//   warps 18-21   gather producers (gather mode only)
// Every wait is bounded (tbn_device.cuh); on a timeout the CTA records the
// error, drains its own in-flight copies and MMAs, frees TMEM and returns.
//
// The kernel is launched as a programmatic dependent of the previous kernel
// on the stream: its start-up (TMEM allocation, barrier set-up, loading and
// decoding the first blocks of codes) may overlap the previous kernel's last
// wave, and only the reads of activations and of the residual wait for that
// kernel to complete (grid_dependency_wait).  Codes and alpha are read
// before that wait, so they must not be written by the immediately
// preceding kernel when that kernel is one of this library's convolutions
// (which let their dependents start early); no convolution writes anything
// but its output.  Each CTA lets its own dependents start once it has passed
// its wait, so everything older than the previous kernel is complete by then.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>

#include <algorithm>
#include <cstdint>
#include <cstring>
#include <mutex>

#include "tbn_device.cuh"
#include "tbn_internal.h"
#include "tbn_quant_core.cuh"

namespace tbn {

// The kernel's arguments and tile plan (plain data; built on the host by
// launch_conv_igemm).
struct IgArgs {
  int N, C, H, W, K, R, S, sh, sw, ph, pw, P, Q;
  int bw, bh, bn;          // output pixels per tile along q, p, image
  int tile_n;              // MMA N: bw*bh*bn rounded up to 16
  int tiles_q, tiles_p, tiles_k, tiles;
  int kblocks;             // ceil(R*S*C / 64): pipeline stages per tile
  int ncodes;              // R*S*C
  int wpf;                 // words per filter
  const __nv_bfloat16* x;  // gather mode
  const uint32_t* codes;
  const float* alpha;
  void* y;
  const void* residual;
  int relu, y_bf16;
  uint32_t* err;
  // patch mode: the patch is rows [p0 sh - ph, + PR) x columns [-pw, W + pw)
  int PR, PW;              // patch rows, patch columns (W + 2 pw)
  int patch_cap;           // bytes per patch buffer (multiple of 16)
  int patch_bulk;          // pw == 0: in-image rows are one contiguous range of x
  long long x_bytes;       // size of x (bulk copies never read past it)
  // split K: tile t is K-block range `split` (t / base_tiles) of the output
  // tile t % base_tiles; the fp32 partial sums go to `partial`
  // [ksplit][N][P][Q][K] and a second kernel adds them in split order
  int ksplit, kb_per, base_tiles;
  // two accumulators (tile_n <= 176): tile i accumulates into columns
  // [176 (i % 2), + 176), so its MMAs need not wait for the epilogue of
  // tile i - 1; the weight ring then starts at column 352
  int acc2;
  float* partial;
  // space-to-depth mode: the convolution in original coordinates (stride
  // s2d_s, C0 channels, R0 x S0 filter, codes in (r, s, c) order)
  int s2d_s, s2d_C, s2d_R, s2d_S;
  // fused quantization (Algorithm 1's quantization loop in the same launch):
  // the CTAs first write codes and alpha from the fp32 filters wq
  // [K][ncodes], then meet at a grid-wide barrier (a cooperative launch)
  // before convolving; null wq: codes and alpha are inputs
  const float* wq;
  uint32_t* codes_w;       // = codes
  float* alpha_w;          // = alpha
  unsigned* gbar;          // barrier word, zero at launch
  int wq_vec;              // 16-byte loads of wq allowed
};

struct TilePlan {
  int bw, bh, bn, T, tile_n, tiles_q, tiles_p, tiles_n;
};

namespace {


constexpr int kBM = 128;            // filters per tile = TMEM lanes
constexpr int kBK = 64;             // codes per K block (128-byte rows)
constexpr int kMaxTileN = 256;      // pixels per tile (MMA N) upper bound
constexpr int kStages = 5;          // pipeline depth: activation ring (shared
                                    // memory) and weight ring (tensor memory)
constexpr int kAColsPerStage = kBK / 2;   // 64 bf16 = 32 columns of 32 bits
constexpr int kAccCols = kMaxTileN;       // the accumulator
constexpr int kAcc2Cols = 176;            // each of two accumulators (tiles of <= 176 pixels)
constexpr int kTmemCols = 512;      // accumulator [0,256) + weight ring [256,416)
constexpr int kExpWarps = 8;
constexpr int kEpiWarps = 8;
constexpr int kGatherWarps = 4;
constexpr int kPatchWarps = 8;      // patch mode: one operand row per thread
constexpr int kTmaProducers = 2;    // TMA mode: warp 0 and warps 18 .. 18 + kTmaProducers - 2
static_assert(kTmaProducers <= kStages, "a producer's parity wait needs kStages >= producers");
constexpr int kFirstExpWarp = 2;
constexpr int kFirstEpiWarp = kFirstExpWarp + kExpWarps;
constexpr int kFirstGatherWarp = kFirstEpiWarp + kEpiWarps;
constexpr int kStageBytes = kMaxTileN * kBK * 2;     // 32 KiB
constexpr int kOutStageBytes = kMaxTileN * kBM * 2;  // 64 KiB bf16 output box
constexpr uint64_t kWaitLimitNs = 1000000000ull;    // 1 s

static_assert(kAccCols + kStages * kAColsPerStage <= kTmemCols, "TMEM budget");
static_assert(2 * kAcc2Cols + kStages * kAColsPerStage <= kTmemCols, "TMEM budget");

// How the activation operand reaches the stage ring.
constexpr int kModeTma64 = 0;   // one 64-channel TMA box per K block (C % 64 == 0)
constexpr int kModeTma32 = 1;   // two 32-channel TMA boxes per K block (C % 32 == 0)
constexpr int kModeGather = 2;  // threads gather each code's activation from global memory
constexpr int kModePatch = 3;   // the tile's input rows are staged in shared memory (bulk
                                // copy, double-buffered) and threads build the rows from there
constexpr int kModeS2d = 4;     // space-to-depth input: 64-channel TMA boxes, and the
                                // filter's K blocks decoded once per CTA into tensor memory
constexpr int kMaxResidentKB = 15;   // resident K blocks: 32 columns each beside the accumulator

__host__ __device__ constexpr bool mode_gathers(int mode) {
  return mode == kModeGather || mode == kModePatch;
}
// the patch buffers take the room of two ring stages
__host__ __device__ constexpr int stages_for(int mode) { return mode == kModePatch ? kStages - 2 : kStages; }

// Producer warps of a mode (warps kFirstGatherWarp.. in the gathering modes).
__host__ __device__ constexpr int producer_warps(int mode) {
  return mode == kModePatch ? kPatchWarps : (mode == kModeGather ? kGatherWarps : 0);
}

template <int kMode>
constexpr int threads_for() {
  return 32 * (kFirstGatherWarp +
               (mode_gathers(kMode) ? producer_warps(kMode) : kTmaProducers - 1));
}


struct SmemCtl {
  // stage s holds K block g (g % kStages == s): its activations (shared
  // memory) and its decoded weights (tensor memory).  full: both operands
  // written; empty: the MMAs that read them have completed.
  uint64_t full[kStages];
  uint64_t empty[kStages];
  uint64_t acc_full[2];     // accumulator b holds a finished tile
  uint64_t acc_empty[2];    // accumulator b has been read by the epilogue
  uint64_t res_full;
  uint64_t mma_drain;      // used only to drain in-flight MMAs after an abort
  uint32_t tmem_base;
  int abort;
  int gtab_off[2][kBK];    // gather: element offset of each code of the K block
  int gtab_rs[2][kBK];     // gather: (r << 16 | s), or -1 beyond the filter
  uint64_t patch_full[2];  // patch mode: a buffer's bulk copy has landed
  uint64_t wready[kMaxResidentKB];   // space-to-depth mode: resident K block decoded
};

constexpr int kSmemLimit = 232448;
constexpr int kPatchMaxKBlocks = 16;   // patch mode keeps a table of every K block's codes

// Dynamic shared memory of a mode: ring, output staging, control block; in
// patch mode also two patch buffers and the code-offset table.
constexpr size_t smem_bytes_for(int mode, size_t patch_cap, int kblocks) {
  return 1024 /*align slack*/ + stages_for(mode) * kStageBytes + kOutStageBytes +
         ((sizeof(SmemCtl) + 15) / 16) * 16 +
         (mode == kModePatch ? 2 * patch_cap + static_cast<size_t>(kblocks) * kBK * 4 : 0);
}
static_assert(smem_bytes_for(kModeTma64, 0, 0) <= kSmemLimit, "shared memory budget");


__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint4 v) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(v.x), "r"(v.y),
               "r"(v.z), "r"(v.w)
               : "memory");
}

// 16-bit shared-memory store by 32-bit shared address.
__device__ __forceinline__ void st_shared_u16(uint32_t addr, uint32_t v) {
  asm volatile("st.shared.u16 [%0], %1;" ::"r"(addr), "h"(static_cast<uint16_t>(v)) : "memory");
}

struct TileCoord {
  int ktile, q0, p0, n0;
  int split, kb0, kb1;   // K blocks [kb0, kb1) of the filter (split K)
};

__device__ __forceinline__ TileCoord tile_coord(const IgArgs& a, int t) {
  TileCoord c;
  c.split = t / a.base_tiles;
  t -= c.split * a.base_tiles;
  c.kb0 = c.split * a.kb_per;
  c.kb1 = min(a.kblocks, c.kb0 + a.kb_per);
  c.ktile = t % a.tiles_k;
  const int pt_lin = t / a.tiles_k;
  const int qt = pt_lin % a.tiles_q;
  const int pt = (pt_lin / a.tiles_q) % a.tiles_p;
  const int nt = pt_lin / (a.tiles_q * a.tiles_p);
  c.q0 = qt * a.bw;
  c.p0 = pt * a.bh;
  c.n0 = nt * a.bn;
  return c;
}

// Direct global store of one output value (the path for fp32 output or
// shapes the TMA store cannot take): fp32 math, residual, ReLU, rounding.
__device__ __forceinline__ void store_out(const IgArgs& a, size_t o, float v) {
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

// kPoolBW: 0 = no pool; 8, 16, 32 = fused 2x2/2 max pool for tiles of whole
// output rows of that width.  kTmaStore: bf16 output through the staging
// tile and TMA stores (else direct global stores).
// Fused quantization prologue: CTA b quantizes filters [b K / G, (b + 1) K / G)
// exactly as the quantize kernel does (the same per-word fields and sums,
// reduced per filter in the same order: bitwise the same codes and alpha),
// with `scratch` (the stage ring, not yet in use) holding a chunk of rows'
// per-word sums and counts; then all CTAs meet at a grid-wide barrier on
// a.gbar (bounded: on expiry the device error word records a timeout and
// the CTA's abort flag is set, so it does no convolution work).
__device__ void quantize_prologue(const IgArgs& a, uint8_t* scratch, int scratch_words,
                                  volatile int* abort_flag) {
  // every thread has read the abort flag before anyone can set it below
  __syncthreads();
  const int G = gridDim.x, b = blockIdx.x, nth = blockDim.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r0 = static_cast<int>(static_cast<int64_t>(b) * a.K / G);
  const int r1 = static_cast<int>(static_cast<int64_t>(b + 1) * a.K / G);
  const int wpf = a.wpf, n = a.ncodes;
  float* ssum = reinterpret_cast<float*>(scratch);
  int* scnt = reinterpret_cast<int*>(scratch + static_cast<size_t>(scratch_words) * 4);
  const int rows_per_chunk = max(1, scratch_words / wpf);
  for (int c0 = r0; c0 < r1; c0 += rows_per_chunk) {
    const int c1 = min(r1, c0 + rows_per_chunk);
    const int words = (c1 - c0) * wpf;
    // two words per thread per pass: eight 16-byte loads in flight
    for (int i0 = threadIdx.x; i0 < words; i0 += 2 * nth) {
      float v[2][16];
      int nv[2];
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const int i = i0 + u * nth;
        nv[u] = 0;
        if (i < words) {
          const int r = i / wpf, j = i - r * wpf;
          load16(a.wq + static_cast<int64_t>(c0 + r) * n, n, j, a.wq_vec != 0, v[u], nv[u]);
        }
      }
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const int i = i0 + u * nth;
        if (i < words) {
          const int r = i / wpf, j = i - r * wpf;
          uint32_t word;
          float sum;
          int c2;
          encode16(v[u], nv[u], word, sum, c2);
          a.codes_w[static_cast<int64_t>(c0 + r) * wpf + j] = word;
          ssum[i] = sum;
          scnt[i] = c2;
        }
      }
    }
    __syncthreads();
    // per filter, as the quantize kernel reduces: words in order by one
    // thread (at most 16 words), else lane-strided and a warp butterfly
    if (wpf <= 16) {
      for (int r = threadIdx.x; r < c1 - c0; r += nth) {
        Sum2 acc{0.0f, 0.0f};
        int cnt2 = 0;
        bool huge = false;
        for (int c = 0; c < wpf; ++c) {
          const float sv = ssum[r * wpf + c];
          huge |= !finite_sum(sv);
          add2(acc, sv);
          cnt2 += scnt[r * wpf + c];
        }
        a.alpha_w[c0 + r] = huge ? alpha_fp64_row(a.wq + static_cast<int64_t>(c0 + r) * n, n)
                                 : alpha_of(acc, cnt2, n);
      }
    } else {
      for (int r = warp; r < c1 - c0; r += nth / 32) {
        Sum2 acc{0.0f, 0.0f};
        int cnt2 = 0;
        bool huge = false;
        for (int c = lane; c < wpf; c += 32) {
          const float sv = ssum[r * wpf + c];
          huge |= !finite_sum(sv);
          add2(acc, sv);
          cnt2 += scnt[r * wpf + c];
        }
        acc = warp_sum2(acc);
        cnt2 = warp_sum(cnt2);
        huge = __any_sync(0xffffffffu, huge);
        if (lane == 0)
          a.alpha_w[c0 + r] = huge ? alpha_fp64_row(a.wq + static_cast<int64_t>(c0 + r) * n, n)
                                   : alpha_of(acc, cnt2, n);
      }
    }
    __syncthreads();
  }
  // grid-wide barrier: every CTA's codes and alpha are written.  A barrier
  // that runs out of time sets the CTA's abort flag (no static shared
  // memory here: the dynamic allocation takes all that the SM offers).
  if (threadIdx.x == 0) {
    __threadfence();
    atomicAdd(a.gbar, 1u);
    const uint64_t t0 = global_timer_ns();
    int ok = 1;
    while (*reinterpret_cast<volatile unsigned*>(a.gbar) < static_cast<unsigned>(G)) {
      if (global_timer_ns() - t0 > kWaitLimitNs) {
        raise_device_error(a.err, TBN_DEVERR_TIMEOUT);
        ok = 0;
        break;
      }
      __nanosleep(64);
    }
    __threadfence();
    if (!ok) *abort_flag = 1;
  }
  fence_proxy_async_smem();   // the scratch is the ring: TMA writes come after these stores
  __syncthreads();
}

// kMode: how activations reach the ring (kModeTma64 / kModeTma32 /
// kModeGather / kModePatch).
template <int kMode, int kPoolBW, bool kTmaStore, bool kFuse>
__global__ void __launch_bounds__(threads_for<kMode>(), 1)
    conv_igemm_kernel(const __grid_constant__ CUtensorMap tmap_x,
                      const __grid_constant__ CUtensorMap tmap_y,
                      const __grid_constant__ CUtensorMap tmap_res,
                      const __grid_constant__ IgArgs a) {
  constexpr bool kGather = mode_gathers(kMode);
  constexpr bool kCh32 = kMode == kModeTma32;
  constexpr bool kPatch = kMode == kModePatch;
  constexpr bool kS2d = kMode == kModeS2d;
  constexpr int kSt = stages_for(kMode);   // ring stages
  extern __shared__ uint8_t smem_raw[];
  // 1024-byte aligned by pointer arithmetic on the shared array, so that the
  // compiler keeps every access derived from it in the shared state space
  uint8_t* smem = smem_raw + ((1024u - (smem_addr(smem_raw) & 1023u)) & 1023u);
  uint8_t* ring = smem;                                   // kSt x 32 KiB
  uint8_t* out_stage = smem + kSt * kStageBytes;          // 64 KiB
  SmemCtl* ctl = reinterpret_cast<SmemCtl*>(out_stage + kOutStageBytes);
  // patch mode: two patch buffers, then the code-offset table
  uint8_t* patch_buf = reinterpret_cast<uint8_t*>(ctl) + ((sizeof(SmemCtl) + 15) / 16) * 16;
  volatile int* abort_flag = &ctl->abort;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int KB = a.kblocks;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kSt; ++i) {
      // space-to-depth mode: the weights are resident, only the activation box fills a stage
      mbar_init(&ctl->full[i], (kS2d ? 0 : 32 * kExpWarps) +
                                   (kGather ? 32 * producer_warps(kMode) : 1));
      mbar_init(&ctl->empty[i], 1);
    }
    mbar_init(&ctl->patch_full[0], 1);
    mbar_init(&ctl->patch_full[1], 1);
    for (int b = 0; b < 2; ++b) {
      mbar_init(&ctl->acc_full[b], 1);
      mbar_init(&ctl->acc_empty[b], 32 * kEpiWarps);
    }
    mbar_init(&ctl->res_full, 1);
    mbar_init(&ctl->mma_drain, 1);
    if (kS2d)
      for (int i = 0; i < KB && i < kMaxResidentKB; ++i) mbar_init(&ctl->wready[i], 32 * kExpWarps);
    ctl->abort = 0;
    fence_mbar_init();
    if (!kGather) prefetch_tmap(&tmap_x);
    if (kTmaStore) prefetch_tmap(&tmap_y);
  }
  if (warp == 1) {
    tmem_alloc(&ctl->tmem_base, kTmemCols);
    tmem_relinquish();
  }
  if (kS2d) {
    // gather table of the resident K blocks: column j of K block kb (tap
    // (kb / S', kb % S') of the space-to-depth grid, channel j = (dy s + dx)
    // C0 + c) holds original code l = ((s r' + dy) S0 + s s' + dx) C0 + c as
    // (l / 16) | (its magnitude bit) << 16, or ~0 where the s x s block
    // reaches past the filter.  It lives in the output staging tile, which
    // the epilogue first writes after the first tile's MMAs, i.e. after the
    // decode.
    uint32_t* tab = reinterpret_cast<uint32_t*>(out_stage);
    const int ss = a.s2d_s, C0 = a.s2d_C;
    for (int e = threadIdx.x; e < KB * kBK; e += blockDim.x) {
      const int kb = e / kBK, j = e - (e / kBK) * kBK;
      uint32_t v = 0xFFFFFFFFu;
      if (j < ss * ss * C0) {
        const int dy = j / (ss * C0), dx = (j / C0) % ss, c = j % C0;
        const int r = ss * (kb / a.S) + dy, q = ss * (kb % a.S) + dx;
        if (r < a.s2d_R && q < a.s2d_S) {
          const int l = (r * a.s2d_S + q) * C0 + c;
          v = static_cast<uint32_t>(l >> 4) | (static_cast<uint32_t>(code_mag_bit(l & 15)) << 16);
        }
      }
      tab[e] = v;
    }
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  // The CTA allocates all 512 columns, so the allocation can only start at
  // lane 0, column 0: every tensor-memory address below is a compile-time
  // constant.  Any other base is reported and the CTA does no work.
  constexpr uint32_t tmem = 0;
  if (ctl->tmem_base != 0u) {
    if (threadIdx.x == 0) {
      raise_device_error(a.err, TBN_DEVERR_BAD_LAUNCH);
      ctl->abort = 1;
    }
  }
  __syncthreads();
  if constexpr (kFuse) {
    if (!*abort_flag)   // uniform: every thread read the flag after the barrier
      quantize_prologue(a, ring, (kSt * kStageBytes) / 8, abort_flag);
  }
  if (*abort_flag) {
    if (warp == 1) tmem_dealloc(ctl->tmem_base, kTmemCols);
    return;
  }
  const uint32_t acc_tmem = tmem;               // columns [0, 256), or two of 176
  const uint32_t a_tmem0 = tmem + (a.acc2 ? 2u * kAcc2Cols : static_cast<uint32_t>(kAccCols));   // weight ring

  if (!kGather && (warp == 0 || warp >= kFirstGatherWarp)) {
    // ================= TMA producers =================
    grid_dependency_wait();   // activations may come from the previous kernel
    grid_dependents_launch();
    // producer pid issues the K blocks g with g % kTmaProducers == pid; the
    // ring has at least as many stages as producers, so the release a
    // producer waits for always follows the previous release of that slot
    // (the MMA warp releases in order) and its parity wait cannot alias
    const int pid = warp == 0 ? 0 : warp - kFirstGatherWarp + 1;
    int turn = 0;   // g % kTmaProducers
    constexpr int kBoxCh = kCh32 ? kBK / 2 : kBK;   // channels per box
    constexpr int kBoxes = kBK / kBoxCh;             // boxes per K block
    const uint32_t box_bytes = static_cast<uint32_t>(a.bw * a.bh * a.bn * kBoxCh * 2);
    const int cblocks = a.C / kBoxCh;                // boxes per tap
    int g = 0;  // global K-block counter of this CTA
    bool ok = true;
    for (int t = blockIdx.x; t < a.tiles && ok; t += gridDim.x) {
      const TileCoord tc = tile_coord(a, t);
      // (tap, channel box) of the next box
      int tap = (tc.kb0 * kBoxes) / cblocks, cb = (tc.kb0 * kBoxes) % cblocks;
      for (int kb = tc.kb0; kb < tc.kb1; ++kb, ++g) {
        const bool mine = turn == pid;
        if (++turn == kTmaProducers) turn = 0;
        if (!mine) {
#pragma unroll
          for (int bx = 0; bx < kBoxes; ++bx)
            if (++cb == cblocks) { cb = 0; ++tap; }
          continue;
        }
        const int sb = g % kSt;
        const uint32_t it = static_cast<uint32_t>(g / kSt);
        ok = mbar_wait(&ctl->empty[sb], (it & 1u) ^ 1u, abort_flag, a.err, kWaitLimitNs);
        if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
        if (elect_one()) {
          mbar_arrive_expect_tx(&ctl->full[sb], box_bytes * kBoxes);
#pragma unroll
          for (int bx = 0; bx < kBoxes; ++bx) {
            // a box past the filter's last tap is requested at channel C:
            // entirely out of range, it arrives zero-filled
            const bool past = tap >= a.R * a.S;
            const int tp = past ? 0 : tap;
            const int r = tp / a.S, s = tp - r * a.S;
            tma_load_4d(ring + sb * kStageBytes + bx * (kStageBytes / kBoxes), &tmap_x,
                        &ctl->full[sb], past ? a.C : cb * kBoxCh, tc.q0 * a.sw - a.pw + s,
                        tc.p0 * a.sh - a.ph + r, tc.n0);
            if (++cb == cblocks) { cb = 0; ++tap; }
          }
        } else {
#pragma unroll
          for (int bx = 0; bx < kBoxes; ++bx)
            if (++cb == cblocks) { cb = 0; ++tap; }
        }
        __syncwarp();
      }
    }
    // drain: every copy this warp issued must land before the CTA may exit
    for (int i = g > kSt ? g - kSt : 0; i < g; ++i)
      if (i % kTmaProducers == pid)
        mbar_wait(&ctl->full[i % kSt], static_cast<uint32_t>(i / kSt) & 1u, nullptr,
                  a.err, kWaitLimitNs);
  } else if (kMode == kModeGather && warp >= kFirstGatherWarp) {
    // ================= gather producers =================
    // The gather warps meet at a named barrier every K block, so none of them
    // may leave the loops early: after a failed wait a warp keeps walking the
    // loop structure (reaching every barrier) but does no more work.
    const int gt = threadIdx.x - 32 * kFirstGatherWarp;   // 0..127
    const bool vec = (a.C & 7) == 0;
    grid_dependency_wait();   // activations may come from the previous kernel
    grid_dependents_launch();
    int g = 0;
    bool ok = true;
    for (int t = blockIdx.x; t < a.tiles; t += gridDim.x) {
      const TileCoord tc = tile_coord(a, t);
      const int T = a.bw * a.bh * a.bn;
      // this thread fills tile rows gt and gt + 128; offset of tap (0, 0)
      int64_t pbase[2];
      int rh[2], rw[2];
      bool rv[2];
#pragma unroll
      for (int i = 0; i < 2; ++i) {
        const int row = gt + 128 * i;
        const int wi = row % a.bw, hi = (row / a.bw) % a.bh, ni = row / (a.bw * a.bh);
        rh[i] = (tc.p0 + hi) * a.sh - a.ph;
        rw[i] = (tc.q0 + wi) * a.sw - a.pw;
        rv[i] = row < T && tc.n0 + ni < a.N && tc.p0 + hi < a.P && tc.q0 + wi < a.Q;
        pbase[i] = ((static_cast<int64_t>(rv[i] ? tc.n0 + ni : 0) * a.H + rh[i]) * a.W + rw[i]) *
                   static_cast<int64_t>(a.C);
      }
      for (int kb = tc.kb0; kb < tc.kb1; ++kb, ++g) {
        // table of this K block's 64 codes: offset from the tap-(0,0) pixel
        const int tb = g & 1;
        if (gt < kBK) {
          const int k = kb * kBK + gt;
          if (k < a.ncodes) {
            const int c = k % a.C, tap = k / a.C;
            const int r = tap / a.S, s = tap - r * a.S;
            ctl->gtab_off[tb][gt] = (r * a.W + s) * a.C + c;
            ctl->gtab_rs[tb][gt] = (r << 16) | s;
          } else {
            ctl->gtab_off[tb][gt] = 0;
            ctl->gtab_rs[tb][gt] = -1;
          }
        }
        named_barrier_sync(2, 32 * kGatherWarps);
        const int sb = g % kSt;
        const uint32_t it = static_cast<uint32_t>(g / kSt);
        if (ok) ok = mbar_wait(&ctl->empty[sb], (it & 1u) ^ 1u, abort_flag, a.err, kWaitLimitNs);
        ok = __all_sync(0xffffffffu, ok);
        if (!ok) continue;
#pragma unroll
        for (int i = 0; i < 2; ++i) {
          const int row = gt + 128 * i;
          if (row >= a.tile_n) continue;
          const uint32_t row_addr = smem_addr(ring + sb * kStageBytes) + static_cast<uint32_t>(row) * 128u;
          uint4 v[8];
          if (vec) {
#pragma unroll
            for (int ch = 0; ch < 8; ++ch) {
              const int rs = ctl->gtab_rs[tb][ch * 8];
              const int h = rh[i] + (rs >> 16), w = rw[i] + (rs & 0xFFFF);
              v[ch] = make_uint4(0u, 0u, 0u, 0u);
              if (rv[i] && rs >= 0 && h >= 0 && h < a.H && w >= 0 && w < a.W)
                v[ch] = __ldg(reinterpret_cast<const uint4*>(a.x + pbase[i] + ctl->gtab_off[tb][ch * 8]));
            }
          } else {
            const unsigned short* xs = reinterpret_cast<const unsigned short*>(a.x);
#pragma unroll
            for (int ch = 0; ch < 8; ++ch) {
              uint32_t e[8];
#pragma unroll
              for (int q = 0; q < 8; ++q) {
                const int rs = ctl->gtab_rs[tb][ch * 8 + q];
                const int h = rh[i] + (rs >> 16), w = rw[i] + (rs & 0xFFFF);
                e[q] = 0u;
                if (rv[i] && rs >= 0 && h >= 0 && h < a.H && w >= 0 && w < a.W)
                  e[q] = __ldg(xs + pbase[i] + ctl->gtab_off[tb][ch * 8 + q]);
              }
              v[ch] = make_uint4(e[0] | (e[1] << 16), e[2] | (e[3] << 16), e[4] | (e[5] << 16),
                                 e[6] | (e[7] << 16));
            }
          }
#pragma unroll
          for (int ch = 0; ch < 8; ++ch)  // 128-byte swizzle: chunk XOR (row mod 8)
            st_shared_v4(row_addr + static_cast<uint32_t>(((ch ^ (row & 7)) & 7) * 16), v[ch]);
        }
        fence_proxy_async_smem();   // generic-proxy writes -> visible to tcgen05.mma
        mbar_arrive(&ctl->full[sb]);
      }
    }
  } else if (kPatch && warp >= kFirstGatherWarp) {
    // ================= patch producers =================
    // Tiles are whole output rows of one image (bn = 1, tiles_q = 1).  The
    // input rows a tile reads, [p0 sh - ph, + PR) x [-pw, W + pw) x C, are
    // staged in a shared-memory patch (zero outside the image); each K block
    // row is then built from the patch with one 32-bit load per pair of codes
    // when the pair is contiguous there, two 16-bit loads otherwise.  With no
    // column padding the in-image rows are one contiguous range of x and one
    // bulk copy (issued a tile ahead, into the other buffer) fetches them.
    const int gt = threadIdx.x - 32 * kFirstGatherWarp;   // 0..255
    const int pitch = a.PW * a.C;                          // patch row, elements
    const int patch_elems = a.PR * pitch;
    const int* ptab = reinterpret_cast<const int*>(patch_buf + 2 * a.patch_cap);
    int* ptab_w = reinterpret_cast<int*>(patch_buf + 2 * a.patch_cap);
    const uint8_t* xb = reinterpret_cast<const uint8_t*>(a.x);
    // offset table of every K block: patch element of code k relative to the
    // pixel's (tap 0, channel 0) element, -1 past the filter
    for (int i = gt; i < KB * kBK; i += 32 * kPatchWarps) {
      const int k = i;
      int off = -1;
      if (k < a.ncodes) {
        const int c = k % a.C, tap = k / a.C;
        const int r = tap / a.S, s = tap - r * a.S;
        off = (r * a.PW + s) * a.C + c;
      }
      asm volatile("st.shared.s32 [%0], %1;" ::"r"(smem_addr(ptab_w + i)), "r"(off) : "memory");
    }
    grid_dependency_wait();   // activations may come from the previous kernel
    grid_dependents_launch();
    named_barrier_sync(2, 32 * kPatchWarps);

    // geometry of tile t's patch: in-image patch rows [lo, hi), the byte
    // offset `src` in x of its first in-image element, and the byte offset of
    // patch element 0 in its buffer (chosen so that the bulk copy's
    // destination is 16-byte aligned)
    auto geom = [&](int t, int& lo, int& hi, long long& src, uint32_t& off0) {
      const TileCoord tc = tile_coord(a, t);
      const int h0 = tc.p0 * a.sh - a.ph;
      lo = max(0, -h0);
      hi = min(a.PR, a.H - h0);
      if (hi < lo) hi = lo;
      const long long e0 = static_cast<long long>(lo) * pitch;
      src = ((static_cast<long long>(tc.n0) * a.H + h0 + lo) * a.W) * a.C * 2;
      off0 = static_cast<uint32_t>(((src & 15) - 2 * e0) & 15);
    };
    // one thread: the bulk copy of tile t's in-image rows into buffer b
    auto issue = [&](int t, int b) {
      int lo, hi;
      long long src;
      uint32_t off0;
      geom(t, lo, hi, src, off0);
      const long long len = static_cast<long long>(hi - lo) * pitch * 2;
      const long long a0 = src & ~15LL;
      long long a1 = (src + len + 15) & ~15LL;
      if (a1 > a.x_bytes) a1 = a.x_bytes & ~15LL;   // the rest is copied by threads
      const uint32_t bytes = a1 > a0 ? static_cast<uint32_t>(a1 - a0) : 0u;
      uint8_t* dst = patch_buf + b * a.patch_cap + off0 + 2 * static_cast<long long>(lo) * pitch -
                     (src & 15);
      fence_proxy_async_smem();   // earlier generic accesses of the buffer come first
      mbar_arrive_expect_tx(&ctl->patch_full[b], bytes);
      if (bytes) bulk_load_1d(dst, xb + a0, bytes, &ctl->patch_full[b]);
    };

    int g = 0;
    bool ok = true;
    uint32_t issued[2] = {0u, 0u};   // bulk copies issued into each buffer (thread 0)
    uint32_t landed[2] = {0u, 0u};   // copies this thread has seen complete
    uint32_t tiles_done = 0;
    if (a.patch_bulk && gt == 0 && static_cast<int>(blockIdx.x) < a.tiles) {
      issue(blockIdx.x, 0);
      ++issued[0];
    }
    __syncwarp();   // reconverge before the aligned named barriers below
    const int T = a.bw * a.bh;
    for (int t = blockIdx.x; t < a.tiles; t += gridDim.x, ++tiles_done) {
      const TileCoord tc = tile_coord(a, t);
      const int b = tiles_done & 1;
      uint8_t* buf = patch_buf + b * a.patch_cap;
      int lo, hi;
      long long src;
      uint32_t off0;
      geom(t, lo, hi, src, off0);
      const uint32_t buf_s = smem_addr(buf);
      const uint32_t pe_s = buf_s + off0;   // patch element e at pe_s + 2 e
      // everyone has finished building the previous tile (the buffer filled
      // next was last read two tiles ago)
      named_barrier_sync(2, 32 * kPatchWarps);
      if (a.patch_bulk) {
        if (gt == 0 && ok && t + static_cast<int>(gridDim.x) < a.tiles) {
          issue(t + gridDim.x, b ^ 1);
          ++issued[b ^ 1];
        }
        if (ok) {
          ok = mbar_wait(&ctl->patch_full[b], landed[b] & 1u, abort_flag, a.err, kWaitLimitNs);
          if (ok) ++landed[b];
        }
        ok = __all_sync(0xffffffffu, ok);
        // rows outside the image are zero; the copy's rounding may have
        // written neighbouring bytes there
        for (int e = gt; e < lo * pitch; e += 32 * kPatchWarps) st_shared_u16(pe_s + 2 * e, 0u);
        for (int e = hi * pitch + gt; e < patch_elems; e += 32 * kPatchWarps)
          st_shared_u16(pe_s + 2 * e, 0u);
        // the last bytes of x that no 16-byte chunk of the copy covered
        const long long len = static_cast<long long>(hi - lo) * pitch * 2;
        const long long cov = a.x_bytes & ~15LL;
        if (src + len > cov) {
          const long long first = max(src, cov);
          for (long long bpos = first + 2 * gt; bpos < src + len; bpos += 2 * 32 * kPatchWarps)
            st_shared_u16(pe_s + 2 * static_cast<uint32_t>(lo * pitch + (bpos - src) / 2),
                          *reinterpret_cast<const uint16_t*>(xb + bpos));
        }
      } else {
        // column padding: element by element, zero outside the image
        const TileCoord tc = tile_coord(a, t);
        const int h0 = tc.p0 * a.sh - a.ph;
        const uint16_t* xs = reinterpret_cast<const uint16_t*>(a.x);
        for (int e = gt; e < patch_elems; e += 32 * kPatchWarps) {
          const int rho = e / pitch, rem = e - rho * pitch;
          const int u = rem / a.C, c = rem - u * a.C;
          const int h = h0 + rho, w = u - a.pw;
          uint16_t v = 0;
          if (h >= 0 && h < a.H && w >= 0 && w < a.W)
            v = __ldg(xs + ((static_cast<long long>(tc.n0) * a.H + h) * a.W + w) * a.C + c);
          st_shared_u16(pe_s + 2 * e, v);
        }
      }
      named_barrier_sync(2, 32 * kPatchWarps);   // patch complete
      // this thread's rows: pixel (i, q) of the tile reads from patch element
      // i sh pitch + q sw C on; base in 16-bit units from the buffer start
      constexpr int kRows = kMaxTileN / (32 * kPatchWarps);   // operand rows per thread
      int base[kRows];
      bool valid[kRows];
#pragma unroll
      for (int j = 0; j < kRows; ++j) {
        const int px = gt + 32 * kPatchWarps * j;
        const int i = px / a.bw, q = px - i * a.bw;
        valid[j] = px < T;
        base[j] = static_cast<int>(off0 / 2) + i * a.sh * pitch + q * a.sw * a.C;
      }
      for (int kb = tc.kb0; kb < tc.kb1; ++kb, ++g) {
        const int sb = g % kSt;
        const uint32_t it = static_cast<uint32_t>(g / kSt);
        if (ok) ok = mbar_wait(&ctl->empty[sb], (it & 1u) ^ 1u, abort_flag, a.err, kWaitLimitNs);
        ok = __all_sync(0xffffffffu, ok);
        if (!ok) continue;
        const int* __restrict__ tab = ptab + kb * kBK;
        uint8_t* __restrict__ stage = ring + sb * kStageBytes;
        const uint16_t* __restrict__ p16 = reinterpret_cast<const uint16_t*>(buf);
        const uint32_t* __restrict__ p32 = reinterpret_cast<const uint32_t*>(buf);
#pragma unroll
        for (int j = 0; j < kRows; ++j) {
          const int row = gt + 32 * kPatchWarps * j;
          if (row >= a.tile_n) continue;
          // four chunks at a time: every load of the group is issued before
          // the first shift or store
#pragma unroll
          for (int cg = 0; cg < 2; ++cg) {
            int4 o[8];
#pragma unroll
            for (int c = 0; c < 4; ++c) {
              o[2 * c] = *reinterpret_cast<const int4*>(tab + 8 * (4 * cg + c));
              o[2 * c + 1] = *reinterpret_cast<const int4*>(tab + 8 * (4 * cg + c) + 4);
            }
            uint32_t wv[4][5];
            bool run[4];
#pragma unroll
            for (int c = 0; c < 4; ++c) {
              // the chunk's 8 codes are 8 consecutive patch elements (one run
              // of a filter row): 5 aligned words, 4 funnel shifts
              run[c] = valid[j] && o[2 * c].x >= 0 && o[2 * c + 1].w == o[2 * c].x + 7;
              const int e = base[j] + (o[2 * c].x >= 0 ? o[2 * c].x : 0);
              const uint32_t* w = p32 + (e >> 1);
#pragma unroll
              for (int u = 0; u < 5; ++u) wv[c][u] = run[c] ? w[u] : 0u;
            }
#pragma unroll
            for (int c = 0; c < 4; ++c) {
              const int ch = 4 * cg + c;
              uint4 v = make_uint4(0u, 0u, 0u, 0u);
              if (run[c]) {
                const int e = base[j] + o[2 * c].x;
                const uint32_t sh = static_cast<uint32_t>(e & 1) * 16u;
                v.x = __funnelshift_r(wv[c][0], wv[c][1], sh);
                v.y = __funnelshift_r(wv[c][1], wv[c][2], sh);
                v.z = __funnelshift_r(wv[c][2], wv[c][3], sh);
                v.w = __funnelshift_r(wv[c][3], wv[c][4], sh);
              } else if (valid[j]) {
                // a chunk across two filter rows, or past the filter's end
                const int off[8] = {o[2 * c].x, o[2 * c].y, o[2 * c].z, o[2 * c].w,
                                    o[2 * c + 1].x, o[2 * c + 1].y, o[2 * c + 1].z,
                                    o[2 * c + 1].w};
                uint32_t h[8];
#pragma unroll
                for (int u = 0; u < 8; ++u)
                  h[u] = off[u] >= 0 ? static_cast<uint32_t>(p16[base[j] + off[u]]) : 0u;
                v = make_uint4(h[0] | (h[1] << 16), h[2] | (h[3] << 16), h[4] | (h[5] << 16),
                               h[6] | (h[7] << 16));
              }
              // 128-byte swizzle: chunk XOR (row mod 8)
              *reinterpret_cast<uint4*>(stage + row * 128 + (((ch ^ (row & 7)) & 7) << 4)) = v;
            }
          }
        }
        fence_proxy_async_smem();   // generic-proxy writes -> visible to tcgen05.mma
        mbar_arrive(&ctl->full[sb]);
      }
    }
    // drain (after an abort): every bulk copy issued must land before the
    // CTA may exit
    if (a.patch_bulk && gt == 0) {
      for (int b = 0; b < 2; ++b)
        while (landed[b] < issued[b] &&
               mbar_wait(&ctl->patch_full[b], landed[b] & 1u, nullptr, a.err, kWaitLimitNs))
          ++landed[b];
    }
    __syncwarp();
  } else if (warp == 1) {
    // ================= MMA issuer =================
    const uint32_t idesc = idesc_bf16_f32(kBM, static_cast<uint32_t>(a.tile_n));
    int g = 0, issued = 0;
    uint32_t tiles_done = 0;
    bool ok = true;
    for (int t = blockIdx.x; t < a.tiles && ok; t += gridDim.x, ++tiles_done) {
      const TileCoord tc = tile_coord(a, t);
      // the epilogue must have drained this accumulator's previous tile
      const uint32_t ab = a.acc2 ? (tiles_done & 1u) : 0u;
      const uint32_t use = a.acc2 ? (tiles_done >> 1) : tiles_done;   // uses of accumulator ab
      const uint32_t acc_t = acc_tmem + ab * kAcc2Cols;
      ok = mbar_wait(&ctl->acc_empty[ab], (use & 1u) ^ 1u, abort_flag, a.err, kWaitLimitNs);
      if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
      tc_fence_after_sync();
      for (int kb = tc.kb0; kb < tc.kb1; ++kb, ++g) {
        const int st = g % kSt;
        ok = mbar_wait(&ctl->full[st], static_cast<uint32_t>(g / kSt) & 1u, abort_flag, a.err,
                       kWaitLimitNs);
        if (kS2d && tiles_done == 0 && ok)   // first use of a resident K block
          ok = mbar_wait(&ctl->wready[kb], 0u, abort_flag, a.err, kWaitLimitNs);
        if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
        tc_fence_after_sync();
        const uint32_t a_col =
            kS2d ? static_cast<uint32_t>(kTmemCols - 32 * KB + 32 * kb)
                 : a_tmem0 + static_cast<uint32_t>(st * kAColsPerStage);
        if (elect_one()) {
          if constexpr (kCh32) {
            // two halves of 32 codes, 64-byte rows with the 64-byte swizzle
#pragma unroll
            for (int kk = 0; kk < kBK / 16; ++kk) {
              const uint64_t bdesc = smem_desc_sw64_kmajor(
                  smem_addr(ring + st * kStageBytes + (kk >> 1) * (kStageBytes / 2)));
              tc_mma_ts(acc_t, a_col + 8u * kk, bdesc + static_cast<uint64_t>(2 * (kk & 1)),
                        idesc, ((kb - tc.kb0) | kk) != 0 ? 1u : 0u);
            }
          } else {
            const uint64_t bdesc = smem_desc_sw128_kmajor(smem_addr(ring + st * kStageBytes));
#pragma unroll
            for (int kk = 0; kk < kBK / 16; ++kk) {
              // K step kk: 16 codes = 8 TMEM columns of A, 32 bytes of B rows
              tc_mma_ts(acc_t, a_col + 8u * kk, bdesc + static_cast<uint64_t>(2 * kk), idesc,
                        ((kb - tc.kb0) | kk) != 0 ? 1u : 0u);
            }
          }
          tc_commit(&ctl->empty[st]);
        }
        __syncwarp();
        ++issued;
      }
      if (ok) {
        if (elect_one()) tc_commit(&ctl->acc_full[ab]);
        __syncwarp();
      }
    }
    if (!ok && issued > 0) {
      // drain in-flight MMAs before TMEM is freed
      if (elect_one()) tc_commit(&ctl->mma_drain);
      __syncwarp();
      mbar_wait(&ctl->mma_drain, 0u, nullptr, a.err, kWaitLimitNs);
    }
  } else if (warp >= kFirstExpWarp && warp < kFirstExpWarp + kExpWarps) {
    // ================= expanders =================
    const int sub = warp & 3;                         // TMEM sub-partition
    const int half = (warp - kFirstExpWarp) >> 2;     // which 32 codes of a K block
    const int m = sub * 32 + lane;                    // filter row within the tile
    const uint32_t lane_off = static_cast<uint32_t>(sub * 32) << 16;
    if constexpr (kS2d) {
      // Decode every K block of the filter once into its resident columns
      // [512 - 32 KB + 32 kb, + 32) (this warp: codes [32 half, + 32) of
      // each, i.e. 16 columns).  Filter rows past K hold zeros.
      const uint32_t* tab = reinterpret_cast<const uint32_t*>(out_stage);
      const uint32_t* crow = m < a.K ? a.codes + static_cast<size_t>(m) * a.wpf : nullptr;
      const uint32_t res0 = static_cast<uint32_t>(kTmemCols - 32 * KB);
      for (int kb = 0; kb < KB; ++kb) {
        uint32_t v[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const uint32_t e0 = tab[kb * kBK + 32 * half + 2 * i];
          const uint32_t e1 = tab[kb * kBK + 32 * half + 2 * i + 1];
          uint32_t lo = 0u, hi = 0u;
          // W~/2 in bf16: 0x3F00 (0.5) | m << 7 (1.0) | s << 15
          if (crow != nullptr && e0 != 0xFFFFFFFFu)
            lo = ((__ldg(crow + (e0 & 0xFFFFu)) >> (e0 >> 16)) & 0x101u) * 128u + 0x3F00u;
          if (crow != nullptr && e1 != 0xFFFFFFFFu)
            hi = ((__ldg(crow + (e1 & 0xFFFFu)) >> (e1 >> 16)) & 0x101u) * 128u + 0x3F00u;
          v[i] = lo | (hi << 16);
        }
        tmem_st_32x32b_x16(tmem + lane_off + res0 + static_cast<uint32_t>(32 * kb + 16 * half), v);
        tmem_wait_st();
        tc_fence_before_sync();
        mbar_arrive(&ctl->wready[kb]);
      }
    } else {
    const bool pair_ok = ((a.wpf & 1) == 0) && ((reinterpret_cast<uintptr_t>(a.codes) & 7) == 0);
    // this CTA's K blocks, all tiles in sequence (g = tile_index * KB + kb)
    int total = 0;   // K blocks of all this CTA's tiles
    for (int t = blockIdx.x; t < a.tiles; t += gridDim.x) {
      const TileCoord tc = tile_coord(a, t);
      total += tc.kb1 - tc.kb0;
    }
    // prefetch cursor over (tile, kb): the codes of K block kb of a filter
    // are words [4 kb, 4 kb + 4) of its row; this warp takes two of them
    int t_ld = blockIdx.x, kb_ld = 0, kb_end = 0;
    const uint32_t* crow_ld = nullptr;
    auto set_row = [&]() {
      const TileCoord tc = tile_coord(a, t_ld < a.tiles ? t_ld : 0);
      kb_ld = tc.kb0;
      kb_end = tc.kb1;
      const int k = tc.ktile * kBM + m;
      crow_ld = (t_ld < a.tiles && k < a.K) ? a.codes + static_cast<size_t>(k) * a.wpf : nullptr;
    };
    set_row();
    auto next_codes = [&]() -> uint2 {
      uint2 r = make_uint2(0u, 0u);
      const int w0 = kb_ld * 4 + half * 2;
      if (crow_ld != nullptr && w0 < a.wpf) {
        // written by this launch's prologue when fused: ordinary (L1-cached,
        // coherent) loads after the grid barrier's acquire then, not the
        // read-only path, which assumes data constant for the whole launch
        if constexpr (kFuse) {
          if (pair_ok) r = __ldca(reinterpret_cast<const uint2*>(crow_ld + w0));
          else r = make_uint2(__ldca(crow_ld + w0), w0 + 1 < a.wpf ? __ldca(crow_ld + w0 + 1) : 0u);
        } else {
          if (pair_ok) r = __ldg(reinterpret_cast<const uint2*>(crow_ld + w0));
          else r = make_uint2(__ldg(crow_ld + w0), w0 + 1 < a.wpf ? __ldg(crow_ld + w0 + 1) : 0u);
        }
      }
      if (++kb_ld == kb_end) {
        t_ld += gridDim.x;
        set_row();
      }
      return r;
    };
    const PairMultipliers pm;
    uint2 q0 = next_codes(), q1 = next_codes(), q2 = next_codes(), q3 = next_codes();
    const uint32_t col = a_tmem0 + lane_off + static_cast<uint32_t>(16 * half);
    // two K blocks per iteration: their tensor-memory stores share one
    // tcgen05.wait::st
    for (int g = 0; g < total; g += 2) {
      const bool two = g + 1 < total;   // warp-uniform
      uint32_t v0[16], v1[16];
      word_to_bf16x2(q0.x, v0 + 0, pm);
      word_to_bf16x2(q0.y, v0 + 8, pm);
      word_to_bf16x2(q1.x, v1 + 0, pm);
      word_to_bf16x2(q1.y, v1 + 8, pm);
      q0 = q2;
      q1 = q3;
      q2 = next_codes();
      q3 = next_codes();
      const int s0 = g % kSt, s1 = (g + 1) % kSt;
      // in patch mode the operand builders are the bottleneck: waiting
      // expanders park instead of spinning, leaving the issue slots to them
      bool ok = kPatch ? mbar_wait_sleep(&ctl->empty[s0], (static_cast<uint32_t>(g / kSt) & 1u) ^ 1u,
                                         abort_flag, a.err, kWaitLimitNs)
                       : mbar_wait(&ctl->empty[s0], (static_cast<uint32_t>(g / kSt) & 1u) ^ 1u,
                                   abort_flag, a.err, kWaitLimitNs);
      if (ok && two)
        ok = kPatch ? mbar_wait_sleep(&ctl->empty[s1],
                                      (static_cast<uint32_t>((g + 1) / kSt) & 1u) ^ 1u, abort_flag,
                                      a.err, kWaitLimitNs)
                    : mbar_wait(&ctl->empty[s1], (static_cast<uint32_t>((g + 1) / kSt) & 1u) ^ 1u,
                                abort_flag, a.err, kWaitLimitNs);
      if (!__all_sync(0xffffffffu, ok)) break;
      tc_fence_after_sync();
      tmem_st_32x32b_x16(col + static_cast<uint32_t>(s0 * kAColsPerStage), v0);
      if (two) tmem_st_32x32b_x16(col + static_cast<uint32_t>(s1 * kAColsPerStage), v1);
      tmem_wait_st();
      tc_fence_before_sync();
      mbar_arrive(&ctl->full[s0]);
      if (two) mbar_arrive(&ctl->full[s1]);
    }
    }
  } else if (warp >= kFirstEpiWarp && warp < kFirstEpiWarp + kEpiWarps) {
    // ================= epilogue =================
    // Two warps per TMEM sub-partition, each reading half of the columns.
    const int sub = warp & 3;
    const int half = (warp - kFirstEpiWarp) >> 2;
    const int m = sub * 32 + lane;
    const int et = threadIdx.x - 32 * kFirstEpiWarp;   // 0..255
    const bool elected = et == 0;
    const uint32_t lane_off = static_cast<uint32_t>(sub * 32) << 16;
    const int Po = kPoolBW ? a.P / 2 : a.P;
    const int Qo = kPoolBW ? a.Q / 2 : a.Q;
    const uint32_t res_bytes = static_cast<uint32_t>(a.bw * a.bh * a.bn * kBM * 2);
    __nv_bfloat16* stage = reinterpret_cast<__nv_bfloat16*>(out_stage);
    grid_dependency_wait();   // the residual may come from the previous kernel
    uint32_t tiles_done = 0;
    bool ok = true;
    // The epilogue warps meet at named barriers, so after a failed wait they
    // keep walking the tile loop (reaching every barrier) without working.
    for (int t = blockIdx.x; t < a.tiles; t += gridDim.x, ++tiles_done) {
      const TileCoord tc = tile_coord(a, t);
      const uint32_t par = tiles_done & 1u;   // the residual box
      const uint32_t ab = a.acc2 ? (tiles_done & 1u) : 0u;
      const uint32_t apar = (a.acc2 ? (tiles_done >> 1) : tiles_done) & 1u;
      const uint32_t acc_b = acc_tmem + ab * kAcc2Cols;
      const uint32_t acc = acc_b + lane_off;
      const int k = tc.ktile * kBM + m;
      const bool kvalid = k < a.K;
      const float a2 = kvalid ? 2.0f * (kFuse ? __ldca(a.alpha + k) : __ldg(a.alpha + k)) : 0.0f;
      if (kTmaStore) {
        // the previous tile's store must have finished reading the staging tile
        if (elected) bulk_wait_group_read<0>();
        named_barrier_sync(1, 32 * kEpiWarps);
        if (ok && a.residual && elected) {
          mbar_arrive_expect_tx(&ctl->res_full, res_bytes);
          asm volatile(
              "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
              " [%0], [%1, {%3, %4, %5, %6}], [%2];" ::"r"(smem_addr(stage)),
              "l"(&tmap_res), "r"(smem_addr(&ctl->res_full)), "r"(tc.ktile * kBM),
              "r"(tc.q0), "r"(tc.p0), "r"(tc.n0)
              : "memory");
        }
      }
      if (ok)
        ok = kPatch ? mbar_wait_sleep(&ctl->acc_full[ab], apar, abort_flag, a.err, kWaitLimitNs)
                    : mbar_wait(&ctl->acc_full[ab], apar, abort_flag, a.err, kWaitLimitNs);
      if (kTmaStore && a.residual && ok)
        ok = mbar_wait(&ctl->res_full, par, abort_flag, a.err, kWaitLimitNs);
      ok = __all_sync(0xffffffffu, ok);
      if (ok) tc_fence_after_sync();
      if (!ok) {
        // skip the work, keep the barrier schedule
      } else if (kPoolBW == 0 && kTmaStore && a.residual == nullptr) {
        // Fragment epilogue: 16x256b loads (lane = filter, column = pixel),
        // scale / ReLU / bf16 pairs, transposed 8x8 stores into the staging
        // tile [pixel][filter] as two 128-byte-swizzled halves of 64
        // filters (chunk c of pixel row px at c ^ (px & 7)).
        const int nchunks = (a.tile_n + 31) / 32;
        const int c_begin = half ? (nchunks + 1) / 2 : 0;
        const int c_end = half ? nchunks : (nchunks + 1) / 2;
        const int fr = lane >> 2;                       // fragment row within 8
        float a2f[2][2];
#pragma unroll
        for (int lg = 0; lg < 2; ++lg) {
#pragma unroll
          for (int u = 0; u < 2; ++u) {
            const int kk = tc.ktile * kBM + sub * 32 + lg * 16 + u * 8 + fr;
            a2f[lg][u] = kk < a.K ? 2.0f * (kFuse ? __ldca(a.alpha + kk) : __ldg(a.alpha + kk)) : 0.0f;
          }
        }
        // this lane's stmatrix row address pieces: matrix mi = lane / 8, row = lane % 8
        const int mi = lane >> 3, mrow = lane & 7;
        const uint32_t stage_s = smem_addr(stage);
        for (int j = c_begin; j < c_end; ++j) {
          uint32_t v[2][16];
#pragma unroll
          for (int lg = 0; lg < 2; ++lg)
            tmem_ld_16x256b_x4(acc_b + (static_cast<uint32_t>(sub * 32 + lg * 16) << 16) +
                                   static_cast<uint32_t>(32 * j),
                               v[lg]);
          tmem_wait_ld();
          if (j == c_end - 1) {
            tc_fence_before_sync();
            mbar_arrive(&ctl->acc_empty[ab]);
          }
#pragma unroll
          for (int lg = 0; lg < 2; ++lg) {
            uint32_t pk[8];
#pragma unroll
            for (int b = 0; b < 4; ++b) {
              float y0 = a2f[lg][0] * __uint_as_float(v[lg][4 * b + 0]);
              float y1 = a2f[lg][0] * __uint_as_float(v[lg][4 * b + 1]);
              float y2 = a2f[lg][1] * __uint_as_float(v[lg][4 * b + 2]);
              float y3 = a2f[lg][1] * __uint_as_float(v[lg][4 * b + 3]);
              if (a.relu) {
                y0 = fmaxf(y0, 0.0f);
                y1 = fmaxf(y1, 0.0f);
                y2 = fmaxf(y2, 0.0f);
                y3 = fmaxf(y3, 0.0f);
              }
              pk[2 * b] = pack_bf16x2(y0, y1);       // filters fr, pixels 2(i%4) + 0/1
              pk[2 * b + 1] = pack_bf16x2(y2, y3);   // filters fr + 8
            }
#pragma unroll
            for (int bp = 0; bp < 2; ++bp) {
              // matrices: (filters +0, block 2bp), (+8, 2bp), (+0, 2bp+1), (+8, 2bp+1)
              const int px = 32 * j + 8 * (2 * bp + (mi >> 1)) + mrow;
              const int chunk = 4 * sub + 2 * lg + (mi & 1);           // 8-filter chunk 0..15
              const uint32_t addr = stage_s + static_cast<uint32_t>((chunk >> 3) * 32768 + px * 128 +
                                                                    (((chunk & 7) ^ (px & 7)) << 4));
              stmatrix_x4_trans(addr, pk[4 * bp + 0], pk[4 * bp + 1], pk[4 * bp + 2],
                                pk[4 * bp + 3]);
            }
          }
        }
        if (c_begin >= c_end) {
          tc_fence_before_sync();
          mbar_arrive(&ctl->acc_empty[ab]);
        }
      } else if constexpr (kPoolBW == 0) {
        const int T = a.bw * a.bh * a.bn;
        const int nchunks = (a.tile_n + 31) / 32;
        const int c_begin = half ? (nchunks + 1) / 2 : 0;
        const int c_end = half ? nchunks : (nchunks + 1) / 2;
        // direct-store path: pixel of chunk c_begin walked in column order
        int px0 = 32 * c_begin;
        int wi = px0 % a.bw, hi = (px0 / a.bw) % a.bh, ni = px0 / (a.bw * a.bh);
        for (int j = c_begin; j < c_end; ++j) {
          uint32_t v[32];
          tmem_ld_32x32b_x32(acc + static_cast<uint32_t>(32 * j), v);
          tmem_wait_ld();
          if (j == c_end - 1) {
            // this warp has read its part of the accumulator
            tc_fence_before_sync();
            mbar_arrive(&ctl->acc_empty[ab]);
          }
          if (!kTmaStore && a.partial != nullptr) {
            // split K (1x1 image): pixel px is image n0 + px; the raw sum of
            // this K range goes to partial[split][n][k]
            float* dst = a.partial + (static_cast<size_t>(tc.split) * a.N + tc.n0 + 32 * j) * a.K + k;
#pragma unroll
            for (int i = 0; i < 32; ++i)
              if (kvalid && 32 * j + i < T && tc.n0 + 32 * j + i < a.N)
                dst[static_cast<size_t>(i) * a.K] = __uint_as_float(v[i]);
          } else if (kTmaStore) {
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const int px = 32 * j + i;
              if (px < T) {
                float y = a2 * __uint_as_float(v[i]);
                __nv_bfloat16* sp = stage + px * kBM + m;
                if (a.residual) y += __bfloat162float(*sp);
                if (a.relu) y = fmaxf(y, 0.0f);
                *sp = __float2bfloat16_rn(y);
              }
            }
          } else {
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const int px = 32 * j + i;
              const int q = tc.q0 + wi, p = tc.p0 + hi, n = tc.n0 + ni;
              if (kvalid && px < T && q < a.Q && p < a.P && n < a.N)
                store_out(a, ((static_cast<size_t>(n) * a.P + p) * a.Q + q) * a.K + k,
                          a2 * __uint_as_float(v[i]));
              if (++wi == a.bw) {
                wi = 0;
                if (++hi == a.bh) { hi = 0; ++ni; }
              }
            }
          }
        }
        if (c_begin >= c_end) {
          tc_fence_before_sync();
          mbar_arrive(&ctl->acc_empty[ab]);
        }
      } else {
        // fused 2x2 max pool: tiles hold whole rows of width kPoolBW (q0 = 0)
        // and an even number of rows per image; one TMEM load covers an even
        // pair of rows or more.
        constexpr int kCols = kPoolBW <= 16 ? 32 : 64;   // columns per load
        constexpr int kPairs = kCols / (2 * kPoolBW);    // row pairs per load
        const int rows_total = a.bh * a.bn;               // tile rows (all images)
        const int bh2 = a.bh / 2;
        const int nloads = (rows_total * kPoolBW + kCols - 1) / kCols;
        const int l_begin = half ? (nloads + 1) / 2 : 0;
        const int l_end = half ? nloads : (nloads + 1) / 2;
        for (int j = l_begin; j < l_end; ++j) {
          uint32_t v[kCols];
          tmem_ld_32x32b_x32(acc + static_cast<uint32_t>(kCols * j),
                             *reinterpret_cast<uint32_t(*)[32]>(v));
          if constexpr (kCols == 64)
            tmem_ld_32x32b_x32(acc + static_cast<uint32_t>(kCols * j + 32),
                               *reinterpret_cast<uint32_t(*)[32]>(v + 32));
          tmem_wait_ld();
          if (j == l_end - 1) {
            tc_fence_before_sync();
            mbar_arrive(&ctl->acc_empty[ab]);
          }
#pragma unroll
          for (int pp = 0; pp < kPairs; ++pp) {
            const int pair = j * kPairs + pp;          // row pair within the tile
            const int ni = pair / bh2;
            const int hi2 = pair - ni * bh2;
            const int p2 = tc.p0 / 2 + hi2, n = tc.n0 + ni;
            const bool pv = ni < a.bn;
#pragma unroll
            for (int q2 = 0; q2 < kPoolBW / 2; ++q2) {
              const int c0 = pp * 2 * kPoolBW + 2 * q2;
              const float m0 = fmaxf(__uint_as_float(v[c0]), __uint_as_float(v[c0 + 1]));
              const float m1 = fmaxf(__uint_as_float(v[c0 + kPoolBW]),
                                     __uint_as_float(v[c0 + kPoolBW + 1]));
              // alpha >= 0, so max commutes with the scaling (and with ReLU)
              float mx = a2 * fmaxf(m0, m1);
              if (kTmaStore) {
                if (pv) {
                  if (a.relu) mx = fmaxf(mx, 0.0f);
                  stage[(pair * (kPoolBW / 2) + q2) * kBM + m] = __float2bfloat16_rn(mx);
                }
              } else if (kvalid && pv && p2 < Po && q2 < Qo && n < a.N) {
                store_out(a, ((static_cast<size_t>(n) * Po + p2) * Qo + q2) * a.K + k, mx);
              }
            }
          }
        }
        if (l_begin >= l_end) {
          tc_fence_before_sync();
          mbar_arrive(&ctl->acc_empty[ab]);
        }
      }
      if (kTmaStore) {
        fence_proxy_async_smem();   // staged values -> visible to the TMA store
        named_barrier_sync(1, 32 * kEpiWarps);
        if (elected && ok) {
          if (kPoolBW) {
            tma_store_4d(&tmap_y, stage, tc.ktile * kBM, 0, tc.p0 / 2, tc.n0);
          } else if (a.residual == nullptr) {
            tma_store_4d(&tmap_y, stage, tc.ktile * kBM, tc.q0, tc.p0, tc.n0);
            if (tc.ktile * kBM + kBM / 2 < a.K)
              tma_store_4d(&tmap_y, reinterpret_cast<uint8_t*>(stage) + 32768,
                           tc.ktile * kBM + kBM / 2, tc.q0, tc.p0, tc.n0);
          } else {
            tma_store_4d(&tmap_y, stage, tc.ktile * kBM, tc.q0, tc.p0, tc.n0);
          }
          bulk_commit_group();
        }
      }
    }
    if (kTmaStore && elected) bulk_wait_group<0>();   // all stores complete before exit
  }

  tc_fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after_sync();
    tmem_dealloc(tmem, kTmemCols);
  }
}


// ---------------------------------------------------------------- host side

inline int ceil_div(int64_t a, int64_t b) { return static_cast<int>((a + b - 1) / b); }

// TMA activations: whole 64-channel boxes, or 32-channel boxes in pairs.
inline bool use_tma(const ConvProblem& p) { return p.C % (kBK / 2) == 0 && p.sh <= 2 && p.sw <= 2; }
inline bool use_ch32(const ConvProblem& p) { return p.C % kBK != 0; }

// Output pixels per tile: whole rows of the output (so one TMA box per tap
// covers the tile), balanced so the last tile along each axis is not a
// sliver, at most 256 pixels.  With a fused 2x2 pool a tile holds whole
// output rows and an even number of them per image.
inline TilePlan plan_tiles(const ConvProblem& p) {
  TilePlan t{};
  const int stride_w = use_tma(p) ? static_cast<int>(p.sw) : 1;
  const int stride_h = use_tma(p) ? static_cast<int>(p.sh) : 1;
  const int bw_max = static_cast<int>(std::min<int64_t>(p.Q, kMaxTileN / stride_w));
  t.tiles_q = ceil_div(p.Q, bw_max);
  t.bw = ceil_div(p.Q, t.tiles_q);
  if (t.tiles_q > 1) {
    t.bh = 1;
    t.bn = 1;
  } else {
    int bh_max = static_cast<int>(std::min<int64_t>({p.P, kMaxTileN / t.bw, 256 / stride_h}));
    if (p.pool) bh_max &= ~1;
    if (bh_max < 1) bh_max = 1;
    const int tp = ceil_div(p.P, bh_max);
    t.bh = ceil_div(p.P, tp);
    if (p.pool && (t.bh & 1)) t.bh += 1;   // <= bh_max when bh_max is even
    if (t.bh < p.P) {
      t.bn = 1;
    } else {
      t.bh = static_cast<int>(p.P) + (p.pool ? static_cast<int>(p.P & 1) : 0);
      const int bn_max = std::max(1, static_cast<int>(std::min<int64_t>(p.N, kMaxTileN / (t.bw * t.bh))));
      t.bn = ceil_div(p.N, ceil_div(p.N, bn_max));
    }
  }
  t.tiles_p = ceil_div(p.P, t.bh);
  t.tiles_n = ceil_div(p.N, t.bn);
  t.T = t.bw * t.bh * t.bn;
  t.tile_n = ((t.T + 15) / 16) * 16;
  return t;
}

inline int pool_width(const ConvProblem& p, const TilePlan& t) {
  if (!p.pool) return 0;
  if (t.tiles_q != 1 || t.T > kMaxTileN || (t.bh & 1)) return -1;
  if (t.bw == 8 || t.bw == 16 || t.bw == 32) return t.bw;
  return -1;
}

inline bool use_tma_store(const ConvProblem& p) {
  return p.ydt == TBN_BF16 && p.K % 8 == 0 && is_aligned(p.y, 16) &&
         (!p.residual || is_aligned(p.residual, 16));
}

// Output map: box = 128 filters x the tile's pixels (no swizzle), or with
// `halves`, 64 filters (128 bytes) per box with the 128-byte swizzle (the
// staging layout of the fragment epilogue, two stores per tile).
inline CUresult encode_out_map(CUtensorMap* m, const void* base, const ConvProblem& p, const TilePlan& t,
                        int pool, bool halves = false) {
  const int64_t Po = pool ? p.P / 2 : p.P, Qo = pool ? p.Q / 2 : p.Q;
  const cuuint64_t gdim[4] = {(cuuint64_t)p.K, (cuuint64_t)Qo, (cuuint64_t)Po, (cuuint64_t)p.N};
  const cuuint64_t gstride[3] = {(cuuint64_t)(p.K * 2), (cuuint64_t)(Qo * p.K * 2),
                                 (cuuint64_t)(Po * Qo * p.K * 2)};
  const cuuint32_t box[4] = {(cuuint32_t)(halves ? kBM / 2 : kBM), (cuuint32_t)(pool ? t.bw / 2 : t.bw),
                             (cuuint32_t)(pool ? t.bh / 2 : t.bh), (cuuint32_t)t.bn};
  const cuuint32_t estr[4] = {1u, 1u, 1u, 1u};
  return get_encode_tiled()(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), gdim,
                            gstride, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                            halves ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
                            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

template <int kMode, int kPoolBW, bool kTmaStore, bool kFuse>
tbn_status launch_t(const ConvProblem& p, const TilePlan& t, IgArgs& a, cudaStream_t s) {
  constexpr bool kGather = mode_gathers(kMode);
  constexpr bool kCh32 = kMode == kModeTma32;
  alignas(64) CUtensorMap tmap_x, tmap_y, tmap_res;
  std::memset(&tmap_x, 0, sizeof(tmap_x));
  std::memset(&tmap_y, 0, sizeof(tmap_y));
  std::memset(&tmap_res, 0, sizeof(tmap_res));
  if (!kGather) {
    const cuuint64_t gdim[4] = {(cuuint64_t)p.C, (cuuint64_t)p.W, (cuuint64_t)p.H, (cuuint64_t)p.N};
    const cuuint64_t gstride[3] = {(cuuint64_t)(p.C * 2), (cuuint64_t)(p.W * p.C * 2),
                                   (cuuint64_t)(p.H * p.W * p.C * 2)};
    const cuuint32_t box[4] = {(cuuint32_t)(kCh32 ? kBK / 2 : kBK), (cuuint32_t)(t.bw * p.sw),
                               (cuuint32_t)(t.bh * p.sh), (cuuint32_t)t.bn};
    const cuuint32_t estr[4] = {1u, (cuuint32_t)p.sw, (cuuint32_t)p.sh, 1u};
    if (box[1] > 256 || box[2] > 256 || box[3] > 256)
      return fail(TBN_ERR_UNSUPPORTED, "implicit GEMM: TMA box too large");
    const CUresult cr = get_encode_tiled()(&tmap_x, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4,
                                           const_cast<void*>(p.x), gdim, gstride, box, estr,
                                           CU_TENSOR_MAP_INTERLEAVE_NONE,
                                           kCh32 ? CU_TENSOR_MAP_SWIZZLE_64B
                                                 : CU_TENSOR_MAP_SWIZZLE_128B,
                                           CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                                           CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (cr != CUDA_SUCCESS) return fail(TBN_ERR_CUDA, "cuTensorMapEncodeTiled(x) failed (%d)", (int)cr);
  }
  if (kTmaStore) {
    // the fragment epilogue (no pool, no residual) stages two swizzled halves
    const bool halves = kPoolBW == 0 && p.residual == nullptr;
    CUresult cr = encode_out_map(&tmap_y, p.y, p, t, kPoolBW ? 1 : 0, halves);
    if (cr != CUDA_SUCCESS) return fail(TBN_ERR_CUDA, "cuTensorMapEncodeTiled(y) failed (%d)", (int)cr);
    if (p.residual) {
      cr = encode_out_map(&tmap_res, p.residual, p, t, 0);
      if (cr != CUDA_SUCCESS)
        return fail(TBN_ERR_CUDA, "cuTensorMapEncodeTiled(residual) failed (%d)", (int)cr);
    }
  }
  auto kern = conv_igemm_kernel<kMode, kPoolBW, kTmaStore, kFuse>;
  const size_t smem = smem_bytes_for(kMode, static_cast<size_t>(a.patch_cap), a.kblocks);
  // kernel attributes: set once per process (one process drives one GPU);
  // the shared-memory limit is the largest any launch of the mode can need
  static std::once_flag once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(once, [&] {
    attr_err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    kSmemLimit);
    if (attr_err == cudaSuccess)
      attr_err = cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
  });
  if (attr_err != cudaSuccess) return cuda_fail(attr_err, "cudaFuncSetAttribute(conv_igemm_kernel)");
  // fused quantization: one CTA per SM whatever the tile count, so that the
  // whole GPU quantizes (CTAs without a tile stop after the barrier)
  const int grid = kFuse ? device_sm_count() : std::min(a.tiles, device_sm_count());
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(static_cast<unsigned>(grid));
  cfg.blockDim = dim3(threads_for<kMode>());
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  if (kFuse) {
    // fused quantization: the CTAs meet at a grid-wide barrier, so they must
    // all be resident at once
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
  } else {
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
  }
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (kFuse) {
    const cudaError_t me = cudaMemsetAsync(a.gbar, 0, sizeof(unsigned), s);
    if (me != cudaSuccess) return cuda_fail(me, "cudaMemsetAsync(barrier word)");
  }
  const cudaError_t le = cudaLaunchKernelEx(&cfg, kern, tmap_x, tmap_y, tmap_res, a);
  if (le != cudaSuccess) return cuda_fail(le, "cudaLaunchKernelEx(conv_igemm_kernel)");
  return check_launch("conv_igemm_kernel");
}

template <int kMode, bool kTmaStore, bool kFuse>
tbn_status launch_pool(const ConvProblem& p, const TilePlan& t, IgArgs& a, int pw, cudaStream_t s) {
  switch (pw) {
    case 8: return launch_t<kMode, 8, kTmaStore, kFuse>(p, t, a, s);
    case 16: return launch_t<kMode, 16, kTmaStore, kFuse>(p, t, a, s);
    case 32: return launch_t<kMode, 32, kTmaStore, kFuse>(p, t, a, s);
    default: return launch_t<kMode, 0, kTmaStore, kFuse>(p, t, a, s);
  }
}

}  // namespace

// The per-mode launchers: pw = the fused pool's tile width (0: none),
// tma_store = the TMA-store epilogue, fuse = quantize the fp32 filters
// a.wq in the same (cooperative) launch.
tbn_status launch_igemm_tma64(const ConvProblem& p, const TilePlan& t, IgArgs& a, int pw,
                              bool tma_store, bool fuse, cudaStream_t s);
tbn_status launch_igemm_tma32(const ConvProblem& p, const TilePlan& t, IgArgs& a, int pw,
                              bool tma_store, bool fuse, cudaStream_t s);

}  // namespace tbn
