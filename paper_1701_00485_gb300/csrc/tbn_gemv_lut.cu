// tbn_gemv_lut.cu -- batch-1 two-bit fully-connected layer with fp32
// activations, by table lookup (Section 3: a fully-connected layer is a
// convolution whose filters span the input; Eq. 1 with one output pixel):
// y_k = alpha_k sum_j x_j W~_kj, all in fp32.
//
// The tensor-core GEMV takes bf16 activations; rounding fp32 inputs to bf16
// would exceed the accuracy bound, and the CUDA-core direct convolution is
// built for many pixels, not one.  For each group of four inputs this
// kernel tabulates, in fp32, the 256 possible sums sum_i W~_i x_i over the
// four codes' (magnitude, sign) bits; one shared-memory lookup then replaces
// four multiply-adds (the products are exact, each entry and each partial
// sum rounds once per addition).  With the byte-planar code layout the table index of
// four codes is two nibbles of the packed word, so a 16-code word costs two
// multiplies by 16 and 256 (shifts on the FMA pipe), two 3-input logic ops,
// four byte permutes that form the lookup addresses directly, four lookups
// and three adds.
//
// Organisation:
// * The input is cut into chunks of 512 columns.  A chunk's tables are
//   built in shared memory by the CTA: lane l of every warp owns columns
//   16 l .. 16 l + 15 of the chunk (one packed word of a row) through four
//   256-entry tables, one per group of four codes: the even codes 0-6 and
//   8-14 (region E) and the odd codes 1-7 and 9-15 (region O).  Entry idx
//   of table t of lane l lives at region + idx * 256 + t * 128 + 4 l, so a
//   warp's 32 lookups hit 32 different banks, and since each region is
//   64 KB aligned the address is one byte permute of the index into a
//   per-lane base.
// * Work units are (chunk, 128-row block) pairs in chunk-major order,
//   split evenly over a persistent grid (one CTA per SM).  A CTA's range
//   touches one or two chunks, so it builds its tables once or twice.
// * Two producer warps stream the units' [128 rows x 32 words] blocks of
//   codes (16 KB, one TMA box each) into a ring of five stages placed around
//   the tables, taking alternate stages.  Both choices were measured: the
//   box rate of one issuing thread is limited (about one box per L2 round
//   trip plus its transfer), so 2-4 KB boxes capped the kernel near 1-2 TB/s
//   and a single producer near 3.8 TB/s.  All sixteen consumer warps share each
//   stage, eight rows per warp, and release it together.  A warp computes,
//   per row, the sum over its lane's 16 columns; a butterfly over the 32
//   lanes then leaves lanes 4r .. 4r + 3 with the chunk's partial sum for
//   row r of the warp's eight.
// * With one chunk (K_in <= 512) that partial is the result.  Otherwise the
//   partials go to a caller-provided workspace [chunk][row], and a second,
//   small kernel adds each row's chunk partials in chunk order, applies
//   alpha and the epilogue and writes y: the result does not depend on
//   which CTA finished first.  The second kernel is a programmatic
//   dependent launch: its CTAs are scheduled while the first kernel runs
//   and wait (griddepcontrol.wait) for its completion and memory flush.  (Publishing partials to a last-arriving CTA
//   instead needs a device-scope fence per unit, which stalled the warps
//   for longer than the whole second launch costs.)
//
// Every mbarrier wait is bounded; on expiry the kernel records a timeout in
// the device error word, stops issuing, drains the copies it started and
// returns.
#include <cuda.h>
#include <cuda_bf16.h>

#include <cstdint>
#include <mutex>

#include "tbn_device.cuh"
#include "tbn_internal.h"

namespace tbn {
namespace {

constexpr int kLutWarps = 16;                          // consumer warps
constexpr int kLutProducers = 2;                       // producer warps
constexpr int kLutThreads = 32 * (kLutWarps + kLutProducers);
constexpr int kLutProducer = kLutWarps;                // first producer warp
constexpr int kChunkCols = 512;                        // 32 lanes x 16 columns
constexpr int kChunkWords = kChunkCols / 16;
constexpr int kWarpRows = 8;                           // rows of a stage per warp
constexpr int kUnitRows = kWarpRows * kLutWarps;       // 128
constexpr uint32_t kStageBytes = kUnitRows * kChunkWords * 4;   // 16 KB
constexpr uint32_t kRegionBytes = 65536;               // 256 entries x 256 bytes
constexpr int kMaxStages = 8;
// dynamic shared memory: ring stages below the first 64 KB boundary, the two
// 64 KB table regions, then more ring stages up to the end
constexpr size_t kLutSmem = 224 * 1024;
constexpr uint64_t kWaitLimitNs = 1000000000ull;

struct LutArgs {
  const void* x;
  const float* alpha;
  void* y;
  const void* residual;
  float* partial;    // [nchunks][NRB * 32] chunk partial sums (nchunks > 1)
  uint32_t* err;
  long long U;       // units = nchunks * NRB
  int K_in, K_out;
  int nchunks, NRB;
  int y_bf16, relu;
};

__device__ __forceinline__ float load_x(const LutArgs& a, int col) {
  return col < a.K_in ? static_cast<const float*>(a.x)[col] : 0.0f;
}

// Lookup of one table entry at shared address `addr`.  The tables do not
// change between the two barriers around a segment, so the load is a pure
// function of its address and of `epoch` (a value produced by the barrier
// that published the tables); the compiler may schedule it freely after that
// barrier but not before it.
__device__ __forceinline__ float lut_load(uint32_t addr, uint32_t epoch) {
  float v;
  asm("ld.shared.f32 %0, [%1];" : "=f"(v) : "r"(addr), "r"(epoch));
  return v;
}

// Consumer-warp barrier that also yields a token for lut_load.
__device__ __forceinline__ uint32_t consumer_barrier(uint32_t epoch) {
  uint32_t next;
  asm volatile("bar.sync 1, %2;\n\tadd.u32 %0, %1, 1;"
               : "=r"(next)
               : "r"(epoch), "n"(32 * kLutWarps)
               : "memory");
  return next;
}

// Role r (0..15) fills entries 64 part .. 64 part + 63 (part = r / 4) of
// table t of region R ((R, t) = ((r % 4) / 2, r % 2)) for all 32 lanes.  Entry idx of
// lane l: idx bits 0-3 are the magnitude bits m_0..m_3 and bits 4-7 the sign
// bits s_0..s_3 of the four codes, whose columns are 16 l + 8 t + 2 i + R;
// the entry is sum_i (1 - 2 s_i)(1 + m_i) x_i, added as (v_0 + v_1) + (v_2 + v_3).
__device__ __forceinline__ void build_tables(float* region_e, float* region_o, int role, int lane,
                                             float x0, float x1, float x2, float x3) {
  const int combo = role & 3, part = role >> 2;
  const int R = combo >> 1, t = combo & 1;
  // v_i for code field m + 2 s: +x, +2x, -x, -2x
  const float a[4] = {x0, 2.0f * x0, -x0, -2.0f * x0};
  const float b[4] = {x1, 2.0f * x1, -x1, -2.0f * x1};
  float p01[16];
#pragma unroll
  for (int k = 0; k < 16; ++k) {
    // k = m0 | m1 << 1 | s0 << 2 | s1 << 3
    p01[k] = a[(k & 1) | (((k >> 2) & 1) << 1)] + b[((k >> 1) & 1) | (((k >> 3) & 1) << 1)];
  }
  // codes 2 and 3 have the signs fixed by this warp's part: s2 = part & 1, s3 = part >> 1
  const float c = (part & 1) ? -x2 : x2;
  const float d = (part & 2) ? -x3 : x3;
  const float p23[4] = {c + d, 2.0f * c + d, c + 2.0f * d, 2.0f * c + 2.0f * d};
  float* out = (R ? region_o : region_e) + part * 64 * 64 + t * 32 + lane;
#pragma unroll
  for (int j = 0; j < 64; ++j) {
    // idx = 64 part + j: m0..m3 = j bits 0-3, s0 = j bit 4, s1 = j bit 5
    out[j * 64] = p01[(j & 3) | (((j >> 4) & 3) << 2)] + p23[(j >> 2) & 3];
  }
}

template <int kO, int kN>
__device__ __forceinline__ void fold(float (&v)[kWarpRows], bool up) {
#pragma unroll
  for (int i = 0; i < kN / 2; ++i) {
    const float send = up ? v[i] : v[i + kN / 2];
    const float keep = up ? v[i + kN / 2] : v[i];
    v[i] = keep + __shfl_xor_sync(0xffffffffu, send, kO);
  }
}

__device__ __forceinline__ void store_y(const LutArgs& a, int row, float sum) {
  float v = a.alpha[row] * sum;
  if (a.y_bf16) {
    if (a.residual) v += __bfloat162float(static_cast<const __nv_bfloat16*>(a.residual)[row]);
    if (a.relu) v = fmaxf(v, 0.0f);
    static_cast<__nv_bfloat16*>(a.y)[row] = __float2bfloat16_rn(v);
  } else {
    if (a.residual) v += static_cast<const float*>(a.residual)[row];
    if (a.relu) v = fmaxf(v, 0.0f);
    static_cast<float*>(a.y)[row] = v;
  }
}

__global__ void __launch_bounds__(kLutThreads, 1)
    gemv_lut_kernel(const __grid_constant__ CUtensorMap tmap_w, const LutArgs a) {
  extern __shared__ __align__(128) uint8_t smem_raw[];
  __shared__ uint64_t full_bar[kMaxStages], empty_bar[kMaxStages];
  __shared__ uint32_t stage_addr[kMaxStages];
  __shared__ int slot_last[kMaxStages];   // last stage issued into each slot
  __shared__ volatile int abort_flag;

  // layout: stages in [ring, tab), region E at tab (the first 64 KB
  // boundary), region O at tab + 64 KB, more stages after it
  const uint32_t dyn = smem_addr(smem_raw);
  const uint32_t dyn_end = dyn + static_cast<uint32_t>(kLutSmem);
  const uint32_t ring = (dyn + 127u) & ~127u;
  const uint32_t tab = (ring + 0xFFFFu) & ~0xFFFFu;
  const uint32_t ring2 = tab + 2 * kRegionBytes;
  const int n_low = static_cast<int>((tab - ring) / kStageBytes);
  const int n_high = ring2 < dyn_end ? static_cast<int>((dyn_end - ring2) / kStageBytes) : 0;
  const int stages = min(n_low + n_high, kMaxStages);
  if (ring2 > dyn_end || stages < 2) {
    if (threadIdx.x == 0) raise_device_error(a.err, TBN_DEVERR_BAD_LAUNCH);
    return;
  }
  float* region_e = reinterpret_cast<float*>(smem_raw + (tab - dyn));
  float* region_o = region_e + kRegionBytes / 4;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    abort_flag = 0;
    for (int s = 0; s < stages; ++s) {
      stage_addr[s] = s < n_low ? ring + s * kStageBytes : ring2 + (s - n_low) * kStageBytes;
      slot_last[s] = -1;
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], kLutWarps);   // every consumer warp releases every stage
    }
    fence_mbar_init();
  }
  __syncthreads();

  // this CTA's units [u0, u1); unit u = chunk u / NRB, row block u % NRB
  const long long u0 = static_cast<long long>(blockIdx.x) * a.U / gridDim.x;
  const long long u1 = static_cast<long long>(blockIdx.x + 1) * a.U / gridDim.x;
  const int n_local = static_cast<int>(u1 - u0);

  // the reduction kernel (a programmatic dependent launch) may be scheduled
  // now; it waits for this grid's completion before reading anything
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  if (warp >= kLutProducer) {
    // --------------------------------------------------------- producers
    // producer p issues stages it = p, p + 2, ...; the ring has more stages
    // than producers, so the release a producer waits for always follows
    // the previous release of that slot (consumers release in order)
    const int pid = warp - kLutProducer;
    if (elect_one()) prefetch_tmap(&tmap_w);
    const long long ufirst = u0 + pid;
    int c = static_cast<int>(ufirst / a.NRB), rb = static_cast<int>(ufirst % a.NRB);
    for (int it = pid; it < n_local; it += kLutProducers) {
      const int slot = it % stages;
      bool ok = true;
      if (it >= stages)
        ok = mbar_wait(&empty_bar[slot], static_cast<uint32_t>((it / stages - 1) & 1), &abort_flag,
                       a.err, kWaitLimitNs);
      if (!__all_sync(0xffffffffu, ok && !abort_flag)) break;
      if (elect_one()) {
        mbar_arrive_expect_tx(&full_bar[slot], kStageBytes);
        tma_load_2d(smem_raw + (stage_addr[slot] - dyn), &tmap_w, &full_bar[slot],
                    c * kChunkWords, rb * kUnitRows);
        slot_last[slot] = it;
      }
      __syncwarp();
      rb += kLutProducers;
      while (rb >= a.NRB) {
        rb -= a.NRB;
        ++c;
      }
    }
    // On abort, wait (bounded) for the last copy issued into each slot so no
    // TMA write lands after the CTA has exited (both producers have stopped
    // issuing once they pass the barrier).
    named_barrier_sync(2, 32 * kLutProducers);
    if (pid == 0 && __shfl_sync(0xffffffffu, abort_flag, 0) && elect_one()) {
      for (int s = 0; s < stages; ++s) {
        const int i = slot_last[s];
        if (i >= 0)
          mbar_wait(&full_bar[s], static_cast<uint32_t>((i / stages) & 1), nullptr, a.err,
                    kWaitLimitNs);
      }
    }
    return;
  }

  // ------------------------------------------------------------ consumers
  const uint32_t lane4 = static_cast<uint32_t>(lane) * 4u;
  const uint32_t base_e0 = tab | lane4, base_e1 = tab | 128u | lane4;
  const uint32_t base_o0 = (tab + kRegionBytes) | lane4, base_o1 = (tab + kRegionBytes) | 128u | lane4;
  const bool up16 = lane & 16, up8 = lane & 8, up4 = lane & 4;
  // 16 and 256 through an opaque move: the products stay multiplies (FMA
  // pipe) instead of becoming shifts on the integer ALU pipe, which the
  // logic ops and byte permutes already load
  uint32_t mul16, mul256;
  asm("mov.b32 %0, 16;" : "=r"(mul16));
  asm("mov.b32 %0, 256;" : "=r"(mul256));
  const size_t pstride = static_cast<size_t>(a.NRB) * kUnitRows;
  // this warp's rows of a stage: warp * 8 .. warp * 8 + 7; lane = word
  const uint32_t warp_off = static_cast<uint32_t>(warp * kWarpRows * kChunkWords * 4) + lane4;

  uint32_t epoch = 0;
  int slot = 0;
  uint32_t full_parity = 0;
  int c = static_cast<int>(u0 / a.NRB), rb = static_cast<int>(u0 % a.NRB);
  // the four inputs of this warp's table role (one role per consumer warp),
  // loaded one chunk ahead so their latency overlaps the previous chunk's rows
  const int role_col = 16 * lane + 8 * (warp & 1) + ((warp >> 1) & 1);
  float x[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) x[i] = load_x(a, c * kChunkCols + role_col + 2 * i);
  for (int j = 0; j < n_local;) {
    const int seg = min(n_local - j, a.NRB - rb);
    epoch = consumer_barrier(epoch);   // every lookup of the previous chunk is done
    build_tables(region_e, region_o, warp, lane, x[0], x[1], x[2], x[3]);
    epoch = consumer_barrier(epoch);   // the tables are complete
    if (j + seg < n_local) {
#pragma unroll
      for (int i = 0; i < 4; ++i) x[i] = load_x(a, (c + 1) * kChunkCols + role_col + 2 * i);
    }
    for (int q = 0; q < seg; ++q, ++rb) {
      const bool ok_lane = mbar_wait(&full_bar[slot], full_parity, &abort_flag, a.err,
                                     kWaitLimitNs);
      const bool go = __shfl_sync(0xffffffffu, ok_lane ? 1 : 0, 0) != 0;
      float v[kWarpRows];
      if (go) {
        const uint32_t* rows =
            reinterpret_cast<const uint32_t*>(smem_raw + (stage_addr[slot] - dyn) + warp_off);
#pragma unroll
        for (int r = 0; r < kWarpRows; ++r) {
          const uint32_t w = rows[r * kChunkWords];
          const uint32_t w16 = w * mul16, w256 = w * mul256;
          // byte 1: nibble-pair index (m bits, then s bits) of codes 0,2,4,6
          // (ia) / 8,..,14 (ib); byte 3: the same for the odd codes 1,..,7
          // (ia) / 9,..,15 (ib)
          const uint32_t ia = (w256 & 0x0F000F00u) | (w16 & 0xF000F000u);
          const uint32_t ib = (w16 & 0x0F000F00u) | (w & 0xF000F000u);
          const float t0 = lut_load(__byte_perm(ia, base_e0, 0x7614), epoch);
          const float t1 = lut_load(__byte_perm(ib, base_e1, 0x7614), epoch);
          const float t2 = lut_load(__byte_perm(ia, base_o0, 0x7634), epoch);
          const float t3 = lut_load(__byte_perm(ib, base_o1, 0x7634), epoch);
          v[r] = (t0 + t1) + (t2 + t3);
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty_bar[slot]);
      if (++slot == stages) {
        slot = 0;
        full_parity ^= 1u;
      }
      if (!go) continue;
      // lanes 4r .. 4r + 3 end with the sum over all 32 lanes of row r
      fold<16, 8>(v, up16);
      fold<8, 4>(v, up8);
      fold<4, 2>(v, up4);
      v[0] += __shfl_xor_sync(0xffffffffu, v[0], 2);
      v[0] += __shfl_xor_sync(0xffffffffu, v[0], 1);
      const int row = rb * kUnitRows + warp * kWarpRows + (lane >> 2);
      if (lane & 3) continue;
      if (a.nchunks == 1) {
        if (row < a.K_out) store_y(a, row, v[0]);
        continue;
      }
      a.partial[static_cast<size_t>(c) * pstride + row] = v[0];
    }
    j += seg;
    rb = 0;
    ++c;
  }
}

// y[row] = epilogue(alpha[row] * sum over chunks c = 0, 1, ... of
// partial[c][row]), one thread per row.
__global__ void __launch_bounds__(256)
    gemv_lut_reduce_kernel(const LutArgs a) {
  // launched as a programmatic dependent of gemv_lut_kernel: wait for that
  // grid to complete and its partials to be visible
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int row = blockIdx.x * blockDim.x + threadIdx.x;
  if (row >= a.K_out) return;
  const size_t pstride = static_cast<size_t>(a.NRB) * kUnitRows;
  const float* p = a.partial + row;
  float sum = p[0];
#pragma unroll 8
  for (int c = 1; c < a.nchunks; ++c) sum += p[static_cast<size_t>(c) * pstride];
  store_y(a, row, sum);
}

struct LutPlan {
  int nchunks, NRB, grid;
  long long U;
  size_t ws_bytes;
};

LutPlan plan_lut(int64_t K_in, int64_t K_out, int sms) {
  LutPlan p{};
  p.nchunks = static_cast<int>((K_in + kChunkCols - 1) / kChunkCols);
  p.NRB = static_cast<int>((K_out + kUnitRows - 1) / kUnitRows);
  p.U = static_cast<long long>(p.nchunks) * p.NRB;
  p.grid = static_cast<int>(p.U < sms ? p.U : sms);
  if (p.nchunks > 1)
    p.ws_bytes = (static_cast<size_t>(p.nchunks) * p.NRB * kUnitRows * sizeof(float) + 255) &
                 ~size_t(255);
  return p;
}

}  // namespace

const char* gemv_lut_shape_reason(tbn_dtype xdt, int64_t B, int64_t K_in, int64_t K_out) {
  if (xdt != TBN_F32) return "table GEMV takes fp32 activations";
  if (B != 1) return "table GEMV needs B == 1";
  if (K_in % 64 != 0) return "table GEMV needs K_in % 64 == 0 (16-byte code rows for TMA)";
  if (K_in >= (1ll << 30) || K_out >= (1ll << 30)) return "table GEMV: K_in / K_out too large";
  return "";
}

const char* gemv_lut_unsupported_reason(tbn_dtype xdt, int64_t B, int64_t K_in, int64_t K_out,
                                        const uint32_t* codes) {
  const char* r = gemv_lut_shape_reason(xdt, B, K_in, K_out);
  if (r[0] != '\0') return r;
  if (!is_aligned(codes, 16)) return "table GEMV needs 16-byte aligned codes";
  if (get_encode_tiled() == nullptr) return "cuTensorMapEncodeTiled unavailable";
  return "";
}

size_t gemv_lut_workspace_bytes(int64_t K_in, int64_t K_out) {
  return plan_lut(K_in, K_out, 1).ws_bytes;
}

tbn_status launch_gemv_lut(const void* x, int64_t K_in, const uint32_t* codes,
                           const float* alpha, int64_t K_out, void* y, tbn_dtype ydt, int relu,
                           const void* residual, void* workspace, size_t workspace_bytes,
                           cudaStream_t s) {
  const size_t ws_needed = gemv_lut_workspace_bytes(K_in, K_out);
  if (ws_needed > 0) {
    if (workspace == nullptr || workspace_bytes < ws_needed)
      return fail(TBN_ERR_INVALID_ARG, "table GEMV: workspace of %zu bytes needed", ws_needed);
    if (!is_aligned(workspace, 256))
      return fail(TBN_ERR_MISALIGNED, "table GEMV: workspace must be 256-byte aligned");
  }
  const LutPlan p = plan_lut(K_in, K_out, device_sm_count());

  alignas(64) CUtensorMap tmap_w;
  {
    const cuuint64_t gdim[2] = {static_cast<cuuint64_t>(K_in / 16), static_cast<cuuint64_t>(K_out)};
    const cuuint64_t gstride[1] = {static_cast<cuuint64_t>(K_in / 4)};
    const cuuint32_t box[2] = {kChunkWords, kUnitRows};
    const cuuint32_t estr[2] = {1, 1};
    const CUresult cr = get_encode_tiled()(
        &tmap_w, CU_TENSOR_MAP_DATA_TYPE_UINT32, 2, const_cast<uint32_t*>(codes), gdim, gstride,
        box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (cr != CUDA_SUCCESS)
      return fail(TBN_ERR_CUDA, "cuTensorMapEncodeTiled(codes) failed (%d)", (int)cr);
  }

  static std::once_flag attr_once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(attr_once, [] {
    attr_err = cudaFuncSetAttribute((const void*)gemv_lut_kernel,
                                    cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    static_cast<int>(kLutSmem));
  });
  if (attr_err != cudaSuccess) return cuda_fail(attr_err, "cudaFuncSetAttribute(gemv_lut)");

  LutArgs a{};
  a.x = x;
  a.alpha = alpha;
  a.y = y;
  a.residual = residual;
  a.err = device_error_word();
  a.U = p.U;
  a.K_in = static_cast<int>(K_in);
  a.K_out = static_cast<int>(K_out);
  a.nchunks = p.nchunks;
  a.NRB = p.NRB;
  a.y_bf16 = ydt == TBN_BF16 ? 1 : 0;
  a.relu = relu;
  if (p.ws_bytes > 0) a.partial = static_cast<float*>(workspace);
  gemv_lut_kernel<<<p.grid, kLutThreads, kLutSmem, s>>>(tmap_w, a);
  const tbn_status st = check_launch("gemv_lut_kernel");
  if (st != TBN_OK || p.nchunks == 1) return st;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(static_cast<unsigned>((K_out + 255) / 256));
  cfg.blockDim = dim3(256);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, gemv_lut_reduce_kernel, a);
  if (e != cudaSuccess) return cuda_fail(e, "cudaLaunchKernelEx(gemv_lut_reduce_kernel)");
  return check_launch("gemv_lut_reduce_kernel");
}

// ---- the same kernel with file-scope scratch (tbn_linear_fwd_noalloc) ----
// Chunk partial sums for callers that cannot allocate device memory: a
// fixed array in the library's own module, enough for any layer whose
// table-GEMV scratch is at most 4 MiB (e.g. 16384 inputs x 32768 outputs).
// One array per device and process, so calls that could overlap race.
constexpr size_t kStaticScratchBytes = size_t(4) << 20;
static __device__ __align__(256) uint8_t g_lut_scratch[kStaticScratchBytes];

namespace {
constexpr int kMaxDevices = 64;
std::mutex g_scratch_mutex;
void* g_scratch_ptr[kMaxDevices] = {};
}  // namespace

size_t gemv_lut_static_scratch_bytes() { return kStaticScratchBytes; }

tbn_status launch_gemv_lut_static(const void* x, int64_t K_in, const uint32_t* codes,
                                  const float* alpha, int64_t K_out, void* y, tbn_dtype ydt,
                                  int relu, const void* residual, cudaStream_t s) {
  const size_t need = gemv_lut_workspace_bytes(K_in, K_out);
  if (need > kStaticScratchBytes)
    return fail(TBN_ERR_UNSUPPORTED,
                "linear (no-alloc): %zu bytes of scratch needed, the static scratch has %zu",
                need, kStaticScratchBytes);
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (dev < 0 || dev >= kMaxDevices)
    return fail(TBN_ERR_UNSUPPORTED, "linear (no-alloc): device ordinal %d out of range", dev);
  void* ptr = nullptr;
  {
    // set-up once per device, with that device current
    std::lock_guard<std::mutex> lock(g_scratch_mutex);
    if (g_scratch_ptr[dev] == nullptr) {
      e = cudaGetSymbolAddress(&g_scratch_ptr[dev], g_lut_scratch);
      if (e != cudaSuccess) {
        g_scratch_ptr[dev] = nullptr;
        return cuda_fail(e, "cudaGetSymbolAddress(table GEMV scratch)");
      }
    }
    ptr = g_scratch_ptr[dev];
  }
  return launch_gemv_lut(x, K_in, codes, alpha, K_out, y, ydt, relu, residual, ptr,
                         kStaticScratchBytes, s);
}

}  // namespace tbn
