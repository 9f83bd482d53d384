// tbn_quantize.cu -- per-filter discretization + optimal scaling factor +
// two-bit packing (Algorithm 1, quantization loop; Eq. 3 and Eq. 5 of
// Section 2), and the inverse unpack.
//
// One streaming pass over W: Eq. 3's thresholds are absolute (+-1, 0), so
// the codes do not depend on alpha and Eq. 5's two sums can be accumulated
// in the same pass that discretizes.  Each thread encodes whole 32-bit
// output words (16 consecutive weights of a filter): it forms the sixteen
// 2-bit fields, sums |W~|*|W| over the word in fp32 (pairwise) and counts
// the magnitude-two codes; per-word results go to shared memory and one
// warp per filter reduces them in word order.
//
// The kernel is persistent (two CTAs per SM).  A launch's filters (all jobs
// of a group: one network's layers) are cut into tasks of whole filters
// carrying about equal bytes, one task per CTA when they fit.  A task whose
// rows are 16-byte aligned with n % 16 == 0 streams its weights (contiguous
// in W, at most 2048 words = 128 KB) through a ring of three 32 KB shared-
// memory stages filled by 1-D TMA bulk copies (thread 0 keeps three in
// flight, every wait bounded); other tasks load through registers, and a
// filter longer than 2048 words is a task of its own with its words strided
// over the threads.
//
// The word sums are accumulated exactly as a two-float (hi, lo) pair
// (TwoSum, fp32 adds only: GB300's fp64 rate is a small fraction of its fp32
// rate) and alpha = num / (n + 3 |B2|) is formed as hi / den plus the
// remainder correction, one fp32 rounding, well inside 1e-6 relative.  A
// word whose fp32 sum overflows (weights near the fp32 maximum) sends its
// filter down an fp64 path.  Bytes moved per weight: 4 read + 1/4 written.
#include <cuda_bf16.h>

#include <algorithm>
#include <cstdint>
#include <mutex>

#include "tbn_device.cuh"
#include "tbn_internal.h"
#include "tbn_quant_core.cuh"

namespace tbn {
namespace {

constexpr int kThreads = 256;
constexpr int kGroupWords = 1024;                        // words of a register-loaded task
constexpr int kItemWords = 2048;                         // words of a streamed item, at most
constexpr int kChunkBytes = 32768;                       // one ring stage: 512 words
constexpr int kChunkWords = kChunkBytes / 64;
constexpr int kStages = 3;
constexpr int kRingBytes = kStages * kChunkBytes;
constexpr int kCtasPerSm = 2;
constexpr uint64_t kWaitLimitNs = 1000000000ull;

struct QJob {
  const float* W;
  uint32_t* codes;
  float* alpha;
  int64_t K;
  int64_t first_task;  // index of this job's first CTA task
  int32_t n;
  int32_t wpf;   // words per filter
  int32_t vec;   // 16-byte loads allowed
  int32_t rows;  // filters per task (0: one long filter per task, strided words)
  int32_t mode;  // kModeStream, kModeRegs or kModeLong
};

enum : int32_t { kModeStream = 0, kModeRegs = 1, kModeLong = 2 };

struct QParams {
  QJob job[TBN_MAX_QUANT_JOBS];
  int njobs;
  uint32_t* err;
};

// Words j0, j0 + stride, ... of one long filter; accumulates the partials.
__device__ __forceinline__ void quantize_words_strided(const float* __restrict__ row,
                                                       uint32_t* __restrict__ out, int n, int wpf,
                                                       bool vec, int j0, int stride, Sum2& acc,
                                                       int& cnt2, bool& huge) {
  constexpr int kU = 2;
  int j = j0;
  for (; j + (kU - 1) * stride < wpf; j += kU * stride) {
    float v[kU][16];
    int nv[kU];
#pragma unroll
    for (int u = 0; u < kU; ++u) load16(row, n, j + u * stride, vec, v[u], nv[u]);
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      uint32_t word;
      float s;
      int c;
      encode16(v[u], nv[u], word, s, c);
      out[j + u * stride] = word;
      huge |= !finite_sum(s);
      add2(acc, s);
      cnt2 += c;
    }
  }
  for (; j < wpf; j += stride) {
    float v[16];
    int nv;
    load16(row, n, j, vec, v, nv);
    uint32_t word;
    float s;
    int c;
    encode16(v, nv, word, s, c);
    out[j] = word;
    huge |= !finite_sum(s);
    add2(acc, s);
    cnt2 += c;
  }
}

struct QShared {
  float sum[kItemWords];
  int cnt[kItemWords];
  Sum2 part[kThreads / 32];
  int pcnt[kThreads / 32];
  int huge;
};

// One warp per filter of a task: two-float sum of its word sums (word order).
__device__ __forceinline__ void reduce_rows(const QJob& jb, int64_t k0, int nrows,
                                            const float* base, QShared& sh) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (jb.wpf <= 16) {
    // short filters: one thread per filter, its words in order
    for (int r = threadIdx.x; r < nrows; r += kThreads) {
      Sum2 acc{0.0f, 0.0f};
      int cnt2 = 0;
      bool huge = false;
      for (int c = 0; c < jb.wpf; ++c) {
        const float sv = sh.sum[r * jb.wpf + c];
        huge |= !finite_sum(sv);
        add2(acc, sv);
        cnt2 += sh.cnt[r * jb.wpf + c];
      }
      jb.alpha[k0 + r] = huge ? alpha_fp64_row(base + static_cast<int64_t>(r) * jb.n, jb.n)
                              : alpha_of(acc, cnt2, jb.n);
    }
    return;
  }
  for (int r = warp; r < nrows; r += kThreads / 32) {
    Sum2 acc{0.0f, 0.0f};
    int cnt2 = 0;
    bool huge = false;
    for (int c = lane; c < jb.wpf; c += 32) {
      const float sv = sh.sum[r * jb.wpf + c];
      huge |= !finite_sum(sv);
      add2(acc, sv);
      cnt2 += sh.cnt[r * jb.wpf + c];
    }
    acc = warp_sum2(acc);
    cnt2 = warp_sum(cnt2);
    huge = __any_sync(0xffffffffu, huge);
    if (lane == 0)
      jb.alpha[k0 + r] = huge ? alpha_fp64_row(base + static_cast<int64_t>(r) * jb.n, jb.n)
                              : alpha_of(acc, cnt2, jb.n);
  }
}

// A streamed task's weights: nrows whole filters from filter k0 of job jb,
// `words` packed words (64 bytes of fp32 weights each), in `nch` chunks.
struct StreamTask {
  const QJob* jb;
  int64_t k0;
  int nrows;
  int words;
  int nch;
  const uint8_t* src;
};

__device__ __forceinline__ StreamTask stream_task(const QJob& jb, int64_t k0, int nrows) {
  StreamTask t;
  t.jb = &jb;
  t.k0 = k0;
  t.nrows = nrows;
  t.words = nrows * jb.wpf;
  t.nch = (t.words + kChunkWords - 1) / kChunkWords;
  t.src = reinterpret_cast<const uint8_t*>(jb.W + k0 * static_cast<int64_t>(jb.n));
  return t;
}

// Thread 0: bulk copy of chunk i of task t into ring slot g % kStages.
__device__ __forceinline__ void issue_chunk(const StreamTask& t, int i, uint32_t g, uint8_t* ring,
                                            uint64_t* full) {
  const uint32_t bytes = static_cast<uint32_t>(t.words) * 64u;
  const uint32_t off = static_cast<uint32_t>(i) * kChunkBytes;
  const uint32_t len = bytes - off < static_cast<uint32_t>(kChunkBytes) ? bytes - off
                                                                        : static_cast<uint32_t>(kChunkBytes);
  mbar_arrive_expect_tx(&full[g % kStages], len);
  bulk_load_1d(ring + (g % kStages) * kChunkBytes, t.src + off, len, &full[g % kStages]);
}

// Streamed task: nrows whole filters (n % 16 == 0, 16-byte aligned rows,
// nrows * wpf <= kItemWords words) flow through the ring of kStages 32 KB
// chunks; thread 0 keeps up to kStages bulk copies in flight.  The chunks of
// all this CTA's consecutive streamed tasks form one sequence: `seq` counts
// the chunks consumed so far (every thread), `issued` those whose copy was
// issued (thread 0, which issues them).  Once a task has issued its last
// chunk, the freed slots take the first chunks of the next task (`nxt`, if
// it streams too), so the ring does not drain at task boundaries.  Returns false if a wait timed
// out (after draining every copy in flight).
__device__ bool task_stream(const StreamTask& t, const StreamTask* nxt, QShared& sh, uint8_t* ring,
                            uint64_t* full, uint32_t& seq, uint32_t& issued, uint32_t* err) {
  const QJob& jb = *t.jb;
  uint32_t* out = jb.codes + t.k0 * static_cast<int64_t>(jb.wpf);
  const uint32_t end = seq + static_cast<uint32_t>(t.nch);   // this task's chunks: [seq, end)
  // issue (thread 0) every chunk of the sequence up to `upto`
  auto top_up = [&](uint32_t upto) {
    while (issued < upto) {
      if (issued < end) {
        issue_chunk(t, static_cast<int>(issued - seq), issued, ring, full);
      } else if (nxt != nullptr && issued < end + static_cast<uint32_t>(nxt->nch)) {
        issue_chunk(*nxt, static_cast<int>(issued - end), issued, ring, full);
      } else {
        break;
      }
      ++issued;
    }
  };
  if (threadIdx.x == 0) top_up(seq + kStages);
  for (int i = 0; i < t.nch; ++i) {
    const uint32_t g = seq + static_cast<uint32_t>(i);
    const bool ok = mbar_wait(&full[g % kStages], (g / kStages) & 1u, nullptr, err, kWaitLimitNs);
    if (ok) {
      const float* chunk = reinterpret_cast<const float*>(ring + (g % kStages) * kChunkBytes);
      const int w0 = i * kChunkWords;
      const int wn = t.words - w0 < kChunkWords ? t.words - w0 : kChunkWords;
#pragma unroll
      for (int u = 0; u < kChunkWords / kThreads; ++u) {
        const int w = threadIdx.x + u * kThreads;
        if (w >= wn) break;
        float v[16];
        const float4* q4 = reinterpret_cast<const float4*>(chunk + 16 * w);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const float4 t4 = q4[q];
          v[4 * q + 0] = t4.x;
          v[4 * q + 1] = t4.y;
          v[4 * q + 2] = t4.z;
          v[4 * q + 3] = t4.w;
        }
        uint32_t word;
        float sum;
        int c2;
        encode16(v, 16, word, sum, c2);
        out[w0 + w] = word;   // the task's words are contiguous in the codes array
        sh.sum[w0 + w] = sum;
        sh.cnt[w0 + w] = c2;
      }
    }
    // everyone is done with this slot (or something timed out)
    if (__syncthreads_or(!ok)) {
      if (threadIdx.x == 0) {
        // copies issued but not consumed: g .. issued - 1
        for (uint32_t gj = g; gj != issued; ++gj)
          mbar_wait(&full[gj % kStages], (gj / kStages) & 1u, nullptr, err, kWaitLimitNs);
      }
      return false;
    }
    if (threadIdx.x == 0) top_up(g + 1 + kStages);
  }
  seq = end;
  reduce_rows(jb, t.k0, t.nrows, reinterpret_cast<const float*>(t.src), sh);
  __syncthreads();   // sums consumed before the next task overwrites them
  return true;
}

// Register-loaded task (rows not 16-byte aligned or n % 16 != 0; small
// layers such as a network's first): one word per thread per round.
__device__ void task_regs(const QJob& jb, int64_t k0, int nrows, QShared& sh) {
  const int nwords = nrows * jb.wpf;
  const float* base = jb.W + k0 * static_cast<int64_t>(jb.n);
  uint32_t* out = jb.codes + k0 * static_cast<int64_t>(jb.wpf);
  for (int j = threadIdx.x; j < nwords; j += kThreads) {
    const int r = j / jb.wpf, c = j - r * jb.wpf;
    float v[16];
    int nv;
    load16(base + static_cast<int64_t>(r) * jb.n, jb.n, c, jb.vec != 0, v, nv);
    uint32_t word;
    float sum;
    int c2;
    encode16(v, nv, word, sum, c2);
    out[j] = word;
    sh.sum[j] = sum;
    sh.cnt[j] = c2;
  }
  __syncthreads();
  reduce_rows(jb, k0, nrows, base, sh);
  __syncthreads();
}

// One long filter (more than kItemWords words): words strided over the
// threads, block reduction.
__device__ void task_long(const QJob& jb, int64_t k, QShared& sh) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const float* row = jb.W + k * static_cast<int64_t>(jb.n);
  uint32_t* out = jb.codes + k * static_cast<int64_t>(jb.wpf);
  Sum2 acc{0.0f, 0.0f};
  int cnt2 = 0;
  bool huge = false;
  if (threadIdx.x == 0) sh.huge = 0;
  quantize_words_strided(row, out, jb.n, jb.wpf, jb.vec != 0, threadIdx.x, kThreads, acc, cnt2,
                         huge);
  acc = warp_sum2(acc);
  cnt2 = warp_sum(cnt2);
  __syncthreads();
  if (huge) sh.huge = 1;
  if (lane == 0) {
    sh.part[warp] = acc;
    sh.pcnt[warp] = cnt2;
  }
  __syncthreads();
  if (warp == 0) {
    Sum2 t = lane < kThreads / 32 ? sh.part[lane] : Sum2{0.0f, 0.0f};
    int c = lane < kThreads / 32 ? sh.pcnt[lane] : 0;
    t = warp_sum2(t);
    c = warp_sum(c);
    if (lane == 0) jb.alpha[k] = sh.huge ? alpha_fp64_row(row, jb.n) : alpha_of(t, c, jb.n);
  }
  __syncthreads();
}

// The job a task belongs to.
__device__ __forceinline__ int job_of(const QParams& prm, int64_t task) {
  int ji = 0;
#pragma unroll 1
  for (int i = 1; i < prm.njobs; ++i)
    if (task >= prm.job[i].first_task) ji = i;
  return ji;
}

// Persistent: CTA b takes tasks b, b + grid, ...; a task is a run of whole
// filters of one job (sized so that tasks carry about equal bytes).
__global__ void __launch_bounds__(kThreads, kCtasPerSm) quantize_pack_kernel(const __grid_constant__ QParams prm,
                                                                    int64_t ntasks) {
  extern __shared__ __align__(128) uint8_t q_ring[];   // kRingBytes when any job streams
  __shared__ QShared sh;
  __shared__ uint64_t full[kStages];
  if (threadIdx.x == 0) {
    for (int i = 0; i < kStages; ++i) mbar_init(&full[i], 1);
    fence_mbar_init();
  }
  __syncthreads();
  uint32_t seq = 0, issued = 0;   // streamed chunks consumed (all threads) / issued (thread 0)
  for (int64_t task = blockIdx.x; task < ntasks; task += gridDim.x) {
    const QJob& jb = prm.job[job_of(prm, task)];
    const int64_t local = task - jb.first_task;
    if (jb.mode == kModeLong) {
      task_long(jb, local, sh);
    } else {
      const int64_t k0 = local * jb.rows;
      const int nrows = static_cast<int>(jb.K - k0 < jb.rows ? jb.K - k0 : jb.rows);
      if (jb.mode == kModeStream) {
        // the CTA's next task, when it streams too, is prefetched into the ring
        StreamTask nt{};
        const StreamTask* nxt = nullptr;
        const int64_t task2 = task + gridDim.x;
        if (task2 < ntasks) {
          const QJob& jb2 = prm.job[job_of(prm, task2)];
          if (jb2.mode == kModeStream) {
            const int64_t k2 = (task2 - jb2.first_task) * jb2.rows;
            nt = stream_task(jb2, k2, static_cast<int>(jb2.K - k2 < jb2.rows ? jb2.K - k2 : jb2.rows));
            nxt = &nt;
          }
        }
        if (!task_stream(stream_task(jb, k0, nrows), nxt, sh, q_ring, full, seq, issued, prm.err))
          return;
      } else {
        task_regs(jb, k0, nrows, sh);
      }
    }
  }
}

template <int kFmt>
__global__ void __launch_bounds__(256) unpack_kernel(const uint32_t* __restrict__ codes,
                                                     const float* __restrict__ alpha, int64_t K,
                                                     int64_t n, int64_t wpf, void* out) {
  const int64_t total = K * wpf;
  for (int64_t t = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; t < total;
       t += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t k = t / wpf, j = t % wpf;
    const uint32_t w = codes[t];
    const float a = (kFmt == TBN_UNPACK_I8) ? 1.0f : alpha[k];
    const int64_t base = k * n + 16 * j;
    const int64_t left = n - 16 * j;
    const int cnt = left < 16 ? static_cast<int>(left) : 16;
    for (int e = 0; e < cnt; ++e) {
      const float v = code_value(code_field(w, e));
      if (kFmt == TBN_UNPACK_I8) {
        static_cast<int8_t*>(out)[base + e] = static_cast<int8_t>(v);
      } else if (kFmt == TBN_UNPACK_F32) {
        static_cast<float*>(out)[base + e] = a * v;
      } else {
        static_cast<__nv_bfloat16*>(out)[base + e] = __float2bfloat16_rn(a * v);
      }
    }
  }
}

// ---- canonical <-> byte-planar repacking ----
// Both layouts hold the same 2-bit field f = m + 2 s per code and 0 in the
// unused fields, so a repack is a fixed permutation of the 32 bits of each
// word.  Canonical: code l (0..15) at bits 2l (m) and 2l + 1 (s).
// Byte-planar: code l = 2p + h at bits 16h + p (m) and 16h + 8 + p (s).
// gather_even(v) moves bits 0, 2, 4, ... 30 of v to bits 0..15; scatter_even
// is its inverse (standard bit (un)interleaving by masks).
__device__ __forceinline__ uint32_t gather_even(uint32_t v) {
  v &= 0x55555555u;
  v = (v | (v >> 1)) & 0x33333333u;
  v = (v | (v >> 2)) & 0x0F0F0F0Fu;
  v = (v | (v >> 4)) & 0x00FF00FFu;
  v = (v | (v >> 8)) & 0x0000FFFFu;
  return v;
}

__device__ __forceinline__ uint32_t scatter_even(uint32_t v) {
  v &= 0x0000FFFFu;
  v = (v | (v << 8)) & 0x00FF00FFu;
  v = (v | (v << 4)) & 0x0F0F0F0Fu;
  v = (v | (v << 2)) & 0x33333333u;
  v = (v | (v << 1)) & 0x55555555u;
  return v;
}

__device__ __forceinline__ uint32_t canonical_to_planar(uint32_t c) {
  const uint32_t m = gather_even(c), sg = gather_even(c >> 1);   // bit l = code l
  return gather_even(m) | (gather_even(sg) << 8) | (gather_even(m >> 1) << 16) |
         (gather_even(sg >> 1) << 24);
}

__device__ __forceinline__ uint32_t planar_to_canonical(uint32_t w) {
  const uint32_t m = scatter_even(w & 0xFFu) | (scatter_even((w >> 16) & 0xFFu) << 1);
  const uint32_t sg = scatter_even((w >> 8) & 0xFFu) | (scatter_even(w >> 24) << 1);
  return scatter_even(m) | (scatter_even(sg) << 1);
}

template <bool kToPlanar>
__global__ void __launch_bounds__(256) repack_kernel(const uint32_t* __restrict__ in,
                                                     int64_t words, uint32_t* __restrict__ out) {
  for (int64_t t = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; t < words;
       t += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const uint32_t w = __ldg(in + t);
    out[t] = kToPlanar ? canonical_to_planar(w) : planar_to_canonical(w);
  }
}

}  // namespace

tbn_status launch_quantize_group(const tbn_quant_job* jobs, int njobs, cudaStream_t s) {
  QParams prm{};
  prm.njobs = njobs;
  prm.err = device_error_word();
  const int slots = device_sm_count() * kCtasPerSm;
  // tasks of about equal bytes: the group's words spread over one task per CTA slot
  int64_t total_words = 0;
  for (int i = 0; i < njobs; ++i) total_words += jobs[i].K * ((jobs[i].n + 15) / 16);
  const int64_t target = std::max<int64_t>(1, (total_words + slots - 1) / std::max(1, slots));
  int64_t tasks = 0;
  bool any_stream = false;
  for (int i = 0; i < njobs; ++i) {
    const tbn_quant_job& j = jobs[i];
    QJob& q = prm.job[i];
    q.W = j.W;
    q.codes = j.codes;
    q.alpha = j.alpha;
    q.K = j.K;
    q.n = static_cast<int32_t>(j.n);
    q.wpf = static_cast<int32_t>((j.n + 15) / 16);
    q.vec = (is_aligned(j.W, 16) && (j.n % 4) == 0) ? 1 : 0;
    if (q.vec && j.n % 16 == 0 && q.wpf <= kItemWords) {
      q.mode = kModeStream;
      const int64_t want = (std::min<int64_t>(target, kItemWords) + q.wpf - 1) / q.wpf;
      q.rows = static_cast<int32_t>(std::max<int64_t>(1, std::min<int64_t>({want, j.K, kItemWords / q.wpf})));
      any_stream = true;
    } else if (q.wpf <= kGroupWords) {
      q.mode = kModeRegs;
      q.rows = static_cast<int32_t>(std::min<int64_t>(j.K, kGroupWords / q.wpf));
    } else {
      q.mode = kModeLong;
      q.rows = 0;
    }
    q.first_task = tasks;
    tasks += q.rows == 0 ? j.K : (j.K + q.rows - 1) / q.rows;
  }
  if (tasks == 0) return TBN_OK;
  if (tasks > 0x7fffffffLL) return fail(TBN_ERR_UNSUPPORTED, "quantize: too many filters (%lld tasks)", (long long)tasks);
  static std::once_flag attr_once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(attr_once, [] {
    attr_err = cudaFuncSetAttribute(quantize_pack_kernel,
                                    cudaFuncAttributeMaxDynamicSharedMemorySize, kRingBytes);
    if (attr_err == cudaSuccess)   // two ring-holding CTAs per SM
      attr_err = cudaFuncSetAttribute(quantize_pack_kernel,
                                      cudaFuncAttributePreferredSharedMemoryCarveout, 100);
  });
  if (attr_err != cudaSuccess) return cuda_fail(attr_err, "cudaFuncSetAttribute(quantize)");
  const unsigned grid = static_cast<unsigned>(std::min<int64_t>(tasks, slots));
  quantize_pack_kernel<<<grid, kThreads, any_stream ? kRingBytes : 0, s>>>(prm, tasks);
  return check_launch("quantize_pack_kernel");
}

tbn_status launch_unpack(const uint32_t* codes, const float* alpha, int64_t K, int64_t n,
                         void* out, tbn_unpack_format fmt, cudaStream_t s) {
  const int64_t wpf = (n + 15) / 16;
  const int64_t total = K * wpf;
  const int64_t blocks = std::min<int64_t>((total + 255) / 256, 65536);
  switch (fmt) {
    case TBN_UNPACK_I8:
      unpack_kernel<TBN_UNPACK_I8><<<blocks, 256, 0, s>>>(codes, alpha, K, n, wpf, out);
      break;
    case TBN_UNPACK_F32:
      unpack_kernel<TBN_UNPACK_F32><<<blocks, 256, 0, s>>>(codes, alpha, K, n, wpf, out);
      break;
    case TBN_UNPACK_BF16:
      unpack_kernel<TBN_UNPACK_BF16><<<blocks, 256, 0, s>>>(codes, alpha, K, n, wpf, out);
      break;
  }
  return check_launch("unpack_kernel");
}

tbn_status launch_repack(const uint32_t* in, int64_t words, uint32_t* out, bool to_planar,
                         cudaStream_t s) {
  const int64_t blocks =
      std::max<int64_t>(1, std::min<int64_t>((words + 255) / 256, int64_t(device_sm_count()) * 8));
  if (to_planar)
    repack_kernel<true><<<static_cast<unsigned>(blocks), 256, 0, s>>>(in, words, out);
  else
    repack_kernel<false><<<static_cast<unsigned>(blocks), 256, 0, s>>>(in, words, out);
  return check_launch("repack_kernel");
}

}  // namespace tbn
