// tbn_conv_smalltap.cu -- two-bit convolution (Eq. 1) for layers whose
// filters are short, n = C*R*S <= 64 (the first layer of an image network:
// 3 channels x 3x3 taps = 27), bf16 activations in NCHW or NHWC.
//
// The implicit-GEMM kernel pads such a layer's K dimension to a 64-code
// block and has its gather warps fetch every activation with a scalar load,
// so the layer ends up bound by latency while its real cost is writing the
// output.  Here a CTA takes an output tile of up to 256 pixels (whole rows
// of one image when they fit) and 128 filters:
//   1. the input patch the tile needs is copied into shared memory with
//      zero padding (coalesced row reads, any stride / padding);
//   2. the threads expand it once into an im2col block [pixels][KP codes]
//      (KP = 32 or 64; codes past n are zero) in shared memory, 16-byte
//      chunks XOR-swizzled so ldmatrix reads are conflict-free;
//   3. each of the 8 warps owns 16 filters: their codes are decoded once
//      per CTA into mma B fragments (bf16 W~/2, byte-planar decode), and the
//      warp runs mma.m16n8k16 over the tile, 16 pixels at a time, with A =
//      im2col rows from ldmatrix and fp32 accumulation;
//   4. the epilogue applies 2 alpha, the residual and ReLU and stores the
//      fragments straight to global memory (each pixel's 8 consecutive
//      filters of an n-tile are 16 contiguous bytes in NHWC).
// CTAs are persistent (a few per SM) and walk the tiles with a grid stride.
// Launched as a programmatic dependent of the previous kernel: the set-up
// before the tile loop may overlap that kernel's end; activations are read
// only after it has completed (grid_dependency_wait).
#include <cuda_bf16.h>

#include <algorithm>
#include <cstdint>
#include <cstring>
#include <mutex>

#include "tbn_device.cuh"
#include "tbn_internal.h"

namespace tbn {
namespace {

constexpr int kThreads = 256;
constexpr int kFiltersPerCta = 128;           // 16 per warp = two 8-filter n-tiles
constexpr int kMaxTilePixels = 256;
constexpr int kMaxCodes = 64;
constexpr int kMaxPatchBytes = 16 * 1024;
constexpr int kCtasPerSm = 2;

struct SmallTapArgs {
  int N, C, H, W, K, R, S, sh, sw, ph, pw, P, Q;
  int n;            // codes per filter, C*R*S
  int wpf;          // words per filter
  int TP, TQ;       // tile rows / columns of output
  int tiles_p, tiles_q, tiles_k, tiles;
  int PH, PW;       // patch rows / columns
  int x_nhwc;       // x is [N][H][W][C] (else [N][C][H][W])
  int rsc;          // codes in (r, s, c) order (else (c, r, s))
  int y_nhwc;       // y and residual are [N][P][Q][K] (else [N][K][P][Q])
  int y_bf16, relu;
  const __nv_bfloat16* x;
  const uint32_t* codes;
  const float* alpha;
  void* y;
  const void* residual;
  // tensor-core variant
  int mma_n;        // MMA N: tile pixels rounded up to 16
  int patch_bytes;  // patch buffer size (multiple of 16)
  uint32_t* err;    // device error word
};

__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], uint32_t a0, uint32_t a1,
                                               uint32_t a2, uint32_t a3, uint32_t b0,
                                               uint32_t b1) {
  asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
      "{%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ void ldmatrix_x4(uint32_t (&r)[4], uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr)
               : "memory");
}

// Byte offset of 16-byte chunk c of im2col row `row` (row = KP codes).
template <int KP>
__device__ __forceinline__ uint32_t im2col_off(int row, int c) {
  if constexpr (KP == 64) {
    return static_cast<uint32_t>(row * 128 + ((c ^ (row & 7)) << 4));
  } else {
    return static_cast<uint32_t>(row * 64 + ((c ^ ((row >> 1) & 3)) << 4));
  }
}

// Pair p of a packed word as bf16x2 of W~/2 (byte-planar layout).
__device__ __forceinline__ uint32_t decode_pair(uint32_t w, int p) {
  return ((w >> p) & 0x01010101u) * 0x80u + 0x3F003F00u;
}

// Epilogue of the general path: one (pixel, filter pair) per call, any
// layout / dtype / residual.
__device__ __forceinline__ void store_pair(const SmallTapArgs& a, int img, int p, int q, int f,
                                           float v0, float v1) {
  const bool has1 = f + 1 < a.K;
  if (a.y_nhwc) {
    const size_t o = ((static_cast<size_t>(img) * a.P + p) * a.Q + q) * a.K + f;
    if (a.residual) {
      if (a.y_bf16) {
        v0 += __bfloat162float(static_cast<const __nv_bfloat16*>(a.residual)[o]);
        if (has1) v1 += __bfloat162float(static_cast<const __nv_bfloat16*>(a.residual)[o + 1]);
      } else {
        v0 += static_cast<const float*>(a.residual)[o];
        if (has1) v1 += static_cast<const float*>(a.residual)[o + 1];
      }
    }
    if (a.relu) {
      v0 = fmaxf(v0, 0.0f);
      v1 = fmaxf(v1, 0.0f);
    }
    if (a.y_bf16) {
      __nv_bfloat16* y = static_cast<__nv_bfloat16*>(a.y);
      if (has1 && (reinterpret_cast<uintptr_t>(y + o) & 3u) == 0) {
        *reinterpret_cast<__nv_bfloat162*>(y + o) = __floats2bfloat162_rn(v0, v1);
      } else {
        y[o] = __float2bfloat16_rn(v0);
        if (has1) y[o + 1] = __float2bfloat16_rn(v1);
      }
    } else {
      float* y = static_cast<float*>(a.y);
      if (has1 && (reinterpret_cast<uintptr_t>(y + o) & 7u) == 0) {
        *reinterpret_cast<float2*>(y + o) = make_float2(v0, v1);
      } else {
        y[o] = v0;
        if (has1) y[o + 1] = v1;
      }
    }
  } else {
    const size_t plane = static_cast<size_t>(a.P) * a.Q;
    const size_t o0 =
        (static_cast<size_t>(img) * a.K + f) * plane + static_cast<size_t>(p) * a.Q + q;
    const size_t o1 = o0 + plane;
    if (a.residual) {
      if (a.y_bf16) {
        v0 += __bfloat162float(static_cast<const __nv_bfloat16*>(a.residual)[o0]);
        if (has1) v1 += __bfloat162float(static_cast<const __nv_bfloat16*>(a.residual)[o1]);
      } else {
        v0 += static_cast<const float*>(a.residual)[o0];
        if (has1) v1 += static_cast<const float*>(a.residual)[o1];
      }
    }
    if (a.relu) {
      v0 = fmaxf(v0, 0.0f);
      v1 = fmaxf(v1, 0.0f);
    }
    if (a.y_bf16) {
      __nv_bfloat16* y = static_cast<__nv_bfloat16*>(a.y);
      y[o0] = __float2bfloat16_rn(v0);
      if (has1) y[o1] = __float2bfloat16_rn(v1);
    } else {
      float* y = static_cast<float*>(a.y);
      y[o0] = v0;
      if (has1) y[o1] = v1;
    }
  }
}

// Byte offset of the 16-byte chunk holding filters 8c .. 8c+7 of staged
// pixel row px (a row = 128 bf16 filters = 256 B; chunks XOR-swizzled by the
// row so that eight rows written or read at once use all 32 banks).
__device__ __forceinline__ uint32_t stage_off(int px, int c) {
  return static_cast<uint32_t>(px * 256 + ((c ^ (px & 15)) << 4));
}

// kStaged: NHWC bf16 output, no residual, K % 8 == 0, 16-byte aligned y.
// The tile's results are staged in shared memory and written with 16-byte
// stores; otherwise every lane stores its fragment pairs directly.
template <int KP, bool kStaged>
__global__ void __launch_bounds__(kThreads, kCtasPerSm) conv_smalltap_kernel(SmallTapArgs a) {
  extern __shared__ __align__(128) uint8_t smem[];
  uint8_t* im2col = smem;
  uint8_t* staging = smem + kMaxTilePixels * KP * 2;
  int* pxtab = reinterpret_cast<int*>(staging + (kStaged ? kMaxTilePixels * kFiltersPerCta * 2 : 0));
  int* pxbase = pxtab + kMaxTilePixels;
  __nv_bfloat16* patch = reinterpret_cast<__nv_bfloat16*>(pxbase + kMaxTilePixels);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, t = lane & 3;
  constexpr int kChunks = KP / 8;   // 16-byte chunks per im2col row

  // Tile-independent tables: pixel px of a tile is output (pp, qq) =
  // (px / TQ, px % TQ) and reads the patch from offset pxbase[px].
  for (int px = tid; px < kMaxTilePixels; px += kThreads) {
    const int pp = px / a.TQ, qq = px % a.TQ;
    pxtab[px] = (pp << 16) | qq;
    pxbase[px] = (pp * a.sh * a.PW + qq * a.sw) * a.C;
  }
  // This thread always builds chunk `my_ch` of its im2col rows: the patch
  // offsets of its eight codes (-1 past n).
  const int my_ch = tid % kChunks;
  int koff[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const int k = my_ch * 8 + j;
    int off = -1;
    if (k < a.n) {
      int c, r, s;
      if (a.rsc) {
        c = k % a.C;
        s = (k / a.C) % a.S;
        r = k / (a.C * a.S);
      } else {
        s = k % a.S;
        r = (k / a.S) % a.R;
        c = k / (a.S * a.R);
      }
      off = (r * a.PW + s) * a.C + c;
    }
    koff[j] = off;
  }

  int cur_ktile = -1;
  uint32_t bfrag[2][KP / 16][2];
  float two_alpha[2][2];
  const uint32_t im2col_s = smem_addr(im2col);
  const int tile_px = a.TP * a.TQ;
  const int m_pad = (tile_px + 15) & ~15;
  const int row_elems = a.PW * a.C;

  grid_dependency_wait();   // activations may come from the previous kernel
  grid_dependents_launch();
  for (int tile = blockIdx.x; tile < a.tiles; tile += gridDim.x) {
    // tile order: k-tile slowest so a CTA keeps its decoded filters
    const int kt = tile / (a.N * a.tiles_p * a.tiles_q);
    int rest = tile % (a.N * a.tiles_p * a.tiles_q);
    const int img = rest / (a.tiles_p * a.tiles_q);
    rest %= a.tiles_p * a.tiles_q;
    const int p0 = (rest / a.tiles_q) * a.TP, q0 = (rest % a.tiles_q) * a.TQ;
    const int p_lim = a.P - p0, q_lim = a.Q - q0;

    if (kt != cur_ktile) {
      cur_ktile = kt;
#pragma unroll
      for (int nt = 0; nt < 2; ++nt) {
        const int f = kt * kFiltersPerCta + warp * 16 + nt * 8 + g;
        const bool fv = f < a.K;
#pragma unroll
        for (int ks = 0; ks < KP / 16; ++ks) {
          const uint32_t w =
              (fv && ks < a.wpf) ? __ldg(a.codes + static_cast<size_t>(f) * a.wpf + ks) : 0u;
          bfrag[nt][ks][0] = decode_pair(w, t);
          bfrag[nt][ks][1] = decode_pair(w, t + 4);
        }
        // epilogue scale for this lane's output filters 2t, 2t + 1 of the n-tile
        const int fo = kt * kFiltersPerCta + warp * 16 + nt * 8 + 2 * t;
        two_alpha[nt][0] = fo < a.K ? 2.0f * __ldg(a.alpha + fo) : 0.0f;
        two_alpha[nt][1] = fo + 1 < a.K ? 2.0f * __ldg(a.alpha + fo + 1) : 0.0f;
      }
    }

    __syncthreads();   // the previous tile is finished with every buffer
    // 1. input patch, zero outside the image: NHWC rows are contiguous runs
    //    of W*C elements, NCHW rows runs of W elements per channel
    const int ih0 = p0 * a.sh - a.ph, iw0 = q0 * a.sw - a.pw;
    if (a.x_nhwc) {
      // thread owns row offsets e = tid, tid + 256, ...; all its loads of a
      // batch of rows are issued before any is stored
      const int e0 = iw0 * a.C, row_len = a.W * a.C;
      const __nv_bfloat16* img_x = a.x + static_cast<size_t>(img) * a.H * row_len;
      constexpr int kBatch = 8;
      for (int e = tid; e < row_elems; e += kThreads) {
        const int ge = e0 + e;
        const bool cv = ge >= 0 && ge < row_len;
        for (int ih0b = 0; ih0b < a.PH; ih0b += kBatch) {
          uint16_t v[kBatch];
#pragma unroll
          for (int j = 0; j < kBatch; ++j) {
            const int gh = ih0 + ih0b + j;
            const bool ok = cv && ih0b + j < a.PH && gh >= 0 && gh < a.H;
            v[j] = ok ? __bfloat16_as_ushort(img_x[static_cast<size_t>(gh) * row_len + ge]) : 0;
          }
#pragma unroll
          for (int j = 0; j < kBatch; ++j)
            if (ih0b + j < a.PH) patch[(ih0b + j) * row_elems + e] = __ushort_as_bfloat16(v[j]);
        }
      }
    } else {
      for (int c = 0; c < a.C; ++c) {
        for (int ih = 0; ih < a.PH; ++ih) {
          const int gh = ih0 + ih;
          const bool hv = gh >= 0 && gh < a.H;
          const __nv_bfloat16* src =
              a.x + ((static_cast<size_t>(img) * a.C + c) * a.H + (hv ? gh : 0)) * a.W;
          for (int iw = tid; iw < a.PW; iw += kThreads) {
            const int gw = iw0 + iw;
            patch[(ih * a.PW + iw) * a.C + c] =
                (hv && gw >= 0 && gw < a.W) ? src[gw] : __float2bfloat16_rn(0.0f);
          }
        }
      }
    }
    __syncthreads();
    // 2. im2col: this thread builds chunk my_ch of rows tid / kChunks + 256 / kChunks * i
    for (int px = tid / kChunks; px < m_pad; px += kThreads / kChunks) {
      const int tab = pxtab[px];
      const bool pv = px < tile_px && (tab >> 16) < p_lim && (tab & 0xFFFF) < q_lim;
      const __nv_bfloat16* src = patch + pxbase[px];
      uint32_t v[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const uint16_t lo = (pv && koff[2 * i] >= 0) ? __bfloat16_as_ushort(src[koff[2 * i]]) : 0;
        const uint16_t hi =
            (pv && koff[2 * i + 1] >= 0) ? __bfloat16_as_ushort(src[koff[2 * i + 1]]) : 0;
        v[i] = static_cast<uint32_t>(lo) | (static_cast<uint32_t>(hi) << 16);
      }
      *reinterpret_cast<uint4*>(im2col + im2col_off<KP>(px, my_ch)) =
          make_uint4(v[0], v[1], v[2], v[3]);
    }
    __syncthreads();

    // 3. mma over 16-pixel groups; ldmatrix lane address: matrix m = lane / 8
    //    (m & 1: pixel rows 8..15, m >> 1: upper 8 codes of the K step)
    const int lm = lane >> 3, lr = lane & 7;
    for (int grp = 0; grp < m_pad / 16; ++grp) {
      const int row = grp * 16 + (lm & 1) * 8 + lr;
      float acc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
#pragma unroll
      for (int ks = 0; ks < KP / 16; ++ks) {
        uint32_t af[4];
        ldmatrix_x4(af, im2col_s + im2col_off<KP>(row, 2 * ks + (lm >> 1)));
        mma_bf16_16816(acc[0], af[0], af[1], af[2], af[3], bfrag[0][ks][0], bfrag[0][ks][1]);
        mma_bf16_16816(acc[1], af[0], af[1], af[2], af[3], bfrag[1][ks][0], bfrag[1][ks][1]);
      }
      // 4. epilogue: lane holds pixels grp*16 + g (+8), filters 2t, 2t+1 of each n-tile
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        const int px = grp * 16 + g + 8 * half;
        if constexpr (kStaged) {
#pragma unroll
          for (int nt = 0; nt < 2; ++nt) {
            float v0 = two_alpha[nt][0] * acc[nt][2 * half];
            float v1 = two_alpha[nt][1] * acc[nt][2 * half + 1];
            if (a.relu) {
              v0 = fmaxf(v0, 0.0f);
              v1 = fmaxf(v1, 0.0f);
            }
            const __nv_bfloat162 pr = __floats2bfloat162_rn(v0, v1);
            *reinterpret_cast<__nv_bfloat162*>(staging + stage_off(px, warp * 2 + nt) + 4 * t) = pr;
          }
        } else {
          const int tab = pxtab[px];
          const int pp = tab >> 16, qq = tab & 0xFFFF;
          if (px >= tile_px || pp >= p_lim || qq >= q_lim) continue;
#pragma unroll
          for (int nt = 0; nt < 2; ++nt) {
            const int f = kt * kFiltersPerCta + warp * 16 + nt * 8 + 2 * t;
            if (f >= a.K) continue;
            store_pair(a, img, p0 + pp, q0 + qq, f, two_alpha[nt][0] * acc[nt][2 * half],
                       two_alpha[nt][1] * acc[nt][2 * half + 1]);
          }
        }
      }
    }
    if constexpr (kStaged) {
      // 5. staged tile -> y with 16-byte stores.  Thread tid always moves
      //    chunk c = tid % 16 (filters 8c .. 8c+7) of pixels tid / 16 + 16 i,
      //    so its swizzle phase (px & 15) is fixed.
      __syncthreads();
      const int k0 = kt * kFiltersPerCta;
      const int kchunks = (a.K - k0) < kFiltersPerCta ? (a.K - k0) / 8 : kFiltersPerCta / 8;
      const int c = tid & 15, pr = tid >> 4;
      if (c < kchunks) {
        const uint32_t soff = static_cast<uint32_t>(((c ^ pr) << 4));
        __nv_bfloat16* yb = static_cast<__nv_bfloat16*>(a.y) + k0 + 8 * c;
        const bool full_rows = a.TQ == a.Q;
        const size_t pix0 = (static_cast<size_t>(img) * a.P + p0) * a.Q + q0;
        const int valid_px = full_rows ? (p_lim < a.TP ? p_lim : a.TP) * a.TQ : tile_px;
        for (int px = pr; px < valid_px; px += kThreads / 16) {
          size_t pix = pix0 + px;
          if (!full_rows) {
            const int tab = pxtab[px];
            const int pp = tab >> 16, qq = tab & 0xFFFF;
            if (pp >= p_lim || qq >= q_lim) continue;
            pix = pix0 + static_cast<size_t>(pp) * a.Q + qq;
          }
          const uint4 v = *reinterpret_cast<const uint4*>(staging + px * 256 + soff);
          *reinterpret_cast<uint4*>(yb + pix * a.K) = v;
        }
      }
    }
  }
}


// ------------------------------------------------------ tensor-core variant
// NHWC bf16 activations and NHWC bf16 output without a residual (K % 8 == 0,
// 16-byte aligned y): the configuration the image networks launch.  The
// mma.sync loop above spends 64 m16n8k16 per warp and tile plus their
// fragment loads; here the whole tile's products are KP/16 tcgen05.mma
// issued by one thread.  A CTA takes a tile of up to 128 output pixels and
// 128 filters:
//   1. the patch goes to shared memory; its first batch of elements was
//      loaded into registers while the previous tile computed;
//   2. the threads build the im2col rows [pixel][64 codes] in the K-major,
//      128-byte-swizzled layout of a tcgen05 operand (codes past n zero);
//   3. one thread issues KP/16 tcgen05.mma, M = 128 filters (decoded codes
//      W~/2, same layout, built once per filter tile), N = the tile's pixels
//      rounded up to 16, fp32 accumulators in tensor memory, while the
//      others load the next tile's first patch batch;
//   4. eight warps read the accumulators as 16x256b fragments, apply
//      2 alpha and ReLU (in the bf16 conversion) and store them transposed
//      (stmatrix) into a staging tile [pixel][filter] (two halves of 64
//      filters, 16-byte chunks XOR-swizzled by the pixel);
//   5. two threads of different warps write the halves with TMA stores
//      (asynchronous: the copy-out overlaps the next tile; a cooperative
//      copy with 16-byte stores from every thread measured slower, and one
//      thread issuing both boxes waited about 0.5 us per tile).
// Three CTAs share an SM, so one CTA's loads overlap another's MMA and
// stores.
constexpr int kTcPixels = 128;
constexpr int kTcCtasPerSm = 3;
constexpr int kTcMaxPatchBytes = 8 * 1024;
constexpr int kTcTmemCols = 128;
constexpr int kTcOperandBytes = 128 * 128;   // 128 rows x 64 bf16 codes
constexpr uint64_t kTcWaitLimitNs = 1000000000ull;

size_t smalltap_tc_smem(size_t patch_bytes) {
  return 1024 /*alignment slack*/ + 4 * static_cast<size_t>(kTcOperandBytes) +
         ((patch_bytes + 15) & ~static_cast<size_t>(15)) + (kTcPixels + kMaxCodes) * sizeof(int) + 64;
}

// Tile t: filter tile slowest (a CTA keeps its decoded filters), then
// image, row block, column block.
struct TcTile {
  int kt, img, p0, q0;
};

__device__ __forceinline__ TcTile tc_tile(const SmallTapArgs& a, int tile) {
  TcTile c;
  const int per_k = a.N * a.tiles_p * a.tiles_q;
  c.kt = tile / per_k;
  int rest = tile - c.kt * per_k;
  c.img = rest / (a.tiles_p * a.tiles_q);
  rest -= c.img * (a.tiles_p * a.tiles_q);
  const int pt = rest / a.tiles_q;
  c.p0 = pt * a.TP;
  c.q0 = (rest - pt * a.tiles_q) * a.TQ;
  return c;
}

template <int KP>
__global__ void __launch_bounds__(kThreads, kTcCtasPerSm)
    conv_smalltap_tc_kernel(const __grid_constant__ CUtensorMap tmap_y, SmallTapArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* opA = smem;                                  // [128 filters][128 B]
  uint8_t* opB = smem + kTcOperandBytes;                // [128 pixels][128 B]
  uint8_t* stage = smem + 2 * kTcOperandBytes;          // 2 x [128 pixels][64 filters]
  __nv_bfloat16* patch = reinterpret_cast<__nv_bfloat16*>(smem + 4 * kTcOperandBytes);
  int* pxbase = reinterpret_cast<int*>(smem + 4 * kTcOperandBytes + a.patch_bytes);
  int* koff_tab = pxbase + kTcPixels;                   // patch offset of code k, -1 past n
  uint64_t* bar = reinterpret_cast<uint64_t*>(koff_tab + kMaxCodes);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bar + 1);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  constexpr int kChunks = KP / 8;   // 16-byte chunks of an im2col row that hold codes

  if (tid < kTcPixels) {
    const int pp = tid / a.TQ, qq = tid % a.TQ;
    pxbase[tid] = (pp * a.sh * a.PW + qq * a.sw) * a.C;
  }
  if (tid < kMaxCodes) {
    int off = -1;
    if (tid < a.n) {
      const int c = tid % a.C, s = (tid / a.C) % a.S, r = tid / (a.C * a.S);
      off = (r * a.PW + s) * a.C + c;
    }
    koff_tab[tid] = off;
  }
  const int my_ch = tid % kChunks;
  if (warp == 0) {
    tmem_alloc(tmem_slot, kTcTmemCols);
    tmem_relinquish();
  }
  if (tid == 0) {
    mbar_init(bar, 1);
    fence_mbar_init();
    prefetch_tmap(&tmap_y);
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t acc = *tmem_slot;
  int koff[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) koff[j] = koff_tab[my_ch * 8 + j];

  const int tile_px = a.TP * a.TQ;
  const int row_elems = a.PW * a.C, patch_elems = a.PH * row_elems;
  const int row_len = a.W * a.C;
  const int r_first = tid / row_elems, e_first = tid % row_elems;
  const int dr = kThreads / row_elems, de = kThreads % row_elems;
  const uint32_t idesc = idesc_bf16_f32(128, static_cast<uint32_t>(a.mma_n));
  const uint64_t adesc = smem_desc_sw128_kmajor(smem_addr(opA));
  const uint64_t bdesc = smem_desc_sw128_kmajor(smem_addr(opB));
  const uint32_t stage_s = smem_addr(stage);
  // epilogue role: TMEM lane quarter `sub` (filters 32 sub ..), pixel half
  const int sub = warp & 3, half = warp >> 2;
  const int fr = lane >> 2;
  const int mi = lane >> 3, mrow = lane & 7;
  const int nchunks = (a.mma_n + 31) / 32;
  const int c_begin = half ? (nchunks + 1) / 2 : 0;
  const int c_end = half ? nchunks : (nchunks + 1) / 2;
  float a2f[2][2] = {{0.f, 0.f}, {0.f, 0.f}};
  const bool relu = a.relu != 0;

  // The patch of a tile: element idx = r * row_elems + e (patch row r,
  // element e of that row) is image row ih0 + r, element e0 + e of the row.
  // A thread holds elements idx = tid + kThreads j; its (r, e) advance by the
  // constant (dr, de) per j.  The first eight (j < 8) of the next tile are
  // loaded into registers while the current tile computes.
  const uint16_t* xbase = reinterpret_cast<const uint16_t*>(a.x);
  auto load_batch = [&](int tile, int idx0, uint32_t (&v)[4]) {
    const TcTile c = tc_tile(a, tile);
    const int ih0 = c.p0 * a.sh - a.ph, e0 = (c.q0 * a.sw - a.pw) * a.C;
    const uint16_t* img_x = xbase + static_cast<size_t>(c.img) * a.H * row_len;
    int r = r_first, e = e_first;
    if (idx0 != tid) {
      r = idx0 / row_elems;
      e = idx0 - r * row_elems;
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int gh = ih0 + r, ge = e0 + e;
      const bool ok = idx0 + j * kThreads < patch_elems &&
                      static_cast<unsigned>(gh) < static_cast<unsigned>(a.H) &&
                      static_cast<unsigned>(ge) < static_cast<unsigned>(row_len);
      const uint32_t el = ok ? __ldg(img_x + gh * row_len + ge) : 0u;
      v[j >> 1] = (j & 1) ? (v[j >> 1] | (el << 16)) : el;
      r += dr;
      e += de;
      if (e >= row_elems) {
        e -= row_elems;
        ++r;
      }
    }
  };
  uint16_t* patch_u = reinterpret_cast<uint16_t*>(patch);

  grid_dependency_wait();   // activations may come from the previous kernel
  grid_dependents_launch();
  uint32_t pre[4];   // next tile's first eight patch elements, two per word
  if (static_cast<int>(blockIdx.x) < a.tiles) load_batch(blockIdx.x, tid, pre);
  int cur_ktile = -1;
  uint32_t tiles_done = 0;
  for (int tile = blockIdx.x; tile < a.tiles; tile += gridDim.x, ++tiles_done) {
    const TcTile tc = tc_tile(a, tile);
    const int kt = tc.kt;
    if (kt != cur_ktile) {
      cur_ktile = kt;
      // operand A: filter f's codes as bf16 W~/2, chunk c of row f at c ^ (f & 7)
      const int f = tid & 127;
      const int fg = kt * kFiltersPerCta + f;
      for (int ks = tid >> 7; ks < KP / 16; ks += 2) {
        const uint32_t w =
            (fg < a.K && ks < a.wpf) ? __ldg(a.codes + static_cast<size_t>(fg) * a.wpf + ks) : 0u;
        uint32_t o[8];
        word_to_bf16x2(w, o);
        uint8_t* row = opA + f * 128;
        *reinterpret_cast<uint4*>(row + (((2 * ks) ^ (f & 7)) << 4)) =
            make_uint4(o[0], o[1], o[2], o[3]);
        *reinterpret_cast<uint4*>(row + (((2 * ks + 1) ^ (f & 7)) << 4)) =
            make_uint4(o[4], o[5], o[6], o[7]);
      }
#pragma unroll
      for (int lg = 0; lg < 2; ++lg) {
#pragma unroll
        for (int u = 0; u < 2; ++u) {
          const int kk = kt * kFiltersPerCta + sub * 32 + lg * 16 + u * 8 + fr;
          a2f[lg][u] = kk < a.K ? 2.0f * __ldg(a.alpha + kk) : 0.0f;
        }
      }
    }
    // 1. input patch (zero outside the image): the prefetched first batch,
    //    then any further batches of a large patch
    auto store_batch = [&](int idx0, const uint32_t (&v)[4]) {
#pragma unroll
      for (int j = 0; j < 8; ++j)
        if (idx0 + j * kThreads < patch_elems)
          patch_u[idx0 + j * kThreads] = static_cast<uint16_t>(v[j >> 1] >> (16 * (j & 1)));
    };
    store_batch(tid, pre);
    for (int idx0 = tid + 8 * kThreads; idx0 - tid < patch_elems; idx0 += 8 * kThreads) {
      uint32_t v[4];
      load_batch(tile, idx0, v);
      store_batch(idx0, v);
    }
    __syncthreads();
    // 2. operand B: im2col rows, chunk c of pixel row px at c ^ (px & 7)
    for (int px = tid / kChunks; px < a.mma_n; px += kThreads / kChunks) {
      uint32_t v[4] = {0u, 0u, 0u, 0u};
      if (px < tile_px) {
        const uint16_t* src = patch_u + pxbase[px];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const uint32_t lo = koff[2 * i] >= 0 ? src[koff[2 * i]] : 0u;
          const uint32_t hi = koff[2 * i + 1] >= 0 ? src[koff[2 * i + 1]] : 0u;
          v[i] = lo | (hi << 16);
        }
      }
      *reinterpret_cast<uint4*>(opB + px * 128 + ((my_ch ^ (px & 7)) << 4)) =
          make_uint4(v[0], v[1], v[2], v[3]);
    }
    fence_proxy_async_smem();   // operands written here are read by the tensor core
    __syncthreads();
    if (tile + static_cast<int>(gridDim.x) < a.tiles) load_batch(tile + gridDim.x, tid, pre);
    // 3. MMA
    if (tid == 0) {
      tc_fence_after_sync();
#pragma unroll
      for (int kk = 0; kk < KP / 16; ++kk)
        tc_mma_ss(acc, adesc + static_cast<uint64_t>(2 * kk), bdesc + static_cast<uint64_t>(2 * kk),
                  idesc, kk > 0 ? 1u : 0u);
      tc_commit(bar);
    }
    // one thread waits for the accumulators, the two storing threads for
    // their previous stores to finish reading the staging tile; the others
    // park at the barrier
    if (tid == 0 || tid == 32) bulk_wait_group_read<0>();
    const bool ok = tid != 0 || mbar_wait(bar, tiles_done & 1u, nullptr, a.err, kTcWaitLimitNs);
    if (!__syncthreads_and(ok)) break;
    tc_fence_after_sync();
    // 4. epilogue: fragments (lane = filter, column = pixel) -> 2 alpha,
    //    ReLU, bf16 pairs -> transposed 8x8 stores into the staging tile
    for (int j = c_begin; j < c_end; ++j) {
      uint32_t v[2][16];
#pragma unroll
      for (int lg = 0; lg < 2; ++lg)
        tmem_ld_16x256b_x4(acc + (static_cast<uint32_t>(sub * 32 + lg * 16) << 16) +
                               static_cast<uint32_t>(32 * j),
                           v[lg]);
      tmem_wait_ld();
#pragma unroll
      for (int lg = 0; lg < 2; ++lg) {
        uint32_t pk[8];
#pragma unroll
        for (int b = 0; b < 4; ++b) {
          const float y0 = a2f[lg][0] * __uint_as_float(v[lg][4 * b + 0]);
          const float y1 = a2f[lg][0] * __uint_as_float(v[lg][4 * b + 1]);
          const float y2 = a2f[lg][1] * __uint_as_float(v[lg][4 * b + 2]);
          const float y3 = a2f[lg][1] * __uint_as_float(v[lg][4 * b + 3]);
          // filter fr, pixels 8b + 2(lane % 4) + 0/1; then filter fr + 8
          pk[2 * b] = relu ? pack_bf16x2_relu(y0, y1) : pack_bf16x2(y0, y1);
          pk[2 * b + 1] = relu ? pack_bf16x2_relu(y2, y3) : pack_bf16x2(y2, y3);
        }
#pragma unroll
        for (int bp = 0; bp < 2; ++bp) {
          const int px = 32 * j + 8 * (2 * bp + (mi >> 1)) + mrow;
          const int chunk = 4 * sub + 2 * lg + (mi & 1);   // 8-filter chunk 0..15
          const uint32_t addr = stage_s + static_cast<uint32_t>((chunk >> 3) * kTcOperandBytes +
                                                                px * 128 +
                                                                (((chunk & 7) ^ (px & 7)) << 4));
          stmatrix_x4_trans(addr, pk[4 * bp + 0], pk[4 * bp + 1], pk[4 * bp + 2], pk[4 * bp + 3]);
        }
      }
    }
    tc_fence_before_sync();
    fence_proxy_async_smem();   // staged values -> visible to the TMA stores
    __syncthreads();
    // 5. two TMA stores from threads of different warps (filters 0-63 from
    //    thread 0, 64-127 from thread 32): one issuing thread per box keeps
    //    the two boxes in flight together
    if (tid == 0 || (tid == 32 && kt * kFiltersPerCta + kFiltersPerCta / 2 < a.K)) {
      const int h = tid >> 5;
      tma_store_4d(&tmap_y, stage + h * kTcOperandBytes, kt * kFiltersPerCta + h * 64, tc.q0,
                   tc.p0, tc.img);
      bulk_commit_group();
    }
  }
  if (tid == 0 || tid == 32) bulk_wait_group<0>();   // stores complete before the CTA exits
  tc_fence_before_sync();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after_sync();
    tmem_dealloc(acc, kTcTmemCols);
  }
}

struct SmallTapPlan {
  int TP, TQ, PH, PW, KP;
  size_t smem;
};

bool smalltap_staged(const ConvProblem& p) {
  return p.layout != TBN_NCHW && p.ydt == TBN_BF16 && p.residual == nullptr && p.K % 8 == 0 &&
         is_aligned(p.y, 16);
}

size_t smalltap_smem(int KP, bool staged, size_t patch_bytes) {
  return static_cast<size_t>(kMaxTilePixels) * KP * 2 +
         (staged ? static_cast<size_t>(kMaxTilePixels) * kFiltersPerCta * 2 : 0) +
         2 * kMaxTilePixels * sizeof(int) + patch_bytes;
}

SmallTapPlan plan_smalltap(const ConvProblem& p) {
  SmallTapPlan t{};
  t.TQ = static_cast<int>(std::min<int64_t>(p.Q, kMaxTilePixels));
  t.TP = static_cast<int>(std::max<int64_t>(1, std::min<int64_t>(p.P, kMaxTilePixels / t.TQ)));
  const int64_t n = p.C * p.R * p.S;
  t.KP = n <= 32 ? 32 : 64;
  // fewer rows per tile while the patch does not fit its shared-memory budget
  for (;;) {
    t.PH = static_cast<int>((t.TP - 1) * p.sh + p.R);
    t.PW = static_cast<int>((t.TQ - 1) * p.sw + p.S);
    if (t.TP == 1 || static_cast<int64_t>(t.PH) * t.PW * p.C * 2 <= kMaxPatchBytes) break;
    --t.TP;
  }
  t.smem = smalltap_smem(t.KP, smalltap_staged(p), static_cast<size_t>(t.PH) * t.PW * p.C * 2);
  return t;
}


// Tile plan of the tensor-core variant: up to 128 pixels (whole rows when
// they fit), fewer rows while the patch exceeds its 8 KB budget.
struct SmallTapTcPlan {
  int TP, TQ, PH, PW, KP, mma_n;
  int patch_bytes;
  size_t smem;
  bool fits;
};

SmallTapTcPlan plan_smalltap_tc(const ConvProblem& p) {
  SmallTapTcPlan t{};
  t.TQ = static_cast<int>(std::min<int64_t>(p.Q, kTcPixels));
  t.TP = static_cast<int>(std::max<int64_t>(1, std::min<int64_t>(p.P, kTcPixels / t.TQ)));
  t.KP = p.C * p.R * p.S <= 32 ? 32 : 64;
  int64_t bytes = 0;
  for (;;) {
    t.PH = static_cast<int>((t.TP - 1) * p.sh + p.R);
    t.PW = static_cast<int>((t.TQ - 1) * p.sw + p.S);
    bytes = static_cast<int64_t>(t.PH) * t.PW * p.C * 2;
    if (t.TP == 1 || bytes <= kTcMaxPatchBytes) break;
    --t.TP;
  }
  t.fits = bytes <= kTcMaxPatchBytes;
  t.patch_bytes = static_cast<int>((bytes + 15) & ~int64_t(15));
  t.mma_n = (t.TP * t.TQ + 15) & ~15;
  t.smem = smalltap_tc_smem(static_cast<size_t>(t.patch_bytes));
  return t;
}

// The tensor-core variant takes NHWC bf16 output without a residual, stored
// by TMA (K % 8 == 0 for the 16-byte row pitch, 16-byte aligned y).
bool smalltap_tc_eligible(const ConvProblem& p) {
  return p.layout == TBN_NHWC && p.ydt == TBN_BF16 && p.residual == nullptr && p.K % 8 == 0 &&
         is_aligned(p.y, 16) && get_encode_tiled() != nullptr && plan_smalltap_tc(p).fits;
}

tbn_status launch_smalltap_tc(const ConvProblem& p, SmallTapArgs a, cudaStream_t s) {
  const SmallTapTcPlan t = plan_smalltap_tc(p);
  a.TP = t.TP; a.TQ = t.TQ; a.PH = t.PH; a.PW = t.PW;
  a.tiles_p = (a.P + a.TP - 1) / a.TP;
  a.tiles_q = (a.Q + a.TQ - 1) / a.TQ;
  const int64_t tiles = static_cast<int64_t>(a.N) * a.tiles_p * a.tiles_q * a.tiles_k;
  if (tiles >= (1ll << 31)) return fail(TBN_ERR_UNSUPPORTED, "small-tap conv: too many tiles");
  a.tiles = static_cast<int>(tiles);
  a.mma_n = t.mma_n;
  a.patch_bytes = t.patch_bytes;
  a.err = device_error_word();

  // output map: box = 64 filters (128 bytes, 128-byte swizzle) x TQ x TP x 1,
  // the layout of a staging half
  alignas(64) CUtensorMap tmap_y;
  std::memset(&tmap_y, 0, sizeof(tmap_y));
  const cuuint64_t gdim[4] = {(cuuint64_t)p.K, (cuuint64_t)p.Q, (cuuint64_t)p.P, (cuuint64_t)p.N};
  const cuuint64_t gstride[3] = {(cuuint64_t)(p.K * 2), (cuuint64_t)(p.Q * p.K * 2),
                                 (cuuint64_t)(p.P * p.Q * p.K * 2)};
  const cuuint32_t box[4] = {(cuuint32_t)(kFiltersPerCta / 2), (cuuint32_t)t.TQ,
                             (cuuint32_t)t.TP, 1u};
  const cuuint32_t estr[4] = {1u, 1u, 1u, 1u};
  const CUresult cr = get_encode_tiled()(
      &tmap_y, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, p.y, gdim, gstride, box, estr,
      CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
      CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (cr != CUDA_SUCCESS)
    return fail(TBN_ERR_CUDA, "small-tap conv: cuTensorMapEncodeTiled(y) failed (%d)", (int)cr);

  static std::once_flag attr_once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(attr_once, [] {
    const void* fns[2] = {(const void*)conv_smalltap_tc_kernel<32>,
                          (const void*)conv_smalltap_tc_kernel<64>};
    for (int i = 0; i < 2 && attr_err == cudaSuccess; ++i) {
      attr_err = cudaFuncSetAttribute(fns[i], cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      (int)smalltap_tc_smem(kTcMaxPatchBytes));
      if (attr_err == cudaSuccess)
        attr_err = cudaFuncSetAttribute(fns[i], cudaFuncAttributePreferredSharedMemoryCarveout, 100);
    }
  });
  if (attr_err != cudaSuccess) return cuda_fail(attr_err, "cudaFuncSetAttribute(smalltap tc)");

  const int64_t slots = static_cast<int64_t>(device_sm_count()) * kTcCtasPerSm;
  const int grid = static_cast<int>(std::min<int64_t>(tiles, slots));
  void (*kern)(const CUtensorMap, SmallTapArgs) =
      t.KP == 32 ? conv_smalltap_tc_kernel<32> : conv_smalltap_tc_kernel<64>;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(static_cast<unsigned>(grid));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = t.smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t le = cudaLaunchKernelEx(&cfg, kern, tmap_y, a);
  if (le != cudaSuccess) return cuda_fail(le, "cudaLaunchKernelEx(conv_smalltap_tc_kernel)");
  return check_launch("conv_smalltap_tc_kernel");
}
}  // namespace

const char* conv_smalltap_unsupported_reason(const ConvProblem& p) {
  if (p.xdt != TBN_BF16) return "small-tap conv needs bf16 activations";
  if (p.C * p.R * p.S > kMaxCodes) return "small-tap conv needs C*R*S <= 64";
  if (p.pool) return "small-tap conv has no fused pool";
  if (p.N >= (1ll << 31) / 4 || p.H * p.W >= (1ll << 30) || p.P * p.Q >= (1ll << 30))
    return "small-tap conv: tensor too large";
  const SmallTapPlan t = plan_smalltap(p);
  if (static_cast<int64_t>(t.PH) * t.PW * p.C * 2 > kMaxPatchBytes)
    return "small-tap conv: input patch exceeds shared memory";
  return "";
}

tbn_status launch_conv_smalltap(const ConvProblem& p, cudaStream_t s) {
  const SmallTapPlan t = plan_smalltap(p);
  SmallTapArgs a{};
  a.N = static_cast<int>(p.N); a.C = static_cast<int>(p.C); a.H = static_cast<int>(p.H);
  a.W = static_cast<int>(p.W); a.K = static_cast<int>(p.K); a.R = static_cast<int>(p.R);
  a.S = static_cast<int>(p.S); a.sh = static_cast<int>(p.sh); a.sw = static_cast<int>(p.sw);
  a.ph = static_cast<int>(p.ph); a.pw = static_cast<int>(p.pw); a.P = static_cast<int>(p.P);
  a.Q = static_cast<int>(p.Q);
  a.n = static_cast<int>(p.C * p.R * p.S);
  a.wpf = (a.n + 15) / 16;
  a.TP = t.TP; a.TQ = t.TQ; a.PH = t.PH; a.PW = t.PW;
  a.tiles_p = (a.P + a.TP - 1) / a.TP;
  a.tiles_q = (a.Q + a.TQ - 1) / a.TQ;
  a.tiles_k = (a.K + kFiltersPerCta - 1) / kFiltersPerCta;
  const int64_t tiles = static_cast<int64_t>(a.N) * a.tiles_p * a.tiles_q * a.tiles_k;
  if (tiles >= (1ll << 31)) return fail(TBN_ERR_UNSUPPORTED, "small-tap conv: too many tiles");
  a.tiles = static_cast<int>(tiles);
  a.x_nhwc = p.layout == TBN_NHWC ? 1 : 0;
  a.rsc = p.layout != TBN_NCHW ? 1 : 0;
  a.y_nhwc = p.layout != TBN_NCHW ? 1 : 0;
  a.y_bf16 = p.ydt == TBN_BF16 ? 1 : 0;
  a.relu = p.relu;
  a.x = static_cast<const __nv_bfloat16*>(p.x);
  a.codes = p.codes;
  a.alpha = p.alpha;
  a.y = p.y;
  a.residual = p.residual;
  if (smalltap_tc_eligible(p)) return launch_smalltap_tc(p, a, s);

  static std::once_flag attr_once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(attr_once, [] {
    const void* fns[4] = {(const void*)conv_smalltap_kernel<32, false>,
                          (const void*)conv_smalltap_kernel<32, true>,
                          (const void*)conv_smalltap_kernel<64, false>,
                          (const void*)conv_smalltap_kernel<64, true>};
    const int kps[4] = {32, 32, 64, 64};
    const bool st[4] = {false, true, false, true};
    for (int i = 0; i < 4 && attr_err == cudaSuccess; ++i) {
      attr_err = cudaFuncSetAttribute(fns[i], cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      (int)smalltap_smem(kps[i], st[i], kMaxPatchBytes));
      // the same shared-memory split as the network's other kernels: no
      // reconfiguration of the SMs between consecutive launches
      if (attr_err == cudaSuccess)
        attr_err = cudaFuncSetAttribute(fns[i], cudaFuncAttributePreferredSharedMemoryCarveout, 100);
    }
  });
  if (attr_err != cudaSuccess) return cuda_fail(attr_err, "cudaFuncSetAttribute(smalltap)");

  const int64_t slots = static_cast<int64_t>(device_sm_count()) * kCtasPerSm;
  const int grid = static_cast<int>(std::min<int64_t>(tiles, slots));
  const bool staged = smalltap_staged(p);
  void (*kern)(SmallTapArgs) = t.KP == 32 ? (staged ? conv_smalltap_kernel<32, true>
                                                    : conv_smalltap_kernel<32, false>)
                                          : (staged ? conv_smalltap_kernel<64, true>
                                                    : conv_smalltap_kernel<64, false>);
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(static_cast<unsigned>(grid));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = t.smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t le = cudaLaunchKernelEx(&cfg, kern, a);
  if (le != cudaSuccess) return cuda_fail(le, "cudaLaunchKernelEx(conv_smalltap_kernel)");
  return check_launch("conv_smalltap_kernel");
}

}  // namespace tbn
