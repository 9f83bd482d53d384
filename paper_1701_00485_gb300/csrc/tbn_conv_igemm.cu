// tbn_conv_igemm.cu -- host dispatch of the tcgen05 implicit-GEMM two-bit
// convolution (Eq. 1, Section 2): the tile plan, the split of K for
// 1x1 layers, the space-to-depth form of a strided first layer, fused
// quantization, and the gathering modes' kernel variants.  The kernel and
// its design are in tbn_conv_igemm.cuh.
#include "tbn_conv_igemm.cuh"

namespace tbn {
namespace {

// Split K: y = 2 alpha[k] * (sum of the K ranges' partial sums, in range
// order) (+ residual), ReLU, rounded to y's dtype.  Deterministic.  Four
// consecutive outputs per thread (K % 4 == 0: 16-byte partial loads).
template <bool kVec>
__global__ void __launch_bounds__(256) splitk_reduce_kernel(const float* __restrict__ partial,
                                                           int S, int64_t mk, int K,
                                                           const float* __restrict__ alpha,
                                                           const void* residual, int relu,
                                                           void* y, int y_bf16) {
  constexpr int kV = kVec ? 4 : 1;
  const int64_t n = mk / kV;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    float acc[kV];
    if constexpr (kVec) {
      float4 t = __ldg(reinterpret_cast<const float4*>(partial) + i);
      for (int s = 1; s < S; ++s) {
        const float4 u = __ldg(reinterpret_cast<const float4*>(partial + s * mk) + i);
        t.x += u.x; t.y += u.y; t.z += u.z; t.w += u.w;
      }
      acc[0] = t.x; acc[1] = t.y; acc[2] = t.z; acc[3] = t.w;
    } else {
      acc[0] = 0.0f;
      for (int s = 0; s < S; ++s) acc[0] += __ldg(partial + s * mk + i);
    }
    const int64_t o = i * kV;
    const int k0 = static_cast<int>(o % K);
#pragma unroll
    for (int e = 0; e < kV; ++e) {
      float v = 2.0f * __ldg(alpha + k0 + e) * acc[e];
      if (y_bf16) {
        if (residual) v += __bfloat162float(static_cast<const __nv_bfloat16*>(residual)[o + e]);
        if (relu) v = fmaxf(v, 0.0f);
        static_cast<__nv_bfloat16*>(y)[o + e] = __float2bfloat16_rn(v);
      } else {
        if (residual) v += static_cast<const float*>(residual)[o + e];
        if (relu) v = fmaxf(v, 0.0f);
        static_cast<float*>(y)[o + e] = v;
      }
    }
  }
}

// Patch mode (gathered activations staged per tile in shared memory) when a
// tile is whole output rows of one image, the filter spans at most
// kPatchMaxKBlocks K blocks and two patches fit beside the ring.
int patch_cap_bytes(const ConvProblem& p, const TilePlan& t) {
  if (use_tma(p) || t.tiles_q != 1 || t.bn != 1) return 0;
  const int64_t kblocks = (p.C * p.R * p.S + kBK - 1) / kBK;
  if (kblocks > kPatchMaxKBlocks) return 0;
  const int64_t rows = static_cast<int64_t>(t.bh - 1) * p.sh + p.R;
  const int64_t elems = rows * (p.W + 2 * p.pw) * p.C;
  const int64_t cap = ((2 * elems + 32) + 15) / 16 * 16;
  if (cap > (int64_t(1) << 20)) return 0;
  if (smem_bytes_for(kModePatch, static_cast<size_t>(cap), static_cast<int>(kblocks)) >
      static_cast<size_t>(kSmemLimit))
    return 0;
  return static_cast<int>(cap);
}

}  // namespace

bool conv_igemm_uses_tma(const ConvProblem& p) { return use_tma(p); }

// Split K when the output tiles fill fewer than half the SMs and the filter
// has at least 8 K blocks.  The tensor core's time per K block is
// proportional to the tile's pixels, but a CTA's time per K block is not
// (measured: it barely moves between 32 and 256 pixels; the operand supply
// sets it), so idle SMs are filled with K ranges of full-width tiles rather
// than with narrower tiles.
int conv_igemm_splitk(const ConvProblem& p, size_t* workspace_bytes) {
  *workspace_bytes = 0;
  // fully-connected shapes only (a 1x1 convolution over a 1x1 image): a
  // tile's pixel i is then image n0 + i, and the partial sums are stored
  // without the pixel walk of a general tile
  if (!use_tma(p) || p.pool || p.P != 1 || p.Q != 1 || p.R != 1 || p.S != 1) return 1;
  const TilePlan t = plan_tiles(p);
  const int64_t base = static_cast<int64_t>(t.tiles_q) * t.tiles_p * t.tiles_n *
                       ((p.K + kBM - 1) / kBM);
  const int64_t kblocks = (p.C * p.R * p.S + kBK - 1) / kBK;
  const int sms = device_sm_count();
  if (2 * base > sms || kblocks < 8) return 1;
  int64_t S = std::min<int64_t>(sms / base, kblocks / 4);
  if (S < 2) return 1;
  const int64_t per = (kblocks + S - 1) / S;
  S = (kblocks + per - 1) / per;
  *workspace_bytes = static_cast<size_t>(S) * p.N * p.P * p.Q * p.K * 4;
  return static_cast<int>(S);
}

// The stride-1 convolution over the space-to-depth input that a
// TBN_S2D_NHWC problem runs as.
ConvProblem s2d_problem(const ConvProblem& p) {
  const S2dGeom g = s2d_geom(p.R, p.S, p.sh, p.P, p.Q);
  ConvProblem q = p;
  q.layout = TBN_NHWC;
  q.C = kS2dChannels;
  q.H = g.Hs;
  q.W = g.Ws;
  q.R = g.Rp;
  q.S = g.Sp;
  q.sh = q.sw = 1;
  q.ph = q.pw = 0;
  return q;
}

const char* s2d_unsupported_reason(const ConvProblem& p) {
  if (p.xdt != TBN_BF16) return "space-to-depth input must be bf16";
  if (p.sh != p.sw || p.sh < 2) return "space-to-depth needs equal strides >= 2";
  if (p.sh * p.sh * p.C > kS2dChannels) return "space-to-depth needs stride^2 * C <= 64";
  if (p.K > kBM) return "space-to-depth keeps one filter block (K <= 128) resident";
  if (p.pool || p.residual) return "space-to-depth takes no pool and no residual";
  if (p.ksplit > 1) return "space-to-depth takes no split K";
  const ConvProblem q = s2d_problem(p);
  const int64_t kb = q.R * q.S;
  if (kb > kMaxResidentKB || plan_tiles(q).tile_n + 32 * kb > kTmemCols)
    return "space-to-depth: the filter's K blocks do not fit in tensor memory beside the tile";
  return "";
}

const char* conv_igemm_unsupported_reason(const ConvProblem& p) {
  if (p.layout == TBN_S2D_NHWC) {
    const char* r = s2d_unsupported_reason(p);
    if (*r) return r;
    return conv_igemm_unsupported_reason(s2d_problem(p));
  }
  if (p.layout != TBN_NHWC) return "implicit GEMM needs NHWC";
  if (p.xdt != TBN_BF16) return "implicit GEMM needs bf16 activations";
  if (!is_aligned(p.x, 16)) return "implicit GEMM needs 16-byte aligned x";
  if (p.pool && p.residual) return "pooling with a residual is not supported";
  if (p.N > (1 << 30) || p.H > (1 << 30) || p.W > (1 << 30) || p.K > (1 << 30))
    return "dimension too large";
  if (p.C * p.R * p.S >= (int64_t(1) << 30)) return "filter too large";
  if (p.H * p.W * p.C >= (int64_t(1) << 31)) return "image too large";
  if (p.R >= (1 << 15) || p.S >= (1 << 15)) return "kernel too large";
  if (use_tma(p) && (p.ph > p.R || p.pw > p.S)) return "implicit GEMM needs pad <= kernel extent";
  if (p.pool && pool_width(p, plan_tiles(p)) < 0)
    return "fused pool needs whole output rows of width 8, 16 or 32 per tile";
  int dev = 0, major = 0, minor = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return "no CUDA device";
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
  if (major != 10 || minor != 3) return "implicit GEMM kernel is built for sm_103a only";
  if ((use_tma(p) || use_tma_store(p)) && get_encode_tiled() == nullptr)
    return "cuTensorMapEncodeTiled unavailable";
  return "";
}

tbn_status launch_conv_igemm(const ConvProblem& p0, cudaStream_t s) {
  const bool s2d = p0.layout == TBN_S2D_NHWC;
  const ConvProblem p = s2d ? s2d_problem(p0) : p0;
  const TilePlan t = plan_tiles(p);
  IgArgs a{};
  a.N = (int)p.N; a.C = (int)p.C; a.H = (int)p.H; a.W = (int)p.W; a.K = (int)p.K;
  a.R = (int)p.R; a.S = (int)p.S; a.sh = (int)p.sh; a.sw = (int)p.sw;
  a.ph = (int)p.ph; a.pw = (int)p.pw; a.P = (int)p.P; a.Q = (int)p.Q;
  a.bw = t.bw; a.bh = t.bh; a.bn = t.bn; a.tile_n = t.tile_n;
  a.tiles_q = t.tiles_q; a.tiles_p = t.tiles_p;
  a.tiles_k = ceil_div(p.K, kBM);
  const int64_t tiles = static_cast<int64_t>(t.tiles_q) * t.tiles_p * t.tiles_n * a.tiles_k;
  a.ncodes = (int)(p.C * p.R * p.S);
  a.kblocks = ceil_div(a.ncodes, kBK);
  const bool split = p.ksplit > 1 && p.partial != nullptr;
  a.ksplit = split ? p.ksplit : 1;
  a.kb_per = ceil_div(a.kblocks, a.ksplit);
  if (split && (!use_tma(p) || p.pool || p.P != 1 || p.Q != 1 || p.R != 1 || p.S != 1 ||
                (a.ksplit - 1) * a.kb_per >= a.kblocks))
    return fail(TBN_ERR_INVALID_ARG, "implicit GEMM: bad split-K request");
  if (tiles * a.ksplit > 0x7fffffffLL) return fail(TBN_ERR_UNSUPPORTED, "implicit GEMM: too many tiles");
  a.base_tiles = static_cast<int>(tiles);
  a.tiles = static_cast<int>(tiles * a.ksplit);
  a.partial = split ? p.partial : nullptr;
  a.wpf = (a.ncodes + 15) / 16;
  if (s2d) {
    // codes of the original (r, s, c) filter
    a.wpf = static_cast<int>((p0.C * p0.R * p0.S + 15) / 16);
    a.s2d_s = static_cast<int>(p0.sh);
    a.s2d_C = static_cast<int>(p0.C);
    a.s2d_R = static_cast<int>(p0.R);
    a.s2d_S = static_cast<int>(p0.S);
    if (split || a.tiles_k != 1 || a.kblocks > kMaxResidentKB ||
        t.tile_n + 32 * a.kblocks > kTmemCols || p.pool || p.residual)
      return fail(TBN_ERR_UNSUPPORTED, "implicit GEMM: space-to-depth problem out of range");
  }
  // tiles of at most 176 pixels: two accumulators, so each tile's MMAs
  // overlap the previous tile's epilogue (space-to-depth mode keeps its
  // resident K blocks where the second accumulator would be)
  a.acc2 = (!s2d && t.tile_n <= kAcc2Cols) ? 1 : 0;
  a.x = static_cast<const __nv_bfloat16*>(p.x);
  a.codes = p.codes; a.alpha = p.alpha; a.y = p.y; a.residual = p.residual;
  if (p0.wq != nullptr) {
    if (s2d || split || !use_tma(p) || a.wpf > 2048 || p0.gbar == nullptr)
      return fail(TBN_ERR_UNSUPPORTED,
                  "implicit GEMM: fused quantization needs TMA activations (C %% 32 == 0, "
                  "stride <= 2), at most 2048 words per filter and no split of K");
    a.wq = p0.wq;
    a.codes_w = const_cast<uint32_t*>(p0.codes);
    a.alpha_w = const_cast<float*>(p0.alpha);
    a.gbar = p0.gbar;
    a.wq_vec = (is_aligned(p0.wq, 16) && a.ncodes % 4 == 0) ? 1 : 0;
  }
  a.relu = p.relu; a.y_bf16 = p.ydt == TBN_BF16 ? 1 : 0;
  a.err = device_error_word();
  const int pw = pool_width(p, t);
  const bool tst = use_tma_store(p) && !split;   // partial sums: direct fp32 stores
  if (split) {
    // the K ranges' partial sums, then their ordered sum with the epilogue
    const tbn_status st = use_ch32(p) ? launch_igemm_tma32(p, t, a, pw, false, false, s)
                                      : launch_igemm_tma64(p, t, a, pw, false, false, s);
    if (st != TBN_OK) return st;
    const int64_t mk = p.N * p.P * p.Q * p.K;
    const bool vec = p.K % 4 == 0 && is_aligned(p.partial, 16);
    const int64_t items = vec ? mk / 4 : mk;
    const int64_t blocks = std::min<int64_t>((items + 255) / 256, int64_t(device_sm_count()) * 16);
    if (vec)
      splitk_reduce_kernel<true><<<static_cast<unsigned>(blocks), 256, 0, s>>>(
          p.partial, a.ksplit, mk, (int)p.K, p.alpha, p.residual, p.relu, p.y,
          p.ydt == TBN_BF16 ? 1 : 0);
    else
      splitk_reduce_kernel<false><<<static_cast<unsigned>(blocks), 256, 0, s>>>(
          p.partial, a.ksplit, mk, (int)p.K, p.alpha, p.residual, p.relu, p.y,
          p.ydt == TBN_BF16 ? 1 : 0);
    return check_launch("splitk_reduce_kernel");
  }
  if (s2d) {
    return tst ? launch_t<kModeS2d, 0, true, false>(p, t, a, s)
               : launch_t<kModeS2d, 0, false, false>(p, t, a, s);
  }
  if (use_tma(p) && use_ch32(p)) {
    return launch_igemm_tma32(p, t, a, pw, tst, a.wq != nullptr, s);
  }
  if (use_tma(p)) {
    return launch_igemm_tma64(p, t, a, pw, tst, a.wq != nullptr, s);
  }
  const int cap = patch_cap_bytes(p, t);
  if (cap > 0) {
    a.PR = (t.bh - 1) * a.sh + a.R;
    a.PW = a.W + 2 * a.pw;
    a.patch_cap = cap;
    a.patch_bulk = a.pw == 0 ? 1 : 0;
    a.x_bytes = static_cast<long long>(p.N) * p.H * p.W * p.C * 2;
    return tst ? launch_pool<kModePatch, true, false>(p, t, a, pw, s)
               : launch_pool<kModePatch, false, false>(p, t, a, pw, s);
  }
  return tst ? launch_pool<kModeGather, true, false>(p, t, a, pw, s)
             : launch_pool<kModeGather, false, false>(p, t, a, pw, s);
}

}  // namespace tbn
