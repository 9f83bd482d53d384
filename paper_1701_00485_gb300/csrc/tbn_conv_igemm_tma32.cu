// tbn_conv_igemm_tma32.cu -- the 32-channel TMA variants of the implicit-GEMM
// convolution kernel (every pool width and epilogue store, with and without
// the fused quantization prologue), compiled apart from the host dispatch.
#include "tbn_conv_igemm.cuh"

namespace tbn {

tbn_status launch_igemm_tma32(const ConvProblem& p, const TilePlan& t, IgArgs& a, int pw,
                              bool tma_store, bool fuse, cudaStream_t s) {
  if (fuse)
    return tma_store ? launch_pool<kModeTma32, true, true>(p, t, a, pw, s)
                     : launch_pool<kModeTma32, false, true>(p, t, a, pw, s);
  return tma_store ? launch_pool<kModeTma32, true, false>(p, t, a, pw, s)
                   : launch_pool<kModeTma32, false, false>(p, t, a, pw, s);
}

}  // namespace tbn
