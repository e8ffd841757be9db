// k_tc_logits.cu -- instantiates the tensor-core GEMM with the logits epilogue.
#include "gemm_tc.cuh"

namespace as2d {

cudaError_t tc_gemm_logits(int nb, const CUtensorMap& x, const TcParams& p,
                          cudaStream_t st) {
  return tc_gemm_dispatch<TC_LOGITS>(nb, x, p, st);
}

}  // namespace as2d
