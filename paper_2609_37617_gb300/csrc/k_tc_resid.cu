// k_tc_resid.cu -- instantiates the tensor-core GEMM with the resid epilogue.
#include "gemm_tc.cuh"

namespace as2d {

cudaError_t tc_gemm_resid(int nb, const CUtensorMap& x, const TcParams& p,
                          cudaStream_t st) {
  return tc_gemm_dispatch<TC_RESID>(nb, x, p, st);
}

}  // namespace as2d
