// k_tc_swiglu.cu -- instantiates the tensor-core GEMM with the swiglu epilogue.
#include "gemm_tc.cuh"

namespace as2d {

cudaError_t tc_gemm_swiglu(int nb, const CUtensorMap& x, const TcParams& p,
                          cudaStream_t st) {
  return tc_gemm_dispatch<TC_SWIGLU>(nb, x, p, st);
}

}  // namespace as2d
