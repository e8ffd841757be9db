// k_tc_qkv.cu -- instantiates the tensor-core GEMM with the qkv epilogue.
#include "gemm_tc.cuh"

namespace as2d {

cudaError_t tc_gemm_qkv(int nb, const CUtensorMap& x, const TcParams& p,
                          cudaStream_t st) {
  return tc_gemm_dispatch<TC_QKV>(nb, x, p, st);
}

cudaError_t tc_gemm_part(int nb, const CUtensorMap& x, const TcParams& p, cudaStream_t st) {
  return tc_gemm_dispatch<TC_PART>(nb, x, p, st);
}

}  // namespace as2d
