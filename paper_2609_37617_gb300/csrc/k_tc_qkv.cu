// k_tc_qkv.cu -- instantiates the tensor-core GEMM for the QKV projection
// (split-K partial sums, finished by qkv_finish_kernel).
#include "gemm_tc.cuh"

namespace as2d {

cudaError_t tc_gemm_part(int nb, const CUtensorMap& x, const TcParams& p, cudaStream_t st) {
  return tc_gemm_dispatch<TC_PART>(nb, x, p, st);
}

}  // namespace as2d
