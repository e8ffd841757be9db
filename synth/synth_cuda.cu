// synth_cuda.cu -- device build of the seeded synthetic-input generator.
// Same published Philox4x32-10 definition and the same value mapping as the
// host build (synth.c); the outputs are bit-identical.  This file fills caller
// buffers with test inputs only; it is not part of the verification library.
#include <cuda_runtime.h>
#include <stdint.h>

#include "synth.h"

namespace {

__device__ __forceinline__ void philox_round(uint32_t c[4], uint32_t k0,
                                             uint32_t k1) {
  const uint32_t m0 = 0xD2511F53u, m1 = 0xCD9E8D57u;
  uint32_t hi0 = __umulhi(m0, c[0]), lo0 = m0 * c[0];
  uint32_t hi1 = __umulhi(m1, c[2]), lo1 = m1 * c[2];
  uint32_t n0 = hi1 ^ c[1] ^ k0;
  uint32_t n2 = hi0 ^ c[3] ^ k1;
  c[0] = n0;
  c[1] = lo1;
  c[2] = n2;
  c[3] = lo0;
}

__device__ __forceinline__ void block_at(uint64_t seed, uint32_t stream,
                                         int64_t i, uint32_t c[4]) {
  c[0] = (uint32_t)(uint64_t)i;
  c[1] = (uint32_t)((uint64_t)i >> 32);
  c[2] = stream;
  c[3] = 0x5EEDu;
  uint32_t k0 = (uint32_t)seed, k1 = (uint32_t)(seed >> 32);
  philox_round(c, k0, k1);
#pragma unroll
  for (int r = 1; r < 10; ++r) {
    k0 += 0x9E3779B9u;
    k1 += 0xBB67AE85u;
    philox_round(c, k0, k1);
  }
}

__device__ __forceinline__ uint16_t f32_to_bf16_rne(float x) {
  uint32_t u = __float_as_uint(x);
  u += 0x7FFFu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

__global__ void fill_normal_bf16_kernel(uint16_t* __restrict__ dst, int64_t n,
                                        uint64_t seed, uint32_t stream,
                                        float scale, float base) {
  int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += stride) {
    uint32_t r[4];
    block_at(seed, stream, i, r);
    int32_t s = 0;
#pragma unroll
    for (int j = 0; j < 4; ++j) s += (int32_t)(r[j] & 0xFFFFu) + (int32_t)(r[j] >> 16);
    int32_t d = 2 * s - 8 * 65535;
    float v = __fmul_rn(__int2float_rn(d), scale);
    dst[i] = f32_to_bf16_rne(__fadd_rn(v, base));
  }
}

__global__ void fill_uniform_int_kernel(int32_t* __restrict__ dst, int64_t n,
                                        uint64_t seed, uint32_t stream,
                                        uint32_t range) {
  int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += stride) {
    uint32_t r[4];
    block_at(seed, stream, i, r);
    dst[i] = (int32_t)(__umulhi(r[0], range));
  }
}

// Candidate block for a benchmark step.  traj[j] is the target's greedy
// trajectory from the initial root (traj[0] = that root).  With m = len - len0
// tokens forwarded so far, the next block's candidates are traj[m+1 ..] for the
// first `ell` places, then a token that differs from the trajectory, then the
// pre-drawn tail tokens.  plan = {ell, corrupt_token, tail[0..k-1]}.
__global__ void build_candidates_kernel(int32_t* __restrict__ cand,
                                        const int32_t* __restrict__ traj,
                                        int32_t traj_len,
                                        const int32_t* __restrict__ len_dev,
                                        int32_t len0,
                                        const int32_t* __restrict__ plan,
                                        int32_t k, int32_t vocab) {
  int i = threadIdx.x;
  if (i >= k) return;
  int32_t m = len_dev[0] - len0;
  int32_t ell = plan[0];
  int32_t j = m + 1 + i;
  int32_t want = (j >= 0 && j < traj_len) ? traj[j] : -1;
  int32_t tok;
  if (i < ell && want >= 0) {
    tok = want;
  } else if (i == ell) {
    tok = plan[1];
    if (tok == want) tok = (tok + 1) % vocab;
  } else {
    tok = plan[2 + i];
  }
  cand[i] = tok;
}

int grid_for(int64_t n) {
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  int64_t want = (n + 255) / 256;
  int64_t cap = (int64_t)sms * 8;
  return (int)(want < cap ? (want > 0 ? want : 1) : cap);
}

}  // namespace

extern "C" int synth_cuda_fill_normal_bf16(void* dst, int64_t n, uint64_t seed,
                                           uint32_t stream, float scale,
                                           float base, void* stream_handle) {
  if (n <= 0) return 0;
  fill_normal_bf16_kernel<<<grid_for(n), 256, 0, (cudaStream_t)stream_handle>>>(
      (uint16_t*)dst, n, seed, stream, scale, base);
  return (int)cudaGetLastError();
}

extern "C" int synth_cuda_build_candidates(void* cand, const void* traj,
                                           int32_t traj_len,
                                           const void* len_dev, int32_t len0,
                                           const void* plan, int32_t k,
                                           int32_t vocab, void* stream_handle) {
  if (k <= 0) return 0;
  if (k > 1024) return (int)cudaErrorInvalidValue;
  build_candidates_kernel<<<1, k, 0, (cudaStream_t)stream_handle>>>(
      (int32_t*)cand, (const int32_t*)traj, traj_len, (const int32_t*)len_dev,
      len0, (const int32_t*)plan, k, vocab);
  return (int)cudaGetLastError();
}

extern "C" int synth_cuda_fill_uniform_int(void* dst, int64_t n, uint64_t seed,
                                           uint32_t stream, uint32_t range,
                                           void* stream_handle) {
  if (n <= 0) return 0;
  fill_uniform_int_kernel<<<grid_for(n), 256, 0, (cudaStream_t)stream_handle>>>(
      (int32_t*)dst, n, seed, stream, range);
  return (int)cudaGetLastError();
}
