/*
 * synth.h -- seeded synthetic inputs shared by the oracle and the CUDA path.
 *
 * This module draws the random-init weights, the prefilled KV caches and the
 * token ids that both sides consume.  It holds none of the verification
 * method's arithmetic: no norm, no projection, no attention, no argmax.
 *
 * Every value is a pure function of (seed, stream, index) through the
 * counter-based generator Philox4x32-10 (Salmon, Moraes, Dror and Shaw,
 * "Parallel random numbers: as easy as 1, 2, 3", SC 2011).  The host build
 * (synth.c) and the device build (synth_cuda.cu) implement the same
 * published definition and produce bit-identical bf16 values, so a tensor
 * can be generated on the device for speed and on the host for the oracle.
 *
 * Normal draws: N(0, sigma) is approximated by the standardised sum of the
 * eight 16-bit halves of one Philox output block (Irwin-Hall, n = 8).  The sum
 * is an exact integer; the single fp32 multiply by `scale` (see
 * synth_normal_scale) is the only rounding, and the bf16 conversion is
 * round-to-nearest-even on the bits, so both builds agree exactly.
 */
#ifndef AS2D_SYNTH_H
#define AS2D_SYNTH_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* One Philox4x32-10 block: out = philox(ctr, key). */
void synth_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2],
                         uint32_t out[4]);

/* fp32 multiplier that maps the centred Irwin-Hall integer to N(0, sigma).
   Computed in double and rounded once to float; pass the same float to the
   host and the device fillers. */
float synth_normal_scale(double sigma);

/* dst[i] = bf16(normal(seed, stream, i)) for i in [0, n).  Host, OpenMP. */
void synth_fill_normal_bf16(uint16_t* dst, int64_t n, uint64_t seed,
                            uint32_t stream, float scale);

/* dst[i] = bf16(base + normal(seed, stream, i)) (gains around `base`). */
void synth_fill_normal_bf16_offset(uint16_t* dst, int64_t n, uint64_t seed,
                                   uint32_t stream, float scale, float base);

/* dst[i] = floor(u32(seed, stream, i) * range / 2^32), uniform in [0, range). */
void synth_fill_uniform_int(int32_t* dst, int64_t n, uint64_t seed,
                            uint32_t stream, uint32_t range);

/* Device fillers (synth_cuda.cu).  dst is a device pointer; `stream_handle`
   is a cudaStream_t (NULL = legacy default stream).  Return 0 on success,
   otherwise the cudaError_t of the launch. */
int synth_cuda_fill_normal_bf16(void* dst, int64_t n, uint64_t seed,
                                uint32_t stream, float scale, float base,
                                void* stream_handle);
int synth_cuda_fill_uniform_int(void* dst, int64_t n, uint64_t seed,
                                uint32_t stream, uint32_t range,
                                void* stream_handle);

/* Benchmark candidate block (device): see synth_cuda.cu. */
int synth_cuda_build_candidates(void* cand, const void* traj, int32_t traj_len,
                                const void* len_dev, int32_t len0,
                                const void* plan, int32_t k, int32_t vocab,
                                void* stream_handle);

#ifdef __cplusplus
}
#endif
#endif
