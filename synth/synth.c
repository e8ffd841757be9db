/*
 * synth.c -- host build of the seeded synthetic-input generator (synth.h).
 * Philox4x32-10 written from its published definition (Salmon et al., SC 2011):
 * ten rounds of two 32x32->64 multiplies with the multipliers 0xD2511F53 and
 * 0xCD9E8D57, the key bumped by the Weyl constants 0x9E3779B9 / 0xBB67AE85
 * between rounds.
 */
#include "synth.h"

#include <math.h>
#include <string.h>

#define PHILOX_M0 0xD2511F53u
#define PHILOX_M1 0xCD9E8D57u
#define PHILOX_W0 0x9E3779B9u
#define PHILOX_W1 0xBB67AE85u

static inline void philox_round(uint32_t c[4], const uint32_t k[2]) {
  uint64_t p0 = (uint64_t)PHILOX_M0 * (uint64_t)c[0];
  uint64_t p1 = (uint64_t)PHILOX_M1 * (uint64_t)c[2];
  uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
  uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
  uint32_t n0 = hi1 ^ c[1] ^ k[0];
  uint32_t n2 = hi0 ^ c[3] ^ k[1];
  c[0] = n0;
  c[1] = lo1;
  c[2] = n2;
  c[3] = lo0;
}

void synth_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2],
                         uint32_t out[4]) {
  uint32_t c[4] = {ctr[0], ctr[1], ctr[2], ctr[3]};
  uint32_t k[2] = {key[0], key[1]};
  philox_round(c, k);
  for (int r = 1; r < 10; ++r) {
    k[0] += PHILOX_W0;
    k[1] += PHILOX_W1;
    philox_round(c, k);
  }
  memcpy(out, c, sizeof(c));
}

float synth_normal_scale(double sigma) {
  double var_s = 8.0 * (65536.0 * 65536.0 - 1.0) / 12.0;
  return (float)(sigma / (2.0 * sqrt(var_s)));
}

static inline void block_at(uint64_t seed, uint32_t stream, int64_t i,
                            uint32_t out[4]) {
  uint32_t ctr[4] = {(uint32_t)(uint64_t)i, (uint32_t)((uint64_t)i >> 32),
                     stream, 0x5EEDu};
  uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
  synth_philox4x32_10(ctr, key, out);
}

/* Centred Irwin-Hall integer: 2*sum(eight 16-bit halves) - 8*65535. */
static inline int32_t centred_sum(const uint32_t r[4]) {
  int32_t s = 0;
  for (int j = 0; j < 4; ++j) s += (int32_t)(r[j] & 0xFFFFu) + (int32_t)(r[j] >> 16);
  return 2 * s - 8 * 65535;
}

static inline uint16_t f32_to_bf16_rne(float x) {
  uint32_t u;
  memcpy(&u, &x, 4);
  u += 0x7FFFu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

void synth_fill_normal_bf16_offset(uint16_t* dst, int64_t n, uint64_t seed,
                                   uint32_t stream, float scale, float base) {
#pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < n; ++i) {
    uint32_t r[4];
    block_at(seed, stream, i, r);
    volatile float v = (float)centred_sum(r) * scale; /* one rounding */
    float x = v + base;                                /* exact when base = 0 */
    dst[i] = f32_to_bf16_rne(x);
  }
}

void synth_fill_normal_bf16(uint16_t* dst, int64_t n, uint64_t seed,
                            uint32_t stream, float scale) {
  synth_fill_normal_bf16_offset(dst, n, seed, stream, scale, 0.0f);
}

void synth_fill_uniform_int(int32_t* dst, int64_t n, uint64_t seed,
                            uint32_t stream, uint32_t range) {
#pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < n; ++i) {
    uint32_t r[4];
    block_at(seed, stream, i, r);
    dst[i] = (int32_t)(((uint64_t)r[0] * (uint64_t)range) >> 32);
  }
}
