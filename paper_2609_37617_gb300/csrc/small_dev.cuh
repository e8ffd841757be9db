// small_dev.cuh -- device functions of the embedding gather and the accept
// scan, shared by the standalone kernels (k_basic.cu) and the persistent
// verification kernel (k_mk.cu), so both paths compute bit for bit alike.
#pragma once

#include "as2d_internal.h"

namespace as2d {

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
  return v;  // identical in every lane: each butterfly step is commutative
}

// Residual stream row r = the embedding row e; the first projection's operand
// h * g0 as bf16 hi + lo parts (lo rows start at ss_ld, the rows allocated);
// the row's sum of squares in tile slot 0 of ss (slots 1.. = 0).  Run by nthr
// threads (128 in every caller, which fixes the summation order); red holds
// nthr / 32 floats of shared memory; bar_id is the group's barrier.
__device__ __forceinline__ void embed_row_body(const bf16* __restrict__ e,
                                               const float* __restrict__ g0, int H, int r,
                                               int ss_ld, float* __restrict__ h,
                                               bf16* __restrict__ xn, float* __restrict__ ss,
                                               int tid, int nthr, float* red, int bar_id) {
  float sq = 0.f;
  for (int c = tid; c < H; c += nthr) {
    const float x = __bfloat162float(e[c]);
    h[(size_t)r * H + c] = x;
    const float xv = x * g0[c];
    const bf16 xh = __float2bfloat16_rn(xv);
    xn[(size_t)r * H + c] = xh;
    xn[(size_t)(ss_ld + r) * H + c] = __float2bfloat16_rn(xv - __bfloat162float(xh));
    sq = fmaf(x, x, sq);
  }
  sq = warp_sum(sq);
  if ((tid & 31) == 0) red[tid >> 5] = sq;
  asm volatile("bar.sync %0, %1;" ::"r"(bar_id), "r"(nthr) : "memory");
  const int nt = H / 128;
  for (int t = tid; t < nt; t += nthr) {
    float tot = 0.f;
    if (t == 0)
      for (int w = 0; w < nthr / 32; ++w) tot += red[w];
    ss[(size_t)t * ss_ld + r] = tot;
  }
  asm volatile("bar.sync %0, %1;" ::"r"(bar_id), "r"(nthr) : "memory");
}

struct AcceptArgs {
  RowMap rm;
  const int32_t* cand;
  unsigned long long* best;
  int32_t* len;
  int32_t* root;
  int32_t* bad;
  int32_t* n_out;
  int32_t* corr_out;
  int32_t* greedy_out;
  int32_t force;  // 1: every row is kept whatever the greedy tokens (prefill)
};

// Accept scan of request b by one warp (App. C.2): g_i from the packed maxima,
// the number of leading candidates equal to the greedy tokens by ballot, the
// correction by shuffle, then L += n + 1 and root = correction.
__device__ __forceinline__ void accept_request(const AcceptArgs& a, int b, int lane) {
  const RowMap& m = a.rm;
  const int r0 = m.start[b];
  const int k = m.start[b + 1] - r0 - 1;
  if (a.force) {
    // every row kept (prefill, up to kPrefillRows rows): the maxima cleared
    // 32 rows at a time, the root is the greedy token after the last row
    int g_last = 0;
    for (int i = lane; i <= k; i += 32) {
      const unsigned long long v = a.best[r0 + i];
      const int g = (int)(0xFFFFFFFFu - (uint32_t)(v & 0xFFFFFFFFull));
      a.best[r0 + i] = 0ull;
      if (a.greedy_out) a.greedy_out[r0 + i] = g;
      if (i == k) g_last = g;
    }
    g_last = __shfl_sync(0xFFFFFFFFu, g_last, k & 31);
    if (lane == 0) {
      if (a.bad[b]) {
        a.n_out[b] = -1;
        a.corr_out[b] = -1;
        a.bad[b] = 0;
      } else {
        a.n_out[b] = k;
        a.corr_out[b] = g_last;
        a.len[b] += k + 1;
        a.root[b] = g_last;
      }
    }
    return;
  }
  int g = 0;
  if (lane <= k) {
    const unsigned long long v = a.best[r0 + lane];
    g = (int)(0xFFFFFFFFu - (uint32_t)(v & 0xFFFFFFFFull));
    a.best[r0 + lane] = 0ull;
    if (a.greedy_out) a.greedy_out[r0 + lane] = g;
  }
  const bool match = (lane < k) && (a.cand[r0 - b + lane] == g);
  const unsigned mm = __ballot_sync(0xFFFFFFFFu, match);
  const int n = __ffs(~mm) - 1;  // bit k of mm is clear, so n <= k
  const int corr = __shfl_sync(0xFFFFFFFFu, g, n);
  if (lane == 0) {
    if (a.bad[b]) {
      a.n_out[b] = -1;
      a.corr_out[b] = -1;
      a.bad[b] = 0;
    } else {
      a.n_out[b] = n;
      a.corr_out[b] = corr;
      a.len[b] += n + 1;
      a.root[b] = corr;
    }
  }
}

}  // namespace as2d
