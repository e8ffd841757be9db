// k_basic.cu -- the verification pass's small kernels: embedding gather (with
// the rotary table and the first projection's operand), the accept scan with
// the on-device state update, rollback, and a load-time conversion.
//
// Every reduction below runs in an order fixed by the reduced dimension alone
// (never by the number of rows in the call), so each row's result is bitwise
// the same whether it is the only row (a k = 0 decode step) or one of the
// k + 1 rows of a block: batched and sequential execution agree exactly, which
// is the pathwise-equivalence requirement of App. C.4 held bit for bit.
#include "as2d_internal.h"
#include "ptx_sm100.cuh"

namespace as2d {
namespace {

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
  return v;  // identical in every lane: each butterfly step is commutative
}

// ---- embedding gather --------------------------------------------------------

// Also writes the row's rotary table: (cos, sin) of pos * theta^(-2e/d) for
// e < d/2, angles and trigonometry in double, rounded once to float.
__global__ void __launch_bounds__(256) embed_kernel(
    RowMap m, const int32_t* __restrict__ cand, const int32_t* __restrict__ root,
    const bf16* __restrict__ E, int H, int V, float* __restrict__ h, int32_t* err, int32_t* bad,
    const int32_t* __restrict__ len, float2* __restrict__ rope, int d, double theta,
    const float* __restrict__ g0, bf16* __restrict__ xn, float* __restrict__ ss, int ss_ld) {
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  __shared__ float part[8];
  int r = blockIdx.x;
  int b = row_request(m, r);
  int i = r - m.start[b];
  if ((int)threadIdx.x < d / 2) {
    const int e = threadIdx.x;
    const double ang = (double)(len[b] + i) * pow(theta, -2.0 * (double)e / (double)d);
    double sn, cs;
    sincos(ang, &sn, &cs);
    rope[(size_t)r * (d / 2) + e] = make_float2((float)cs, (float)sn);
  }
  int tok = (i == 0) ? root[b] : cand[m.start[b] - b + i - 1];
  if (tok < 0 || tok >= V) {
    if (threadIdx.x == 0) {
      atomicOr(err, kErrBadToken);
      bad[b] = 1;
    }
    tok = 0;
  }
  // residual stream = embedding row; the first projection's operand is
  // h * g as bf16 hi + lo parts (lo rows start at ss_ld = rows allocated) and
  // its row sum of squares goes to tile slot 0 (slots 1.. = 0)
  const bf16* e = E + (size_t)tok * H;
  float sq = 0.f;
  for (int c = threadIdx.x; c < H; c += blockDim.x) {
    const float x = __bfloat162float(e[c]);
    h[(size_t)r * H + c] = x;
    const float xv = x * g0[c];
    const bf16 xh = __float2bfloat16_rn(xv);
    xn[(size_t)r * H + c] = xh;
    xn[(size_t)(ss_ld + r) * H + c] = __float2bfloat16_rn(xv - __bfloat162float(xh));
    sq = fmaf(x, x, sq);
  }
  sq = warp_sum(sq);
  if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = sq;
  __syncthreads();
  const int nt = H / 128;
  for (int t = threadIdx.x; t < nt; t += blockDim.x) {
    float tot = 0.f;
    if (t == 0)
      for (int w = 0; w < 8; ++w) tot += part[w];
    ss[(size_t)t * ss_ld + r] = tot;
  }
}

// ---- accept scan + state update ---------------------------------------------------

// One warp per request (App. C.2): g_i from the packed maxima, the number of
// leading candidates equal to the greedy tokens by ballot, the correction by
// shuffle, then L += n + 1 and root = correction, all on the device.
__global__ void accept_kernel(RowMap m, const int32_t* __restrict__ cand,
                              unsigned long long* best, int32_t* len,
                              int32_t* root, int32_t* bad, int32_t* n_out,
                              int32_t* corr_out, int32_t* greedy_out) {
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  const int b = blockIdx.x, lane = threadIdx.x;
  const int r0 = m.start[b];
  const int k = m.start[b + 1] - r0 - 1;
  int g = 0;
  if (lane <= k) {
    unsigned long long v = best[r0 + lane];
    g = (int)(0xFFFFFFFFu - (uint32_t)(v & 0xFFFFFFFFull));
    best[r0 + lane] = 0ull;
    if (greedy_out) greedy_out[r0 + lane] = g;
  }
  const bool match = (lane < k) && (cand[r0 - b + lane] == g);
  const unsigned mm = __ballot_sync(0xFFFFFFFFu, match);
  const int n = __ffs(~mm) - 1;  // bit k of mm is clear, so n <= k
  const int corr = __shfl_sync(0xFFFFFFFFu, g, n);
  if (lane == 0) {
    if (bad[b]) {
      n_out[b] = -1;
      corr_out[b] = -1;
      bad[b] = 0;
    } else {
      n_out[b] = n;
      corr_out[b] = corr;
      len[b] += n + 1;
      root[b] = corr;
    }
  }
}

struct RollbackArgs {
  int32_t batch;
  int32_t len[kMaxBatch];
  int32_t root[kMaxBatch];
};

__global__ void rollback_kernel(RollbackArgs a, int32_t* len, int32_t* root,
                                int32_t* err) {
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  int b = threadIdx.x;
  if (b >= a.batch) return;
  if (a.len[b] <= len[b]) {
    len[b] = a.len[b];
    root[b] = a.root[b];
  } else {
    atomicOr(err, kErrRollback);
  }
}

__global__ void f32_from_bf16_kernel(float* dst, const bf16* src, int64_t n) {
  int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) dst[i] = __bfloat162float(src[i]);
}

}  // namespace

// ---- launchers ------------------------------------------------------------------------

cudaError_t launch_embed(const RowMap& m, const Model& md, KvState& kv,
                         const int32_t* cand, cudaStream_t st) {
  ++kv.launches;
  return launch_pdl(embed_kernel, dim3(m.rows), dim3(256), 0, st, m, cand,
                    (const int32_t*)kv.d_root, (const bf16*)md.embed, md.cfg.hidden,
                    md.cfg.vocab, kv.h, kv.d_err, kv.d_err + 1, (const int32_t*)kv.d_len,
                    kv.rope, md.cfg.head_dim, (double)md.cfg.rope_theta, md.attn_norm[0], kv.xn,
                    kv.ss, kv.rows_alloc);
}

cudaError_t launch_accept(const RowMap& m, const Model& md, KvState& kv,
                          const int32_t* cand, const as2d_verify_out& out,
                          cudaStream_t st) {
  (void)md;
  ++kv.launches;
  return launch_pdl(accept_kernel, dim3(m.batch), dim3(32), 0, st, m, cand, kv.best, kv.d_len,
                    kv.d_root, kv.d_err + 1, out.n_accepted, out.correction_token, out.greedy);
}

cudaError_t launch_rollback(KvState& kv, const int32_t* new_len,
                            const int32_t* new_root, cudaStream_t st) {
  RollbackArgs a;
  a.batch = kv.batch;
  for (int b = 0; b < kv.batch; ++b) {
    a.len[b] = new_len[b];
    a.root[b] = new_root[b];
  }
  return launch_pdl(rollback_kernel, dim3(1), dim3(kMaxBatch), 0, st, a, kv.d_len, kv.d_root,
                    kv.d_err);
}

cudaError_t launch_f32_from_bf16(float* dst, const void* src, int64_t n,
                                 cudaStream_t st) {
  f32_from_bf16_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(
      dst, (const bf16*)src, n);
  return cudaGetLastError();
}

}  // namespace as2d
