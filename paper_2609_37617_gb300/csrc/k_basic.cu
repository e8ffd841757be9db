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
#include "small_dev.cuh"

namespace as2d {
namespace {

// ---- embedding gather --------------------------------------------------------

// (cos, sin) of pos * theta^(-2e/d), e < d/2: angle and trigonometry in
// double, rounded once to float.
__device__ __forceinline__ float2 rope_angle(int pos, int e, int d, double theta) {
  const double ang = (double)pos * pow(theta, -2.0 * (double)e / (double)d);
  double sn, cs;
  sincos(ang, &sn, &cs);
  return make_float2((float)cs, (float)sn);
}

// The rotary table of every position of a state, built once at set-up.
__global__ void rope_table_kernel(float2* __restrict__ out, int d, double theta) {
  const int pos = blockIdx.x, e = threadIdx.x;
  out[(size_t)pos * (d / 2) + e] = rope_angle(pos, e, d, theta);
}

// Also writes the row's rotary table -- gathered from the state's table of
// every position when there is one (rope_full), else computed.
__global__ void __launch_bounds__(128) embed_kernel(
    RowMap m, const int32_t* __restrict__ cand, const int32_t* __restrict__ root,
    const int32_t* __restrict__ root_override, const bf16* __restrict__ E, int H, int V, float* __restrict__ h, int32_t* err, int32_t* bad,
    const int32_t* __restrict__ len, int cap, float2* __restrict__ rope,
    const float2* __restrict__ rope_full, int d, double theta, const float* __restrict__ g0,
    bf16* __restrict__ xn, float* __restrict__ ss, int ss_ld) {
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  __shared__ float part[4];
  const int r = blockIdx.x;
  const int b = row_request(m, r);
  const int i = r - m.start[b];
  // a request whose length leaves no room for its rows is flagged and skipped
  // downstream (rows_fit); its rows take position 0's rotary entries
  const bool fits = rows_fit(len[b], m.start[b + 1] - m.start[b], cap);
  if (!fits && threadIdx.x == 0) {
    atomicOr(err, kErrCapacity);
    bad[b] = 1;
  }
  if ((int)threadIdx.x < d / 2) {
    const int e = threadIdx.x, pos = fits ? len[b] + i : 0;
    rope[(size_t)r * (d / 2) + e] =
        rope_full ? rope_full[(size_t)pos * (d / 2) + e] : rope_angle(pos, e, d, theta);
  }
  int tok = (i == 0) ? (root_override ? root_override[b] : root[b]) : cand[m.start[b] - b + i - 1];
  if (tok < 0 || tok >= V) {
    if (threadIdx.x == 0) {
      atomicOr(err, kErrBadToken);
      bad[b] = 1;
    }
    tok = 0;
  }
  embed_row_body(E + (size_t)tok * H, g0, H, r, ss_ld, h, xn, ss, threadIdx.x, 128, part, 0);
}

// ---- accept scan + state update ---------------------------------------------------

// One warp per request (App. C.2): g_i from the packed maxima, the number of
// leading candidates equal to the greedy tokens by ballot, the correction by
// shuffle, then L += n + 1 and root = correction, all on the device.
__global__ void accept_kernel(AcceptArgs a) {
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  accept_request(a, blockIdx.x, threadIdx.x);
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
                         const int32_t* cand, cudaStream_t st, const int32_t* root_override) {
  ++kv.launches;
  return launch_pdl(embed_kernel, dim3(m.rows), dim3(128), 0, st, m, cand,
                    (const int32_t*)kv.d_root, root_override, (const bf16*)md.embed, md.cfg.hidden,
                    md.cfg.vocab, kv.h, kv.d_err, kv.d_err + 1, (const int32_t*)kv.d_len,
                    kv.capacity, kv.rope, (const float2*)kv.rope_full, md.cfg.head_dim,
                    (double)md.cfg.rope_theta, md.attn_norm[0], kv.xn, kv.ss, kv.rows_alloc);
}

cudaError_t launch_rope_table(const Model& md, KvState& kv, cudaStream_t st) {
  rope_table_kernel<<<kv.capacity, md.cfg.head_dim / 2, 0, st>>>(
      kv.rope_full, md.cfg.head_dim, (double)md.cfg.rope_theta);
  return cudaGetLastError();
}

cudaError_t launch_accept(const RowMap& m, const Model& md, KvState& kv,
                          const int32_t* cand, const as2d_verify_out& out,
                          cudaStream_t st, bool force) {
  (void)md;
  ++kv.launches;
  AcceptArgs a{m, cand, kv.best, kv.d_len, kv.d_root, kv.d_err + 1, out.n_accepted,
               out.correction_token, out.greedy, force ? 1 : 0};
  return launch_pdl(accept_kernel, dim3(m.batch), dim3(32), 0, st, a);
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
