// k_basic.cu -- the verification pass's small kernels and the CUDA-core
// matrix-vector path.
//
// Every reduction below runs in an order fixed by the reduced dimension alone
// (never by the number of rows in the call), so each row's result is bitwise
// the same whether it is the only row (a k = 0 decode step) or one of the
// k + 1 rows of a block: batched and sequential execution agree exactly, which
// is the pathwise-equivalence requirement of App. C.4 held bit for bit.
#include "as2d_internal.h"

namespace as2d {
namespace {

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
  return v;  // identical in every lane: each butterfly step is commutative
}

__device__ __forceinline__ float dot8_acc(float acc, const uint4& w, const uint4& x) {
  const __nv_bfloat162* wp = reinterpret_cast<const __nv_bfloat162*>(&w);
  const __nv_bfloat162* xp = reinterpret_cast<const __nv_bfloat162*>(&x);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    float2 wf = __bfloat1622float2(wp[i]);
    float2 xf = __bfloat1622float2(xp[i]);
    acc = fmaf(wf.x, xf.x, acc);
    acc = fmaf(wf.y, xf.y, acc);
  }
  return acc;
}

// Orderable key of a float (larger float -> larger unsigned key).
__device__ __forceinline__ uint32_t float_key(float f) {
  uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// (logit, index) packed so that an unsigned max picks the largest logit and,
// among equal logits, the lowest index (the deterministic tie-break of Eq. 1).
__device__ __forceinline__ unsigned long long pack_best(float v, int idx) {
  return ((unsigned long long)float_key(v) << 32) |
         (unsigned long long)(0xFFFFFFFFu - (uint32_t)idx);
}

__device__ __forceinline__ float silu(float x) { return x / (1.0f + expf(-x)); }

// ---- embedding gather --------------------------------------------------------

__global__ void embed_kernel(RowMap m, const int32_t* __restrict__ cand,
                             const int32_t* __restrict__ root,
                             const bf16* __restrict__ E, int H, int V,
                             float* __restrict__ h, int32_t* err,
                             int32_t* bad) {
  int r = blockIdx.x;
  int b = row_request(m, r);
  int i = r - m.start[b];
  int tok = (i == 0) ? root[b] : cand[m.start[b] - b + i - 1];
  if (tok < 0 || tok >= V) {
    if (threadIdx.x == 0) {
      atomicOr(err, kErrBadToken);
      bad[b] = 1;
    }
    tok = 0;
  }
  const bf16* e = E + (size_t)tok * H;
  for (int c = threadIdx.x; c < H; c += blockDim.x)
    h[(size_t)r * H + c] = __bfloat162float(e[c]);
}

// ---- RMSNorm -> bf16 operand ---------------------------------------------------

__global__ void __launch_bounds__(256) rmsnorm_kernel(
    const float* __restrict__ h, const float* __restrict__ gain, int H,
    float eps, bf16* __restrict__ xn) {
  __shared__ float part[8];
  int r = blockIdx.x;
  const float* x = h + (size_t)r * H;
  float ss = 0.f;
  for (int c = threadIdx.x; c < H; c += blockDim.x) ss = fmaf(x[c], x[c], ss);
  ss = warp_sum(ss);
  if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = ss;
  __syncthreads();
  float tot = 0.f;
#pragma unroll
  for (int w = 0; w < 8; ++w) tot += part[w];
  float inv = rsqrtf(tot / (float)H + eps);
  for (int c = threadIdx.x; c < H; c += blockDim.x)
    xn[(size_t)r * H + c] = __float2bfloat16_rn(x[c] * inv * gain[c]);
}

// ---- matrix-vector products (CUDA cores) ------------------------------------------

enum { EPI_STORE = 0, EPI_RESID = 1, EPI_SWIGLU = 2, EPI_LOGITS = 3 };

struct GemvArgs {
  const bf16* X;
  int ldx;
  const bf16* W;
  int N, K;
  float* out_f32;
  int ldo;
  bf16* out_bf16;
  unsigned long long* best;
  int rows;
};

// One warp per output feature n, all rows of the call in chunks of four.
// Lane l reduces K positions l*8 + 256 j in increasing j, then the warp adds
// lane partials in a fixed butterfly: the order never depends on `rows`.
template <int EPI>
__global__ void __launch_bounds__(256) gemv_kernel(GemvArgs a) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n = blockIdx.x * 8 + warp;
  if (n >= a.N) return;
  const bf16* w0;
  const bf16* w1 = nullptr;
  if (EPI == EPI_SWIGLU) {
    w0 = a.W + ((size_t)(n >> 6) * 128 + (n & 63)) * a.K;  // gate row
    w1 = w0 + (size_t)64 * a.K;                             // matching up row
  } else {
    w0 = a.W + (size_t)n * a.K;
  }
  for (int r0 = 0; r0 < a.rows; r0 += 4) {
    float acc0[4] = {0.f, 0.f, 0.f, 0.f}, acc1[4] = {0.f, 0.f, 0.f, 0.f};
    for (int c = lane * 8; c < a.K; c += 256) {
      uint4 wv = __ldg(reinterpret_cast<const uint4*>(w0 + c));
      uint4 wu = make_uint4(0, 0, 0, 0);
      if (EPI == EPI_SWIGLU) wu = __ldg(reinterpret_cast<const uint4*>(w1 + c));
#pragma unroll
      for (int rr = 0; rr < 4; ++rr) {
        if (r0 + rr < a.rows) {
          uint4 xv = *reinterpret_cast<const uint4*>(a.X + (size_t)(r0 + rr) * a.ldx + c);
          acc0[rr] = dot8_acc(acc0[rr], wv, xv);
          if (EPI == EPI_SWIGLU) acc1[rr] = dot8_acc(acc1[rr], wu, xv);
        }
      }
    }
#pragma unroll
    for (int rr = 0; rr < 4; ++rr) {
      acc0[rr] = warp_sum(acc0[rr]);
      if (EPI == EPI_SWIGLU) acc1[rr] = warp_sum(acc1[rr]);
    }
    if (lane == 0) {
#pragma unroll
      for (int rr = 0; rr < 4; ++rr) {
        const int r = r0 + rr;
        if (r >= a.rows) break;
        if (EPI == EPI_STORE) {
          a.out_f32[(size_t)r * a.ldo + n] = acc0[rr];
        } else if (EPI == EPI_RESID) {
          a.out_f32[(size_t)r * a.ldo + n] += acc0[rr];
        } else if (EPI == EPI_SWIGLU) {
          a.out_bf16[(size_t)r * a.ldo + n] = __float2bfloat16_rn(silu(acc0[rr]) * acc1[rr]);
        } else {
          if (a.out_f32) a.out_f32[(size_t)r * a.ldo + n] = acc0[rr];
          atomicMax(&a.best[r], pack_best(acc0[rr], n));
        }
      }
    }
  }
}

// ---- RoPE + KV append -----------------------------------------------------------

// Block (row r, head slot hd) with d/2 threads.  Slots [0, nq) are query heads
// (rotated, kept fp32), [nq, nq + nkv) key heads (rotated, stored bf16 at the
// row's position), [nq + nkv, nq + 2 nkv) value heads (stored bf16).
__global__ void rope_append_kernel(RowMap m, const float* __restrict__ qkv,
                                   int qkv_ld, const int32_t* __restrict__ len,
                                   int nq, int nkv, int d, double theta,
                                   float* __restrict__ q_out, bf16* kc, bf16* vc,
                                   int layer, int batch, int cap) {
  const int r = blockIdx.x, hd = blockIdx.y, i = threadIdx.x, half = d >> 1;
  const int b = row_request(m, r);
  const int pos = len[b] + (r - m.start[b]);
  const float* src = qkv + (size_t)r * qkv_ld + (size_t)hd * d;
  float x0 = src[i], x1 = src[i + half];
  if (hd < nq + nkv) {
    double ang = (double)pos * pow(theta, -2.0 * (double)i / (double)d);
    double sn, cs;
    sincos(ang, &sn, &cs);
    float c = (float)cs, s = (float)sn;
    float y0 = x0 * c - x1 * s;
    float y1 = x1 * c + x0 * s;
    if (hd < nq) {
      float* qo = q_out + ((size_t)r * nq + hd) * d;
      qo[i] = y0;
      qo[i + half] = y1;
    } else {
      size_t base = ((((size_t)layer * batch + b) * nkv + (hd - nq)) * cap + pos) * d;
      kc[base + i] = __float2bfloat16_rn(y0);
      kc[base + i + half] = __float2bfloat16_rn(y1);
    }
  } else {
    size_t base = ((((size_t)layer * batch + b) * nkv + (hd - nq - nkv)) * cap + pos) * d;
    vc[base + i] = __float2bfloat16_rn(x0);
    vc[base + i + half] = __float2bfloat16_rn(x1);
  }
}

// ---- attention (CUDA cores, one block per row and query head) ----------------------

// Row r at position p attends to keys [0, p]: the prefix and the block's rows
// up to and including itself (causal inside the block).  Warp w takes keys
// w, w + 8, ... with an online softmax; the eight partial states are merged
// in warp order.  Nothing depends on the other rows of the call.
template <int D>
__global__ void __launch_bounds__(256) attention_kernel(
    RowMap m, const float* __restrict__ q, const int32_t* __restrict__ len,
    const bf16* __restrict__ kc, const bf16* __restrict__ vc, int layer,
    int batch, int cap, int nq, int nkv, bf16* __restrict__ ao) {
  constexpr int EPL = D / 32;
  __shared__ float s_m[8], s_l[8], s_acc[8][D];
  const int j = blockIdx.x, r = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int b = row_request(m, r);
  const int pos = len[b] + (r - m.start[b]);
  const int g = j / (nq / nkv);
  const float scale = rsqrtf((float)D);
  float qv[EPL];
#pragma unroll
  for (int e = 0; e < EPL; ++e) qv[e] = q[((size_t)r * nq + j) * D + lane * EPL + e] * scale;
  const size_t head = (((size_t)layer * batch + b) * nkv + g) * (size_t)cap * D;
  const bf16* K = kc + head;
  const bf16* V = vc + head;
  float mx = -INFINITY, l = 0.f, acc[EPL];
#pragma unroll
  for (int e = 0; e < EPL; ++e) acc[e] = 0.f;
  for (int t = warp; t <= pos; t += 8) {
    float kv[EPL], vv[EPL];
#pragma unroll
    for (int e = 0; e < EPL; ++e) {
      kv[e] = __bfloat162float(K[(size_t)t * D + lane * EPL + e]);
      vv[e] = __bfloat162float(V[(size_t)t * D + lane * EPL + e]);
    }
    float s = 0.f;
#pragma unroll
    for (int e = 0; e < EPL; ++e) s = fmaf(qv[e], kv[e], s);
    s = warp_sum(s);
    float mn = fmaxf(mx, s);
    float corr = expf(mx - mn);
    float p = expf(s - mn);
    l = l * corr + p;
#pragma unroll
    for (int e = 0; e < EPL; ++e) acc[e] = acc[e] * corr + p * vv[e];
    mx = mn;
  }
  if (lane == 0) {
    s_m[warp] = mx;
    s_l[warp] = l;
  }
#pragma unroll
  for (int e = 0; e < EPL; ++e) s_acc[warp][lane * EPL + e] = acc[e];
  __syncthreads();
  if (warp == 0) {
    float M = -INFINITY;
    for (int w = 0; w < 8; ++w) M = fmaxf(M, s_m[w]);
    float L = 0.f, o[EPL];
#pragma unroll
    for (int e = 0; e < EPL; ++e) o[e] = 0.f;
    for (int w = 0; w < 8; ++w) {
      float f = (s_l[w] > 0.f) ? expf(s_m[w] - M) : 0.f;
      L += s_l[w] * f;
#pragma unroll
      for (int e = 0; e < EPL; ++e) o[e] += s_acc[w][lane * EPL + e] * f;
    }
    float inv = 1.f / L;
#pragma unroll
    for (int e = 0; e < EPL; ++e)
      ao[((size_t)r * nq + j) * D + lane * EPL + e] = __float2bfloat16_rn(o[e] * inv);
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

template <int EPI>
cudaError_t run_gemv(const GemvArgs& a, cudaStream_t st) {
  dim3 grid((a.N + 7) / 8);
  gemv_kernel<EPI><<<grid, 256, 0, st>>>(a);
  return cudaGetLastError();
}

}  // namespace

// ---- launchers ------------------------------------------------------------------------

cudaError_t launch_embed(const RowMap& m, const Model& md, KvState& kv,
                         const int32_t* cand, cudaStream_t st) {
  embed_kernel<<<m.rows, 256, 0, st>>>(m, cand, kv.d_root, md.embed,
                                       md.cfg.hidden, md.cfg.vocab, kv.h,
                                       kv.d_err, kv.d_err + 1);
  return cudaGetLastError();
}

cudaError_t launch_rmsnorm(const RowMap& m, const Model& md, KvState& kv,
                           const float* gain, cudaStream_t st) {
  rmsnorm_kernel<<<m.rows, 256, 0, st>>>(kv.h, gain, md.cfg.hidden,
                                         md.cfg.rms_eps, kv.xn);
  return cudaGetLastError();
}

cudaError_t launch_gemv_qkv(const RowMap& m, const Model& md, KvState& kv,
                            int layer, cudaStream_t st) {
  GemvArgs a{kv.xn, md.cfg.hidden, md.w_qkv[layer], md.qkv_rows, md.cfg.hidden,
             kv.qkv, md.qkv_rows, nullptr, nullptr, m.rows};
  return run_gemv<EPI_STORE>(a, st);
}

cudaError_t launch_rope_append(const RowMap& m, const Model& md, KvState& kv,
                               int layer, cudaStream_t st) {
  const as2d_config& c = md.cfg;
  dim3 grid(m.rows, c.n_q_heads + 2 * c.n_kv_heads);
  rope_append_kernel<<<grid, c.head_dim / 2, 0, st>>>(
      m, kv.qkv, md.qkv_rows, kv.d_len, c.n_q_heads, c.n_kv_heads, c.head_dim,
      (double)c.rope_theta, kv.q, kv.k_cache, kv.v_cache, layer, kv.batch,
      kv.capacity);
  return cudaGetLastError();
}

cudaError_t launch_attention(const RowMap& m, const Model& md, KvState& kv,
                             int layer, cudaStream_t st) {
  const as2d_config& c = md.cfg;
  dim3 grid(c.n_q_heads, m.rows);
  if (c.head_dim == 128)
    attention_kernel<128><<<grid, 256, 0, st>>>(m, kv.q, kv.d_len, kv.k_cache,
                                                kv.v_cache, layer, kv.batch,
                                                kv.capacity, c.n_q_heads,
                                                c.n_kv_heads, kv.ao);
  else
    attention_kernel<64><<<grid, 256, 0, st>>>(m, kv.q, kv.d_len, kv.k_cache,
                                               kv.v_cache, layer, kv.batch,
                                               kv.capacity, c.n_q_heads,
                                               c.n_kv_heads, kv.ao);
  return cudaGetLastError();
}

cudaError_t launch_gemv_o(const RowMap& m, const Model& md, KvState& kv,
                          int layer, cudaStream_t st) {
  GemvArgs a{kv.ao, md.q_dim, md.w_o[layer], md.cfg.hidden, md.q_dim,
             kv.h, md.cfg.hidden, nullptr, nullptr, m.rows};
  return run_gemv<EPI_RESID>(a, st);
}

cudaError_t launch_gemv_gate_up(const RowMap& m, const Model& md, KvState& kv,
                                int layer, cudaStream_t st) {
  GemvArgs a{kv.xn, md.cfg.hidden, md.w_gu[layer], md.cfg.ffn, md.cfg.hidden,
             nullptr, md.cfg.ffn, kv.u, nullptr, m.rows};
  return run_gemv<EPI_SWIGLU>(a, st);
}

cudaError_t launch_gemv_down(const RowMap& m, const Model& md, KvState& kv,
                             int layer, cudaStream_t st) {
  GemvArgs a{kv.u, md.cfg.ffn, md.w_down[layer], md.cfg.hidden, md.cfg.ffn,
             kv.h, md.cfg.hidden, nullptr, nullptr, m.rows};
  return run_gemv<EPI_RESID>(a, st);
}

cudaError_t launch_lm_head(const RowMap& m, const Model& md, KvState& kv,
                           float* logits, cudaStream_t st) {
  GemvArgs a{kv.xn, md.cfg.hidden, md.lm_head, md.cfg.vocab, md.cfg.hidden,
             logits, md.cfg.vocab, nullptr, kv.best, m.rows};
  return run_gemv<EPI_LOGITS>(a, st);
}

cudaError_t launch_accept(const RowMap& m, const Model& md, KvState& kv,
                          const int32_t* cand, const as2d_verify_out& out,
                          cudaStream_t st) {
  (void)md;
  accept_kernel<<<m.batch, 32, 0, st>>>(m, cand, kv.best, kv.d_len, kv.d_root,
                                        kv.d_err + 1, out.n_accepted,
                                        out.correction_token, out.greedy);
  return cudaGetLastError();
}

cudaError_t launch_rollback(KvState& kv, const int32_t* new_len,
                            const int32_t* new_root, cudaStream_t st) {
  RollbackArgs a;
  a.batch = kv.batch;
  for (int b = 0; b < kv.batch; ++b) {
    a.len[b] = new_len[b];
    a.root[b] = new_root[b];
  }
  rollback_kernel<<<1, kMaxBatch, 0, st>>>(a, kv.d_len, kv.d_root, kv.d_err);
  return cudaGetLastError();
}

cudaError_t launch_f32_from_bf16(float* dst, const void* src, int64_t n,
                                 cudaStream_t st) {
  f32_from_bf16_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(
      dst, (const bf16*)src, n);
  return cudaGetLastError();
}

}  // namespace as2d
