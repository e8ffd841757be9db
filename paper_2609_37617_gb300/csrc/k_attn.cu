// k_attn.cu -- grouped-query attention of a verification block over the
// retained prefix, split over the key axis (flash-decode), with the causal
// mask inside the block.
//
// Row i of request b sits at position L_b + i and attends to keys [0, L_b + i]:
// the prefilled audio/instruction prefix, the committed tokens, and the
// block's own rows up to itself.  All G = n_q / n_kv query heads of a key/value
// head, for all k + 1 rows, form one query matrix of (k + 1) * G rows, so each
// key/value entry is read from HBM once per block.
//
// Pass 0 (qkv_finish_kernel): the QKV projection arrives as split-K partial
// sums (TC_PART); one CTA per (token row, head) adds them in rank order,
// scales by the row's 1 / rms, rotates (RoPE) and writes the queries, and
// appends the new keys and values to the cache.
// Pass 1 (attn_part_kernel): one CTA per (64-key partition, kv head, request).
// Keys and values are staged in shared memory -- those already in the cache
// before the kernel waits for pass 0, the block's own after; each warp takes
// 16 query rows at a time (4 to 8 warps, by the largest request);
// S = Q K^T and O = P V run on the tensor cores (mma.sync m16n8k16, bf16 in,
// fp32 accumulate), with Q and P each split into bf16 hi + lo parts (two MMAs)
// so that only the bf16 cache itself limits precision; the softmax runs in
// fp32 in base 2.  Partition boundaries
// are fixed multiples of 64 positions, so a query's partial results do not
// depend on the other rows of the call (batch invariance).
// Pass 2 (attn_merge_kernel): per (row, query head) the partitions' (max,
// sum, unnormalised output) are combined (log-sum-exp) in an order fixed by
// the row's own number of partitions.
#include "attn_dev.cuh"

namespace as2d {
namespace {

using namespace attn;

template <int D>
__global__ void __launch_bounds__(256, 1) attn_part_kernel(AttnArgs a) {
  __shared__ __align__(16) bf16 sK[kPart][kPitch];
  __shared__ __align__(16) bf16 sV[kPart][kPitch];
  // item blockIdx.x -> (request, partition): only each request's own partitions
  int b = 0;
  while (b + 1 < a.batch && a.part_start[b + 1] <= (int)blockIdx.x) ++b;
  const int part = (int)blockIdx.x - a.part_start[b];
  const bool fits = rows_fit(a.len[b], a.rm.start[b + 1] - a.rm.start[b], a.cap);
  // the keys/values already in the cache do not depend on the predecessor
  if (fits) stage_old_kv<D>(a, a.layer, part, blockIdx.y, b, sK, sV, threadIdx.x, blockDim.x);
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  if (!fits) return;  // flagged by the embedding kernel; nothing of the cache is read
  part_item<D, true>(a, a.layer, part, blockIdx.y, b, sK, sV, threadIdx.x, blockDim.x, 0);
}

// The QKV projection finished from its split-K sums (TC_PART): one CTA of
// D / 2 threads per (token row, head); thread e
// forms the pair (e, e + D/2) -- rotated queries into q, rotated keys and
// values appended to the cache.  Every load of a thread is issued before the
// first is used.
template <int D>
__global__ void __launch_bounds__(D / 2) qkv_finish_kernel(AttnArgs a) {
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  constexpr int H2 = D / 2;
  const int gm = blockIdx.x, head = blockIdx.y, e = threadIdx.x;
  const int b = row_request(a.rm, gm), pos = a.len[b] + (gm - a.rm.start[b]);
  if (!rows_fit(a.len[b], a.rm.start[b + 1] - a.rm.start[b], a.cap)) return;  // no append
  const float2 y = (head < a.nq + a.nkv) ? qk_rotated<D>(a, head, e, gm)
                                         : make_float2(qkv_value(a, head * D + e, gm),
                                                       qkv_value(a, head * D + e + H2, gm));
  if (head < a.nq) {
    float* q = const_cast<float*>(a.q) + (size_t)gm * a.nq * D + head * D;
    q[e] = y.x;
    q[e + H2] = y.y;
  } else {
    const bool is_k = head < a.nq + a.nkv;
    const int g = is_k ? head - a.nq : head - a.nq - a.nkv;
    bf16* dst = const_cast<bf16*>(is_k ? a.kc : a.vc) +
                ((((size_t)a.layer * a.batch + b) * a.nkv + g) * a.cap + pos) * D;
    dst[e] = __float2bfloat16_rn(y.x);
    dst[e + H2] = __float2bfloat16_rn(y.y);
  }
}

// Pass 2 for one (row, query head) per CTA of D x (1..4) threads.  All the
// partitions' (max, sum) pairs are loaded together into shared memory; the
// maximum, the weights 2^(m_p - M) and the total (warp 0: lane e adds
// partitions e, e + 32, ... in order, then a butterfly) follow; the outputs
// are added by gs = min(4, ceil(parts / 32)) groups of D threads, group q
// taking a contiguous run of partitions in order, 32 loads in flight, and the
// groups' sums are added in group order.  Every order depends on the row's
// own number of partitions alone; with at most 32 partitions (positions below
// 2048) it is the single in-order sum.
constexpr int kMergeGroups = 4;

template <int D>
__global__ void __launch_bounds__(kMergeGroups * D) attn_merge_kernel(AttnArgs a) {
  constexpr int PF = 32;
  __shared__ float2 s_ml[kMaxParts];
  __shared__ float s_w[kMaxParts];
  __shared__ float s_red[kMergeGroups * D / 32];
  __shared__ float s_o[kMergeGroups - 1][D];
  __shared__ float s_l;
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  const int r = blockIdx.x, j = blockIdx.y, tid = threadIdx.x, nthr = blockDim.x;
  const int G = a.nq / a.nkv;
  const int b = row_request(a.rm, r);
  const int i = r - a.rm.start[b];
  const int g = j / G, qr = i * G + (j - g * G);
  if (!rows_fit(a.len[b], a.rm.start[b + 1] - a.rm.start[b], a.cap)) {
    // a skipped request: zero output, no partition is read
    for (int e = tid; e < D; e += nthr) {
      a.ao[(size_t)r * a.nq * D + (size_t)j * D + e] = __float2bfloat16_rn(0.f);
      a.ao[(size_t)(a.lo_row + r) * a.nq * D + (size_t)j * D + e] = __float2bfloat16_rn(0.f);
    }
    return;
  }
  const int pos = a.len[b] + i;
  const int nparts = pos / kPart + 1;
  const size_t base = (size_t)(b * a.nkv + g) * a.parts_max * a.qmax + qr;
  const int want = (nparts + 31) / 32;
  const int gs = want < kMergeGroups ? want : kMergeGroups;
  const int chunk = (nparts + gs - 1) / gs;
  const int grp = tid / D, e = tid - grp * D;
  const int p_begin = grp * chunk;
  const int p_end = (p_begin + chunk) < nparts ? (p_begin + chunk) : nparts;
  // the group's first PF outputs are in flight with the (max, sum) loads
  float ov[PF];
  if (grp < gs) {
#pragma unroll
    for (int u = 0; u < PF; ++u)
      ov[u] = (p_begin + u < p_end) ? a.ws_o[(base + (size_t)(p_begin + u) * a.qmax) * D + e] : 0.f;
  }
  for (int p = tid; p < nparts; p += nthr) s_ml[p] = a.ws_ml[base + (size_t)p * a.qmax];
  __syncthreads();
  float M = -INFINITY;
  for (int p = tid; p < nparts; p += nthr) M = fmaxf(M, s_ml[p].x);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xFFFFFFFFu, M, o));
  if ((tid & 31) == 0) s_red[tid >> 5] = M;
  __syncthreads();
  M = s_red[0];
  for (int w = 1; w < nthr / 32; ++w) M = fmaxf(M, s_red[w]);
  for (int p = tid; p < nparts; p += nthr) {
    const float mp = s_ml[p].x;
    s_w[p] = (mp == -INFINITY) ? 0.f : exp2f(mp - M);
  }
  __syncthreads();
  if (tid < 32) {
    float l = 0.f;
    for (int p = tid; p < nparts; p += 32) l += s_ml[p].y * s_w[p];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) l += __shfl_xor_sync(0xFFFFFFFFu, l, o);
    if (tid == 0) s_l = l;
  }
  float o = 0.f;
  if (grp < gs) {
    for (int p0 = p_begin; p0 < p_end; p0 += PF) {
      if (p0 > p_begin) {
#pragma unroll
        for (int u = 0; u < PF; ++u)
          ov[u] = (p0 + u < p_end) ? a.ws_o[(base + (size_t)(p0 + u) * a.qmax) * D + e] : 0.f;
      }
#pragma unroll
      for (int u = 0; u < PF; ++u)
        if (p0 + u < p_end) o += ov[u] * s_w[p0 + u];
    }
    if (grp > 0) s_o[grp - 1][e] = o;
  }
  __syncthreads();
  if (grp == 0) {
    for (int q = 1; q < gs; ++q) o += s_o[q - 1][e];
    const float ov_ = o / s_l;
    const bf16 oh = __float2bfloat16_rn(ov_);
    a.ao[(size_t)r * a.nq * D + (size_t)j * D + e] = oh;
    a.ao[(size_t)(a.lo_row + r) * a.nq * D + (size_t)j * D + e] =
        __float2bfloat16_rn(ov_ - __bfloat162float(oh));
  }
}

}  // namespace

int attn_partitions(int capacity) { return (capacity + kPart - 1) / kPart; }

cudaError_t launch_attention_split(const RowMap& m, const Model& md, KvState& kv, int layer,
                                   cudaStream_t st) {
  const as2d_config& c = md.cfg;
  AttnArgs a;
  a.rm = m;
  a.q = kv.q;
  a.len = kv.d_len;
  a.kc = kv.k_cache;
  a.vc = kv.v_cache;
  a.layer = layer;
  a.batch = kv.batch;
  a.cap = kv.capacity;
  a.nq = c.n_q_heads;
  a.nkv = c.n_kv_heads;
  a.qscale = 1.4426950408889634f / sqrtf((float)c.head_dim);
  a.ws_o = kv.attn_o;
  a.ws_ml = kv.attn_ml;
  a.parts_max = kv.attn_parts;
  a.qmax = kv.attn_qmax;
  a.ao = kv.ao;
  a.lo_row = kv.rows_alloc;
  int64_t max_len = 0;
  a.part_start[0] = 0;
  for (int b = 0; b < kv.batch; ++b) {
    const int64_t e = kv.len_upper[b] + (m.start[b + 1] - m.start[b]);
    max_len = e > max_len ? e : max_len;
    a.part_start[b + 1] = a.part_start[b] + (int)((e + kPart - 1) / kPart);
  }
  const int parts = (int)((max_len + kPart - 1) / kPart);
  const int items = a.part_start[kv.batch];
  dim3 g1(items, c.n_kv_heads);
  dim3 g2(m.rows, c.n_q_heads);
  a.qkv_part = kv.qkv_part;
  a.qkv_rinv = kv.qkv_rinv;
  a.rope = kv.rope;
  a.qkv_split = kv.qkv_split;
  a.qkv_ld = kv.rows_alloc;
  const dim3 gf(m.rows, c.n_q_heads + 2 * c.n_kv_heads);
  // merge groups for the call's longest row (each row uses min(4, its own
  // partitions / 32 rounded up) of them)
  int mg = (parts + 31) / 32;
  mg = mg < 1 ? 1 : (mg > kMergeGroups ? kMergeGroups : mg);
  // Eight warps stage a partition fastest; when there are more items than
  // SMs, one warp per 16 query rows of the largest request (at least four,
  // for the staging copies) lets two CTAs share an SM, so long prefixes need
  // half the waves.  Which warp takes a row tile does not change its
  // arithmetic.
  int warps = 8;
  if ((long long)items * c.n_kv_heads > md.sm_count) {
    int qn_max = 0;
    for (int b = 0; b < kv.batch; ++b) {
      const int qn = (m.start[b + 1] - m.start[b]) * (c.n_q_heads / c.n_kv_heads);
      qn_max = qn > qn_max ? qn : qn_max;
    }
    warps = (qn_max + 15) / 16;
    warps = warps < 4 ? 4 : (warps > 8 ? 8 : warps);
  }
  const dim3 tpart(32 * warps);
  cudaError_t e;
  kv.launches += 3;
  if (c.head_dim == 128) {
    e = launch_pdl(qkv_finish_kernel<128>, gf, dim3(64), 0, st, a);
    if (e == cudaSuccess) e = launch_pdl(attn_part_kernel<128>, g1, tpart, 0, st, a);
    if (e == cudaSuccess) e = launch_pdl(attn_merge_kernel<128>, g2, dim3(128 * mg), 0, st, a);
  } else {
    e = launch_pdl(qkv_finish_kernel<64>, gf, dim3(32), 0, st, a);
    if (e == cudaSuccess) e = launch_pdl(attn_part_kernel<64>, g1, tpart, 0, st, a);
    if (e == cudaSuccess) e = launch_pdl(attn_merge_kernel<64>, g2, dim3(64 * mg), 0, st, a);
  }
  return e;
}

}  // namespace as2d
