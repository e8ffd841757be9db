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
// sum, unnormalised output) are combined in partition order (log-sum-exp).
#include "attn_dev.cuh"

namespace as2d {
namespace {

using namespace attn;

template <int D>
__global__ void __launch_bounds__(256, 1) attn_part_kernel(AttnArgs a) {
  __shared__ __align__(16) bf16 sK[kPart][kPitch];
  __shared__ __align__(16) bf16 sV[kPart][kPitch];
  // the keys/values already in the cache do not depend on the predecessor
  stage_old_kv<D>(a, a.layer, blockIdx.x, blockIdx.y, blockIdx.z, sK, sV, threadIdx.x, blockDim.x);
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  part_item<D, true>(a, a.layer, blockIdx.x, blockIdx.y, blockIdx.z, sK, sV, threadIdx.x,
                     blockDim.x, 0);
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

template <int D>
__global__ void __launch_bounds__(D) attn_merge_kernel(AttnArgs a) {
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  __shared__ float w[kMaxParts];
  __shared__ float s_l;
  merge_item<D>(a, blockIdx.x, blockIdx.y, w, &s_l, threadIdx.x, blockDim.x, 0);
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
  for (int b = 0; b < kv.batch; ++b) {
    const int64_t e = kv.len_upper[b] + (m.start[b + 1] - m.start[b]);
    max_len = e > max_len ? e : max_len;
  }
  const int parts = (int)((max_len + kPart - 1) / kPart);
  dim3 g1(parts, c.n_kv_heads, kv.batch);
  dim3 g2(m.rows, c.n_q_heads);
  a.qkv_part = kv.qkv_part;
  a.qkv_rinv = kv.qkv_rinv;
  a.rope = kv.rope;
  a.qkv_split = kv.qkv_split;
  a.qkv_ld = kv.rows_alloc;
  const dim3 gf(m.rows, c.n_q_heads + 2 * c.n_kv_heads);
  // Eight warps stage a partition fastest; when there are more items than
  // SMs, one warp per 16 query rows of the largest request (at least four,
  // for the staging copies) lets two CTAs share an SM, so long prefixes need
  // half the waves.  Which warp takes a row tile does not change its
  // arithmetic.
  int warps = 8;
  if ((long long)parts * c.n_kv_heads * kv.batch > md.sm_count) {
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
    if (e == cudaSuccess) e = launch_pdl(attn_merge_kernel<128>, g2, dim3(128), 0, st, a);
  } else {
    e = launch_pdl(qkv_finish_kernel<64>, gf, dim3(32), 0, st, a);
    if (e == cudaSuccess) e = launch_pdl(attn_part_kernel<64>, g1, tpart, 0, st, a);
    if (e == cudaSuccess) e = launch_pdl(attn_merge_kernel<64>, g2, dim3(64), 0, st, a);
  }
  return e;
}

}  // namespace as2d
