// attn_dev.cuh -- the attention of a verification block as device functions
// run by a group of threads: one (64-key partition, kv head, request) item of
// the split-KV pass, and one (row, query head) item of the merge.  Used by the
// standalone kernels (k_attn.cu) and by the persistent verification kernel.
#pragma once

#include "as2d_internal.h"
#include "ptx_sm100.cuh"

namespace as2d {
namespace attn {

__device__ __forceinline__ void bar_sync(int id, int n) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory");
}

constexpr int kPart = 64;      // keys per partition (fixed)
constexpr int kPitch = 136;    // bf16 per shared row: 128 + 8 (272 B, conflict-free)

// x, y -> packed bf16 hi parts and packed bf16 lo parts (x - hi).
__device__ __forceinline__ void split_bf16x2(float x, float y, uint32_t& hi, uint32_t& lo) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(x, y);
  const float2 hf = __bfloat1622float2(h);
  const __nv_bfloat162 l = __floats2bfloat162_rn(x - hf.x, y - hf.y);
  hi = *reinterpret_cast<const uint32_t*>(&h);
  lo = *reinterpret_cast<const uint32_t*>(&l);
}

__device__ __forceinline__ void mma_16816(float (&c)[4], const uint32_t (&a)[4], uint32_t b0,
                                          uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
      "{%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ void ldmatrix_x4_trans(uint32_t (&r)[4], const void* p) {
  const uint32_t a = (uint32_t)__cvta_generic_to_shared(p);
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(a));
}

__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  const uint32_t d = (uint32_t)__cvta_generic_to_shared(dst);
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(d), "l"(src) : "memory");
}

struct AttnArgs {
  RowMap rm;
  const float* q;       // [rows][nq * D] rotated queries
  const int32_t* len;
  const bf16* kc;
  const bf16* vc;
  int layer, batch, cap, nq, nkv;
  float qscale;         // log2(e) / sqrt(D)
  float* ws_o;          // [batch][nkv][parts_max][qmax][D]
  float2* ws_ml;        // [batch][nkv][parts_max][qmax] (max, sum), base 2
  int parts_max, qmax;
  bf16* ao;             // [2 rows][nq * D]: hi rows, then lo rows from lo_row
  int lo_row;
  // split-K sums of the QKV projection (TC_PART), when attention finishes them
  const float* qkv_part;  // [tile][split][qkv_ld][128], tile = column / 128
  const float* qkv_rinv;  // [qkv_ld] 1 / rms of each token row
  const float2* rope;     // [rows][D / 2] (cos, sin)
  int qkv_split, qkv_ld;
  // partition items of the split-KV pass, request by request: request b owns
  // items [part_start[b], part_start[b + 1]) (its own partitions only)
  int32_t part_start[kMaxBatch + 1];
};

// ---- finishing the QKV projection from its split-K sums ----------------------

// Projection value of column col (q, k or v head * D + e) for token row gm:
// the split parts added in rank order, times the row's 1 / rms.
__device__ __forceinline__ float qkv_value(const AttnArgs& a, int col, int gm) {
  const float* src = a.qkv_part + ((size_t)(col >> 7) * a.qkv_split * a.qkv_ld + gm) * 128 + (col & 127);
  float v[8];
#pragma unroll
  for (int r = 0; r < 8; ++r) v[r] = r < a.qkv_split ? src[(size_t)r * a.qkv_ld * 128] : 0.f;
  float acc = 0.f;
#pragma unroll
  for (int r = 0; r < 8; ++r)
    if (r < a.qkv_split) acc += v[r];
  return acc * a.qkv_rinv[gm];
}

// Rotate-half RoPE of the pair (x at e, xp at e + D/2): returns the rotated
// value at e (first) and at e + D/2 (second).
__device__ __forceinline__ float2 rope_pair(float x, float xp, float2 cs) {
  return make_float2(fmaf(x, cs.x, -(xp * cs.y)), fmaf(xp, cs.x, x * cs.y));
}

// Rotated query / key pair (e, e + D/2) of head `head` (column head * D) at
// token row gm, e < D/2.
template <int D>
__device__ __forceinline__ float2 qk_rotated(const AttnArgs& a, int head, int e, int gm) {
  const float x = qkv_value(a, head * D + e, gm), xp = qkv_value(a, head * D + e + D / 2, gm);
  return rope_pair(x, xp, a.rope[(size_t)gm * (D / 2) + e]);
}


// Stages keys/values [p0, p0 + 64) of the item into sK/sV: rows below `from`
// are left alone, rows in [from, kend) are copied from the cache (cp.async,
// committed), rows at or beyond kend are zero.
template <int D>
__device__ __forceinline__ void stage_kv(const AttnArgs& a, int layer, int part, int g, int b,
                                         int from, bf16 (*sK)[kPitch], bf16 (*sV)[kPitch],
                                         int tid, int nthr, int upto) {
  const int p0 = part * kPart;
  const size_t head = (((size_t)layer * a.batch + b) * a.nkv + g) * (size_t)a.cap;
  constexpr int SEGS = D / 8;  // 16-byte pieces per row
  for (int idx = tid; idx < kPart * SEGS; idx += nthr) {
    const int t = idx / SEGS, sg = idx - t * SEGS;
    const int pos = p0 + t;
    if (pos < from) continue;
    if (pos < upto) {
      cp_async16(&sK[t][sg * 8], a.kc + (head + pos) * D + sg * 8);
      cp_async16(&sV[t][sg * 8], a.vc + (head + pos) * D + sg * 8);
    } else {
      *reinterpret_cast<uint4*>(&sK[t][sg * 8]) = make_uint4(0, 0, 0, 0);
      *reinterpret_cast<uint4*>(&sV[t][sg * 8]) = make_uint4(0, 0, 0, 0);
    }
  }
  asm volatile("cp.async.commit_group;" ::: "memory");
}

// The item's keys/values already in the cache ([0, L) of the request) go to
// sK/sV before the block's own rows exist (cp.async, committed); positions at
// or beyond L + M are zero.  Rows [L, L + M) are left for part_item.
template <int D>
__device__ __forceinline__ void stage_old_kv(const AttnArgs& a, int layer, int part, int g,
                                             int b, bf16 (*sK)[kPitch], bf16 (*sV)[kPitch],
                                             int tid, int nthr) {
  const int L = a.len[b], M = a.rm.start[b + 1] - a.rm.start[b];
  const int p0 = part * kPart;
  if (p0 >= L + M) return;
  const size_t head = (((size_t)layer * a.batch + b) * a.nkv + g) * (size_t)a.cap;
  constexpr int SEGS = D / 8;
  for (int idx = tid; idx < kPart * SEGS; idx += nthr) {
    const int t = idx / SEGS, sg = idx - t * SEGS;
    const int pos = p0 + t;
    if (pos < L) {
      cp_async16(&sK[t][sg * 8], a.kc + (head + pos) * D + sg * 8);
      cp_async16(&sV[t][sg * 8], a.vc + (head + pos) * D + sg * 8);
    } else if (pos >= L + M) {
      *reinterpret_cast<uint4*>(&sK[t][sg * 8]) = make_uint4(0, 0, 0, 0);
      *reinterpret_cast<uint4*>(&sV[t][sg * 8]) = make_uint4(0, 0, 0, 0);
    }
  }
  asm volatile("cp.async.commit_group;" ::: "memory");
}

// Split-KV item: keys [64 part, 64 part + 64) of kv head g of request b for
// all (k + 1) * group queries; writes the partition's (max, sum) and
// unnormalised output per query.  nthr threads (a multiple of 32) of the
// calling group, thread index tid, barrier bar_id; sK/sV hold 64 x kPitch bf16.
// OLD_STAGED: rows [0, L) (and zeros at or beyond L + M) were staged by
// stage_old_kv; only the block's own rows [L, L + M) are copied here.
template <int D, bool OLD_STAGED = false>
__device__ __forceinline__ void part_item(const AttnArgs& a, int layer, int part, int g, int b,
                                          bf16 (*sK)[kPitch], bf16 (*sV)[kPitch], int tid,
                                          int nthr, int bar_id) {
  const int G = a.nq / a.nkv;
  const int r0 = a.rm.start[b], M = a.rm.start[b + 1] - r0;
  const int L = a.len[b];
  const int p0 = part * kPart;
  const int kend = L + M;  // keys [0, L + M) exist once the block's rows are appended
  if (p0 >= kend) return;  // uniform over the CTA
  const int Qn = M * G;

  stage_kv<D>(a, layer, part, g, b, OLD_STAGED ? L : 0, sK, sV, tid, nthr, kend);

  const int warp = tid >> 5, lane = tid & 31;
  const int gq = lane >> 2, tq = lane & 3;
  const int q_dim = a.nq * D;
  const size_t ws_base = ((size_t)(b * a.nkv + g) * a.parts_max + part) * a.qmax;

  // the thread's query elements of a 16-row tile (rows qa = tile*16 + gq and
  // qb = qa + 8), zero for rows past Qn; the first tile's loads are in flight
  // together with the key/value copies
  float2 qv[D / 16][4];
  auto load_q = [&](int tile) {
    const int qa = tile * 16 + gq, qb = qa + 8;
    const bool va = qa < Qn, vb = qb < Qn;
    const int ia = va ? qa / G : 0, ib = vb ? qb / G : 0;
    const float* qpa = a.q + (size_t)(r0 + ia) * q_dim + (size_t)(g * G + (va ? qa % G : 0)) * D;
    const float* qpb = a.q + (size_t)(r0 + ib) * q_dim + (size_t)(g * G + (vb ? qb % G : 0)) * D;
#pragma unroll
    for (int ks = 0; ks < D / 16; ++ks) {
      const int c0 = ks * 16 + 2 * tq;
      qv[ks][0] = va ? *reinterpret_cast<const float2*>(qpa + c0) : make_float2(0.f, 0.f);
      qv[ks][1] = va ? *reinterpret_cast<const float2*>(qpa + c0 + 8) : make_float2(0.f, 0.f);
      qv[ks][2] = vb ? *reinterpret_cast<const float2*>(qpb + c0) : make_float2(0.f, 0.f);
      qv[ks][3] = vb ? *reinterpret_cast<const float2*>(qpb + c0 + 8) : make_float2(0.f, 0.f);
    }
  };
  if (warp * 16 < Qn) load_q(warp);
  asm volatile("cp.async.wait_group 0;" ::: "memory");
  bar_sync(bar_id, nthr);

  for (int tile = warp; tile * 16 < Qn; tile += nthr / 32) {
    // query rows of this tile owned by the thread: qa = tile*16 + gq, qb = qa + 8
    const int qa = tile * 16 + gq, qb = qa + 8;
    const bool va = qa < Qn, vb = qb < Qn;
    const int ia = va ? qa / G : 0, ib = vb ? qb / G : 0;
    if (tile != warp) load_q(tile);

    // S = Q K^T for 64 keys: 8 n-tiles of 8 keys
    float s[8][4];
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
#pragma unroll
    for (int ks = 0; ks < D / 16; ++ks) {
      const int c0 = ks * 16 + 2 * tq;
      const float2 xa0 = qv[ks][0], xa1 = qv[ks][1], xb0 = qv[ks][2], xb1 = qv[ks][3];
      // q as bf16 hi + lo parts: S = Q_hi K^T + Q_lo K^T
      uint32_t ah[4], al[4];
      split_bf16x2(xa0.x * a.qscale, xa0.y * a.qscale, ah[0], al[0]);
      split_bf16x2(xb0.x * a.qscale, xb0.y * a.qscale, ah[1], al[1]);
      split_bf16x2(xa1.x * a.qscale, xa1.y * a.qscale, ah[2], al[2]);
      split_bf16x2(xb1.x * a.qscale, xb1.y * a.qscale, ah[3], al[3]);
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) {
        const uint32_t b0 = *reinterpret_cast<const uint32_t*>(&sK[nt * 8 + gq][c0]);
        const uint32_t b1 = *reinterpret_cast<const uint32_t*>(&sK[nt * 8 + gq][c0 + 8]);
        mma_16816(s[nt], ah, b0, b1);
        mma_16816(s[nt], al, b0, b1);
      }
    }
    // causal mask: row i sees keys up to L + i
    const int lima = va ? L + ia : -1, limb = vb ? L + ib : -1;
    float ma = -INFINITY, mb = -INFINITY;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      const int t0 = p0 + nt * 8 + 2 * tq;
      if (t0 > lima) s[nt][0] = -INFINITY;
      if (t0 + 1 > lima) s[nt][1] = -INFINITY;
      if (t0 > limb) s[nt][2] = -INFINITY;
      if (t0 + 1 > limb) s[nt][3] = -INFINITY;
      ma = fmaxf(ma, fmaxf(s[nt][0], s[nt][1]));
      mb = fmaxf(mb, fmaxf(s[nt][2], s[nt][3]));
    }
    ma = fmaxf(ma, __shfl_xor_sync(0xFFFFFFFFu, ma, 1));
    ma = fmaxf(ma, __shfl_xor_sync(0xFFFFFFFFu, ma, 2));
    mb = fmaxf(mb, __shfl_xor_sync(0xFFFFFFFFu, mb, 1));
    mb = fmaxf(mb, __shfl_xor_sync(0xFFFFFFFFu, mb, 2));
    const float sa = (ma == -INFINITY) ? 0.f : ma, sb = (mb == -INFINITY) ? 0.f : mb;
    float la = 0.f, lb = 0.f;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      s[nt][0] = exp2f(s[nt][0] - sa);
      s[nt][1] = exp2f(s[nt][1] - sa);
      s[nt][2] = exp2f(s[nt][2] - sb);
      s[nt][3] = exp2f(s[nt][3] - sb);
      la += s[nt][0] + s[nt][1];
      lb += s[nt][2] + s[nt][3];
    }
    la += __shfl_xor_sync(0xFFFFFFFFu, la, 1);
    la += __shfl_xor_sync(0xFFFFFFFFu, la, 2);
    lb += __shfl_xor_sync(0xFFFFFFFFu, lb, 1);
    lb += __shfl_xor_sync(0xFFFFFFFFu, lb, 2);

    // O = P V: P from the S accumulators (16 x 64), V (64 x D) via ldmatrix.trans
    // P as bf16 hi + lo parts: O = P_hi V + P_lo V
    uint32_t pf[4][4], pl[4][4];
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      split_bf16x2(s[2 * kk][0], s[2 * kk][1], pf[kk][0], pl[kk][0]);
      split_bf16x2(s[2 * kk][2], s[2 * kk][3], pf[kk][1], pl[kk][1]);
      split_bf16x2(s[2 * kk + 1][0], s[2 * kk + 1][1], pf[kk][2], pl[kk][2]);
      split_bf16x2(s[2 * kk + 1][2], s[2 * kk + 1][3], pf[kk][3], pl[kk][3]);
    }
    const int lr = lane & 7, lm = lane >> 3;
#pragma unroll
    for (int dp = 0; dp < D / 16; ++dp) {  // pairs of 8-column output tiles
      float o0[4] = {0.f, 0.f, 0.f, 0.f}, o1[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        uint32_t vb4[4];
        ldmatrix_x4_trans(vb4, &sV[kk * 16 + lr + (lm & 1) * 8][dp * 16 + (lm >> 1) * 8]);
        mma_16816(o0, pf[kk], vb4[0], vb4[1]);
        mma_16816(o0, pl[kk], vb4[0], vb4[1]);
        mma_16816(o1, pf[kk], vb4[2], vb4[3]);
        mma_16816(o1, pl[kk], vb4[2], vb4[3]);
      }
      const int col = dp * 16 + 2 * tq;
      if (va) {
        float* dst = a.ws_o + (ws_base + qa) * D;
        *reinterpret_cast<float2*>(dst + col) = make_float2(o0[0], o0[1]);
        *reinterpret_cast<float2*>(dst + col + 8) = make_float2(o1[0], o1[1]);
      }
      if (vb) {
        float* dst = a.ws_o + (ws_base + qb) * D;
        *reinterpret_cast<float2*>(dst + col) = make_float2(o0[2], o0[3]);
        *reinterpret_cast<float2*>(dst + col + 8) = make_float2(o1[2], o1[3]);
      }
    }
    if (tq == 0) {
      if (va) a.ws_ml[ws_base + qa] = make_float2(ma, la);
      if (vb) a.ws_ml[ws_base + qb] = make_float2(mb, lb);
    }
  }
  bar_sync(bar_id, nthr);  // staging buffers free for the group's next item
}

// Combine the partitions of one (row, query head).  Warp 0 reads the
// partitions' (max, sum) pairs 32 at a time (one round trip per 32), forms the
// weights 2^(m_p - M) in shared memory and the total; then every thread (one
// output element) adds its partitions' outputs, 32 loads in flight, in
// partition order.  Every order is fixed by the number of partitions alone.
constexpr int kMaxParts = 1024;  // capacity <= 65536 positions

// Merge item for token row r and query head j; w holds kMaxParts floats and
// s_l one float of shared memory.  Needs nthr >= D.
template <int D, int PF = 32>
__device__ __forceinline__ void merge_item(const AttnArgs& a, int r, int j, float* w, float* s_l,
                                           int tid, int nthr, int bar_id) {
  // PF partitions' loads are in flight at a time; the sum runs in partition
  // order whatever PF is
  const int e = tid;
  const int G = a.nq / a.nkv;
  const int b = row_request(a.rm, r);
  const int i = r - a.rm.start[b];
  const int g = j / G, qr = i * G + (j - g * G);
  const int pos = a.len[b] + i;
  const int nparts = pos / kPart + 1;
  const size_t base = (size_t)(b * a.nkv + g) * a.parts_max * a.qmax + qr;
  // the first PF partitions' outputs and the first 32 (max, sum) pairs are
  // loaded together: one round trip while nparts <= min(PF, 32)
  float ov[PF];
  if (e < D) {
#pragma unroll
    for (int u = 0; u < PF; ++u)
      ov[u] = (u < nparts) ? a.ws_o[(base + (size_t)u * a.qmax) * D + e] : 0.f;
  }
  if (e < 32) {
    const float2 ml0 = e < nparts ? a.ws_ml[base + (size_t)e * a.qmax] : make_float2(-INFINITY, 0.f);
    float M = ml0.x;
    for (int p0 = 32; p0 < nparts; p0 += 32) {
      const int pp = p0 + e;
      const float mp = pp < nparts ? a.ws_ml[base + (size_t)pp * a.qmax].x : -INFINITY;
      M = fmaxf(M, mp);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xFFFFFFFFu, M, o));
    float l = 0.f;
    for (int p0 = 0; p0 < nparts; p0 += 32) {
      const int pp = p0 + e;
      if (pp < nparts) {
        const float2 ml = p0 == 0 ? ml0 : a.ws_ml[base + (size_t)pp * a.qmax];
        const float wp = (ml.x == -INFINITY) ? 0.f : exp2f(ml.x - M);
        w[pp] = wp;
        l += ml.y * wp;
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) l += __shfl_xor_sync(0xFFFFFFFFu, l, o);
    if (e == 0) *s_l = l;
  }
  bar_sync(bar_id, nthr);
  if (e < D) {
  float o = 0.f;
  for (int p0 = 0; p0 < nparts; p0 += PF) {
    if (p0 > 0) {
#pragma unroll
      for (int u = 0; u < PF; ++u)
        ov[u] = (p0 + u < nparts) ? a.ws_o[(base + (size_t)(p0 + u) * a.qmax) * D + e] : 0.f;
    }
#pragma unroll
    for (int u = 0; u < PF; ++u)
      if (p0 + u < nparts) o += ov[u] * w[p0 + u];
  }
  const float ov_ = o / *s_l;
  const bf16 oh = __float2bfloat16_rn(ov_);
  a.ao[(size_t)r * a.nq * D + (size_t)j * D + e] = oh;
  a.ao[(size_t)(a.lo_row + r) * a.nq * D + (size_t)j * D + e] =
      __float2bfloat16_rn(ov_ - __bfloat162float(oh));
  }
  bar_sync(bar_id, nthr);  // w and s_l free for the group's next item
}

}  // namespace attn
}  // namespace as2d
