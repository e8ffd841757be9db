// k_attn.cu -- grouped-query attention of a verification block over the
// retained prefix (Section 3.2: one causal pass over the root and the
// candidates; App. C.4: rows attend to the committed prefix and to the
// block's own earlier rows).
//
// Row i of request b sits at position L_b + i and attends to keys [0, L_b + i].
// All G = n_q / n_kv query heads of a key/value head, for all rows of the
// request, form one query matrix of M * G rows, so each key/value entry is
// read from HBM once per block (twice when a request has more than 64 query
// rows, the second time from L2).
//
// qkv_finish_kernel: the QKV projection arrives as split-K partial sums
// (TC_PART); one CTA per (token row, head) adds them in rank order, scales by
// the row's 1 / rms and rotates (RoPE).  Keys and values are appended to the
// cache; queries, scaled by log2(e) / sqrt(d), are written as bf16 hi and lo
// parts straight into the tensor-core operand image of their (request, kv
// head, 64-query tile): 128 rows (row 2q the hi part of query q, row 2q + 1
// its lo part) of d elements in the 128-byte-swizzled K-major layout, one
// 16 KB region per 64 columns.
//
// attn_tc_kernel: one CTA per 128-key tile of one (request, kv head, query
// tile); a cluster of 8 CTAs covers one chunk of 1024 keys.  Per CTA:
//   * the tile's keys and values arrive by TMA (3D map over the cache, 128-
//     byte swizzle; tiles holding only entries older than this call are
//     requested before the wait for the finishing kernel), the query image
//     by one bulk copy;
//   * S = Q K^T on tcgen05 (M = 128: the hi and lo rows of 64 queries
//     interleaved, N = 128 keys) into TMEM; thread t reads lane t, so each
//     query's hi and lo scores sit in adjacent lanes of one warp and are
//     added by a shuffle, each lane keeping half of the keys; masking (causal,
//     and keys past the call's end) and P = 2^(S - m) with the tile's own
//     maximum m and sum l;
//   * O = P V on tcgen05 (P's hi and lo rows interleaved the same way, as
//     the A operand in TMEM over S, or in the narrow layout as a shared-memory
//     image over Q; B = V read MN-major from the TMA image); hi + lo added by
//     a shuffle, each lane keeping half of the dims;
//   * the tile partials (m, l, O) are pushed through distributed shared
//     memory to the CTA that folds their query rows (CTA r: rows 8r..8r+7),
//     which folds the chunk's 8 tiles in tile order.  With one chunk the
//     result is normalised and written (bf16 hi, lo).  With two chunks in a
//     cluster of 16 (PAIR), CTA r receives rows 4r..4r+3 from all 16 tiles
//     and folds each chunk's tiles, then the two chunks.  Otherwise the
//     CTA's rows of the chunk partial go to memory and the last CTA of those
//     rows to arrive, over the chunks of the (request, kv head, query tile),
//     folds them in chunk order (9 to 15 chunks staged in shared memory).
// Shared-memory layouts (the same arithmetic): wide, K and V in their own
// images, two CTAs per SM; NARROW, V loaded over K once the first product is
// done (from L2, where the launch is small enough to prefetch it) and O
// accumulated over S in TMEM, three CTAs per SM, for launches of more
// clusters than the wide layout serves well; and attn_tc4_kernel, four CTAs
// per SM in 48 KB, for launches of more clusters than the narrow layout
// keeps resident.
// Every fold boundary is a fixed absolute key position (128-key tiles,
// 1024-key chunks), and a fold with a part a row cannot see (fully masked:
// m = -inf, l = 0, O = 0) leaves it bitwise unchanged, so a row's result does
// not depend on the other rows of the call (batch invariance).
#include "as2d_internal.h"
#include "ptx_sm100.cuh"

namespace as2d {
namespace {

constexpr int kTile = 128;    // keys per CTA
constexpr int kCluster = 8;   // CTAs per cluster
constexpr int kChunk = kTile * kCluster;
constexpr int kQT = 64;       // queries per query tile (hi and lo rows interleaved)
constexpr uint32_t kRegion = 128 * 128;  // one 64-column region of 128 rows, bytes
// chunks whose partial rows the last arriver stages in shared memory: [15][8
// rows][128] floats and [15][8] (max, sum) within the first two 32 KB images
constexpr int kStage = 15;
static_assert(kStage * 8 * 128 * 4 + kStage * 8 * 8 <= 2 * 32768, "staging fits two images");
// Shared memory: the Q / P image, then the K and V tiles.  Wide (launches of
// up to kWideClusters clusters of 8): K and V in separate images, both
// requested at the start.  Narrow (larger launches): V is loaded over K once
// the first product has consumed it, so that three CTAs fit on an SM.
// Pair (wide only): clusters of 16 CTAs over two chunks, each CTA folding 4
// query rows of both, so that the chunks fold without going through global
// memory.
template <bool NARROW, bool PAIR>
constexpr uint32_t attn_smem() {
  return (NARROW ? 2 : 3) * 32768 + 64 * 8 + 8 * 4 + 5 * 8 + 16 + 1024;
}
static_assert(3 * (attn_smem<true, false>() + 1024) <= 228 * 1024, "three narrow CTAs per SM");
static_assert(2 * (attn_smem<false, true>() + 1024) <= 228 * 1024, "two wide CTAs per SM");
// A launch of more clusters of 8 than this takes the narrow layout.  The wide
// kernel's shared memory allows 36 clusters of 8 at two CTAs per SM (the
// occupancy calculator reports 15); measured on 7B and 1.5B calls, the wide
// layout is the faster up to 32 clusters and much the slower at 36.
constexpr int kWideClusters = 32;
// clusters of 8 the narrow layout keeps resident (three CTAs per SM, residency
// probe); larger launches take four CTAs per SM
constexpr int kNarrowClusters = 51;

struct AttnArgs {
  RowMap rm;
  const int32_t* len;
  int layer, batch, cap, nq, nkv;
  float qscale;  // log2(e) / sqrt(d), folded into the stored queries
  // split-K sums of the QKV projection (TC_PART)
  const float* qkv_part;  // [tile][split][qkv_ld][128], tile = column / 128
  const float* qkv_rinv;  // [qkv_ld] 1 / rms of each token row
  const float2* rope;     // [rows][d / 2] (cos, sin)
  int qkv_split, qkv_ld;
  bf16* kc;
  bf16* vc;
  uint8_t* qimg;          // [batch][nkv][qt_max] operand images, 256 d bytes each
  int qt_max;
  float* ws_o;            // [batch][nkv][qt_max][chunks_max][64][d] chunk partials
  float2* ws_ml;          // [batch][nkv][qt_max][chunks_max][64] (max, sum), base 2
  int chunks_max;
  int* cnt;               // [batch][nkv][qt_max][8] chunks arrived per 8-row group
  bf16* ao;               // [2 rows][nq d]: hi rows, then lo rows from lo_row
  int lo_row;
  int32_t* err;
  unsigned long long timeout_ns;
  int v_prefetch;         // narrow and quad: bring each tile's V into L2 with its K
  // clusters of request b: [cl_start[b], cl_start[b + 1]); n_ch[b] of them per
  // query tile (chunks covering the host's bound of the request's keys)
  int32_t cl_start[kMaxBatch + 1];
  int32_t n_ch[kMaxBatch];
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

// Byte offset of element (row r, column e) in a 128-row operand image of
// 128-byte-swizzled K-major bf16: 64-column regions of kRegion bytes, 16-byte
// chunk j of row r stored at chunk j ^ (r mod 8).
__device__ __forceinline__ uint32_t img_off(int r, int e) {
  const int reg = e >> 6, j = (e & 63) >> 3;
  return (uint32_t)reg * kRegion + (uint32_t)r * 128u + (uint32_t)((j ^ (r & 7)) << 4) +
         (uint32_t)((e & 7) << 1);
}

// One CTA of D / 2 threads per (token row, head); thread e forms the pair
// (e, e + D/2).  Rotate-half RoPE: x' = x cos - x_p sin at e, x_p cos + x sin
// at e + D/2.
template <int D>
__global__ void __launch_bounds__(D / 2) qkv_finish_kernel(AttnArgs a) {
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  constexpr int H2 = D / 2;
  const int gm = blockIdx.x, head = blockIdx.y, e = threadIdx.x;
  const int b = row_request(a.rm, gm), i = gm - a.rm.start[b];
  // every load is issued before any is used: one memory round trip
  const int len_b = a.len[b];
  const float x = qkv_value(a, head * D + e, gm), xp = qkv_value(a, head * D + e + H2, gm);
  const bool rotate = head < a.nq + a.nkv;
  const float2 cs = rotate ? a.rope[(size_t)gm * H2 + e] : make_float2(1.f, 0.f);
  if (!rows_fit(len_b, a.rm.start[b + 1] - a.rm.start[b], a.cap)) return;  // flagged
  const int pos = len_b + i;
  float y0, y1;
  if (rotate) {
    y0 = fmaf(x, cs.x, -(xp * cs.y));
    y1 = fmaf(xp, cs.x, x * cs.y);
  } else {
    y0 = x;
    y1 = xp;
  }
  if (head < a.nq) {
    const int G = a.nq / a.nkv, g = head / G;
    const int qg = i * G + (head - g * G);
    const int qt = qg / kQT, q = qg - qt * kQT;
    uint8_t* img = a.qimg + ((size_t)(b * a.nkv + g) * a.qt_max + qt) * (size_t)(256 * D);
    const float v0 = y0 * a.qscale, v1 = y1 * a.qscale;
    const bf16 h0 = __float2bfloat16_rn(v0), h1 = __float2bfloat16_rn(v1);
    *reinterpret_cast<bf16*>(img + img_off(2 * q, e)) = h0;
    *reinterpret_cast<bf16*>(img + img_off(2 * q, e + H2)) = h1;
    *reinterpret_cast<bf16*>(img + img_off(2 * q + 1, e)) =
        __float2bfloat16_rn(v0 - __bfloat162float(h0));
    *reinterpret_cast<bf16*>(img + img_off(2 * q + 1, e + H2)) =
        __float2bfloat16_rn(v1 - __bfloat162float(h1));
  } else {
    const bool is_k = head < a.nq + a.nkv;
    const int g = is_k ? head - a.nq : head - a.nq - a.nkv;
    bf16* dst = (is_k ? a.kc : a.vc) + ((((size_t)a.layer * a.batch + b) * a.nkv + g) * a.cap + pos) * D;
    dst[e] = __float2bfloat16_rn(y0);
    dst[e + H2] = __float2bfloat16_rn(y1);
  }
}

// ---- attention over 128-key tiles on the tensor cores ------------------------

// 2^x on the special-function unit (ftz: results below 2^-126 are 0).
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Values x[0..7] (>= 0) of columns e0..e0+7 (e0 % 8 == 0) of query q, as bf16
// hi parts into row 2q and lo parts into row 2q + 1 of an operand image: hi =
// x with its low 16 bits cleared (exact in bf16), lo = bf16(x - hi), so that
// hi + lo matches x to about 17 bits.  A thread of the odd half (pt = 1)
// stores its lo row first: the two rows of one store instruction then cover
// all eight 16-byte positions of the swizzle, not four.
__device__ __forceinline__ void put_hilo8(uint8_t* img, int q, int pt, int e0, const float* x) {
  uint32_t hw[4], lw[4];
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const uint32_t b0 = __float_as_uint(x[2 * u]), b1 = __float_as_uint(x[2 * u + 1]);
    hw[u] = (b0 >> 16) | (b1 & 0xFFFF0000u);
    const __nv_bfloat162 lv = __floats2bfloat162_rn(x[2 * u] - __uint_as_float(b0 & 0xFFFF0000u),
                                                    x[2 * u + 1] - __uint_as_float(b1 & 0xFFFF0000u));
    lw[u] = *reinterpret_cast<const uint32_t*>(&lv);
  }
  const uint4 h = make_uint4(hw[0], hw[1], hw[2], hw[3]), l = make_uint4(lw[0], lw[1], lw[2], lw[3]);
  *reinterpret_cast<uint4*>(img + img_off(2 * q + pt, e0)) = pt ? l : h;
  *reinterpret_cast<uint4*>(img + img_off(2 * q + 1 - pt, e0)) = pt ? h : l;
}

__device__ __forceinline__ void dsmem_st_f4(uint32_t addr, float4 v) {
  asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "f"(v.x), "f"(v.y),
               "f"(v.z), "f"(v.w)
               : "memory");
}

__device__ __forceinline__ void dsmem_st_f2(uint32_t addr, float2 v) {
  asm volatile("st.shared::cluster.v2.f32 [%0], {%1, %2};" ::"r"(addr), "f"(v.x), "f"(v.y)
               : "memory");
}

// 128 columns of this thread's TMEM lane starting at taddr: two loads, one
// wait.
__device__ __forceinline__ void tmem_ld128(uint32_t taddr, float (&v0)[64], float (&v1)[64]) {
  uint32_t a[64], b[64];
  ptx::tmem_ld_x64(taddr, a);
  ptx::tmem_ld_x64(taddr + 64, b);
  ptx::tmem_ld_wait();
#pragma unroll
  for (int j = 0; j < 64; ++j) {
    v0[j] = __uint_as_float(a[j]);
    v1[j] = __uint_as_float(b[j]);
  }
}

// 64 columns of this thread's TMEM lane starting at `col`, into v.
__device__ __forceinline__ void tmem_ld64(uint32_t taddr, float (&v)[64]) {
  uint32_t a[64];
  ptx::tmem_ld_x64(taddr, a);
  ptx::tmem_ld_wait();
#pragma unroll
  for (int j = 0; j < 64; ++j) v[j] = __uint_as_float(a[j]);
}

// The weight of a part (max m) in a fold whose maximum is M: 2^(m - M), 0
// where m = -inf (nothing of the part is visible to the row), exactly 1 for
// the part holding the maximum.  Parts of weight 0 are skipped by the folds,
// so a part a row cannot see leaves its result bitwise unchanged.
__device__ __forceinline__ float part_weight(float m, float M) {
  return m == -INFINITY ? 0.f : (m == M ? 1.f : ex2(m - M));
}

// The tile's scores of this thread's 64 keys kb .. kb + 63 (hi + lo, in sv)
// -> P = 2^(S - m) in sv (visible keys: key <= lim; a masked key gets 0,
// never -inf), with the tile's maximum m and sum l over both halves of the
// keys (the partner lane holds the other half).
__device__ __forceinline__ void softmax_tail(float (&sv)[64], int pt, int kb, int lim, float& m,
                                             float& l) {
  // a half-tile wholly at or below the row's limit needs no mask
  const bool all_vis = kb + 63 <= lim;
  float mx4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
  if (all_vis) {
#pragma unroll
    for (int j = 0; j < 64; ++j) mx4[j & 3] = fmaxf(mx4[j & 3], sv[j]);
  } else {
#pragma unroll
    for (int j = 0; j < 64; ++j)
      if (kb + j <= lim) mx4[j & 3] = fmaxf(mx4[j & 3], sv[j]);
  }
  const float mx = fmaxf(fmaxf(mx4[0], mx4[1]), fmaxf(mx4[2], mx4[3]));
  m = fmaxf(mx, __shfl_xor_sync(0xFFFFFFFFu, mx, 1));
  // sums in four interleaved parts, then ((0 + 1) + (2 + 3)): a fixed order
  float ls4[4] = {0.f, 0.f, 0.f, 0.f};
  if (all_vis) {
#pragma unroll
    for (int j = 0; j < 64; ++j) {
      sv[j] = ex2(sv[j] - m);
      ls4[j & 3] += sv[j];
    }
  } else {
#pragma unroll
    for (int j = 0; j < 64; ++j) {
      sv[j] = (kb + j <= lim) ? ex2(sv[j] - m) : 0.f;
      ls4[j & 3] += sv[j];
    }
  }
  const float ls = (ls4[0] + ls4[1]) + (ls4[2] + ls4[3]);
  const float lo_ = __shfl_xor_sync(0xFFFFFFFFu, ls, 1);
  l = pt ? lo_ + ls : ls + lo_;  // keys 0..63, then 64..127
}

// Dims [fd, fd + DT) of row fr of query tile qt, normalised (o / l), as
// bf16 hi and lo parts into the attention output; rows past the call's
// queries are skipped.
template <int D, int DT>
__device__ __forceinline__ void write_rows(const AttnArgs& a, const float* o_, float Ls, int fr,
                                           int fd, int qt, int qn, int G, int g, int r0) {
  const int fqg = qt * kQT + fr;
  if (fqg >= qn) return;
  const int i = fqg / G, hq = g * G + (fqg - i * G);
  const size_t at = (size_t)(r0 + i) * a.nq * D + (size_t)hq * D + fd;
  uint32_t hw[DT / 2], lw[DT / 2];
#pragma unroll
  for (int e = 0; e < DT / 2; ++e) {
    const float v0 = o_[2 * e] / Ls, v1 = o_[2 * e + 1] / Ls;
    const __nv_bfloat162 hv = __floats2bfloat162_rn(v0, v1);
    const float2 hf = __bfloat1622float2(hv);
    const __nv_bfloat162 lv = __floats2bfloat162_rn(v0 - hf.x, v1 - hf.y);
    hw[e] = *reinterpret_cast<const uint32_t*>(&hv);
    lw[e] = *reinterpret_cast<const uint32_t*>(&lv);
  }
#pragma unroll
  for (int u = 0; u < DT / 8; ++u) {
    *reinterpret_cast<uint4*>(a.ao + at + 8 * u) =
        make_uint4(hw[4 * u], hw[4 * u + 1], hw[4 * u + 2], hw[4 * u + 3]);
    *reinterpret_cast<uint4*>(a.ao + (size_t)a.lo_row * a.nq * D + at + 8 * u) =
        make_uint4(lw[4 * u], lw[4 * u + 1], lw[4 * u + 2], lw[4 * u + 3]);
  }
  if (DT % 8) {  // four dims
    *reinterpret_cast<uint2*>(a.ao + at) = make_uint2(hw[0], hw[1]);
    *reinterpret_cast<uint2*>(a.ao + (size_t)a.lo_row * a.nq * D + at) = make_uint2(lw[0], lw[1]);
  }
}

// The fold of a chunk's 8 tile partials for query rows 8 rank .. 8 rank + 7
// (received into s_rml [8 tiles][8 rows] and recv [8 tiles][8 rows][D]) and
// what follows it: with one chunk the rows are normalised and written; with
// several, the rows of the chunk partial go to memory and the last CTA of
// these rows to arrive folds the chunks in chunk order (9 to stage_max chunks
// staged in shared memory at sm, whose images are no longer read).
template <int D>
__device__ __forceinline__ void fold_chunk8(const AttnArgs& a, const float* recv,
                                            const float2* s_rml, int* s_flag, uint8_t* sm,
                                            int stage_max, uint32_t rank, int c, int n_tiles,
                                            int n_chunks, int b, int g, int qt, int qn, int G,
                                            int r0) {
  constexpr int DT = D / 16;  // dims per thread (8 rows x 16 threads)
  const int tid = threadIdx.x;
  // ---- fold (thread: query row 8 rank + fj, dims [fd, fd + DT)) ----------
  const int n_here = min(kCluster, n_tiles - c * kCluster);  // tiles of this chunk with keys
  const int fj = tid >> 4, fr = 8 * (int)rank + fj, fd = DT * (tid & 15);
  float fm = -INFINITY;
  float2 pml[kCluster];
#pragma unroll
  for (int i = 0; i < kCluster; ++i) {
    pml[i] = (i < n_here) ? s_rml[i * 8 + fj] : make_float2(-INFINITY, 0.f);
    fm = fmaxf(fm, pml[i].x);
  }
  float fl = 0.f, fo[DT];
#pragma unroll
  for (int e = 0; e < DT; ++e) fo[e] = 0.f;
#pragma unroll
  for (int i = 0; i < kCluster; ++i) {
    const float w = part_weight(pml[i].x, fm);
    if (w != 0.f) {
      fl += pml[i].y * w;
      const float4* src = reinterpret_cast<const float4*>(recv + (i * 8 + fj) * D + fd);
#pragma unroll
      for (int u = 0; u < DT / 4; ++u) {
        const float4 v = src[u];
        fo[4 * u + 0] += v.x * w;
        fo[4 * u + 1] += v.y * w;
        fo[4 * u + 2] += v.z * w;
        fo[4 * u + 3] += v.w * w;
      }
    }
  }
  // normalise and write the row's dims (o / l as bf16 hi, lo)
  auto write_out = [&](const float* o_, float Ls) {
    write_rows<D, DT>(a, o_, Ls, fr, fd, qt, qn, G, g, r0);
  };
  if (n_chunks == 1) {
    write_out(fo, fl);
    return;
  }
  // ---- several chunks: this CTA's rows of the chunk partial go to memory;
  // the last chunk's CTA of these rows to arrive folds them in chunk order
  const size_t item = (size_t)(b * a.nkv + g) * a.qt_max + qt;
  {
    const size_t pc = item * a.chunks_max + c;
    float4* dst = reinterpret_cast<float4*>(a.ws_o + (pc * kQT + fr) * D + fd);
#pragma unroll
    for (int u = 0; u < DT / 4; ++u)
      dst[u] = make_float4(fo[4 * u], fo[4 * u + 1], fo[4 * u + 2], fo[4 * u + 3]);
    if ((tid & 15) == 0) a.ws_ml[pc * kQT + fr] = make_float2(fm, fl);
  }
  __syncthreads();
  int* cnt = a.cnt + item * kCluster + rank;
  if (tid == 0) {
    // the arrival releases the CTA's writes above (ordered before it by the
    // barrier) and acquires the other chunks' partials for the last arriver
    int prev;
    asm volatile("atom.add.acq_rel.gpu.s32 %0, [%1], 1;" : "=r"(prev) : "l"(cnt) : "memory");
    const int last = prev == n_chunks - 1;
    if (last) *cnt = 0;  // every chunk of these rows has arrived
    *s_flag = last;
  }
  __syncthreads();
  if (!*s_flag) return;
  float cl_ = 0.f, co[DT];
#pragma unroll
  for (int e = 0; e < DT; ++e) co[e] = 0.f;
  if (n_chunks > 8 && n_chunks <= stage_max) {
    // nine or more chunks: every chunk's rows come into shared memory (over
    // the Q / P and K images, no longer read) by copies issued together, one
    // memory round trip instead of two through registers
    float* st_o = reinterpret_cast<float*>(sm);                          // [chunk][8 rows][D]
    float2* st_ml = reinterpret_cast<float2*>(sm + stage_max * 8 * D * 4);  // [chunk][8 rows]
    for (int cc = 0; cc < n_chunks; ++cc) {
      const size_t pc = item * a.chunks_max + cc;
      const float* src = a.ws_o + (pc * kQT + fr) * D + fd;
      float* dst = st_o + (cc * 8 + fj) * D + fd;
#pragma unroll
      for (int u = 0; u < DT / 4; ++u) ptx::cp_async16(dst + 4 * u, src + 4 * u);
      // (max, sum) of rows fj and fj + 1 in one copy
      if ((tid & 15) == 0 && (fj & 1) == 0) ptx::cp_async16(st_ml + cc * 8 + fj, a.ws_ml + pc * kQT + fr);
    }
    ptx::cp_async_wait_all();
    __syncthreads();
    float cm = -INFINITY;
    for (int cc = 0; cc < n_chunks; ++cc) cm = fmaxf(cm, st_ml[cc * 8 + fj].x);
    for (int cc = 0; cc < n_chunks; ++cc) {
      const float2 ml = st_ml[cc * 8 + fj];
      const float w = part_weight(ml.x, cm);
      if (w != 0.f) {
        cl_ += ml.y * w;
        const float4* src = reinterpret_cast<const float4*>(st_o + (cc * 8 + fj) * D + fd);
#pragma unroll
        for (int u = 0; u < DT / 4; ++u) {
          const float4 v = src[u];
          co[4 * u + 0] += v.x * w;
          co[4 * u + 1] += v.y * w;
          co[4 * u + 2] += v.z * w;
          co[4 * u + 3] += v.w * w;
        }
      }
    }
    write_out(co, cl_);
    return;
  }
  // eight chunks' values in flight at a time; the first eight are requested
  // together with every chunk's maximum, so that up to eight chunks take one
  // memory round trip
  float4 v[8][DT / 4];
  float2 ml[8];
  auto load8 = [&](int c0) {
#pragma unroll
    for (int u8 = 0; u8 < 8; ++u8)
      if (c0 + u8 < n_chunks) {
        const size_t pc = item * a.chunks_max + c0 + u8;
        ml[u8] = __ldcg(a.ws_ml + pc * kQT + fr);
        const float4* src = reinterpret_cast<const float4*>(a.ws_o + (pc * kQT + fr) * D + fd);
#pragma unroll
        for (int u = 0; u < DT / 4; ++u) v[u8][u] = __ldcg(src + u);
      }
  };
  // more chunks than shared memory holds, but no more than eight plus that:
  // chunks 8.. come into shared memory by copies issued together with the
  // first eight's loads, so that all of them take one memory round trip
  const bool hybrid = n_chunks > 8 && n_chunks - 8 <= stage_max;
  float* st_o = reinterpret_cast<float*>(sm);                          // [chunk - 8][8 rows][D]
  float2* st_ml = reinterpret_cast<float2*>(sm + stage_max * 8 * D * 4);  // [chunk - 8][8 rows]
  if (hybrid) {
    for (int cc = 8; cc < n_chunks; ++cc) {
      const size_t pc = item * a.chunks_max + cc;
      const float* src = a.ws_o + (pc * kQT + fr) * D + fd;
      float* dst = st_o + ((cc - 8) * 8 + fj) * D + fd;
#pragma unroll
      for (int u = 0; u < DT / 4; ++u) ptx::cp_async16(dst + 4 * u, src + 4 * u);
      if ((tid & 15) == 0 && (fj & 1) == 0)
        ptx::cp_async16(st_ml + (cc - 8) * 8 + fj, a.ws_ml + pc * kQT + fr);
    }
  }
  load8(0);
  float cm = -INFINITY;
  for (int cc = 8; cc < n_chunks; ++cc)
    cm = fmaxf(cm, __ldcg(a.ws_ml + (item * a.chunks_max + cc) * kQT + fr).x);
#pragma unroll
  for (int u8 = 0; u8 < 8; ++u8)
    if (u8 < n_chunks) cm = fmaxf(cm, ml[u8].x);
  for (int c0 = 0; c0 < n_chunks; c0 += 8) {
    if (hybrid && c0 == 8) {
      ptx::cp_async_wait_all();
      __syncthreads();
      for (int cc = 8; cc < n_chunks; ++cc) {
        const float2 mlc = st_ml[(cc - 8) * 8 + fj];
        const float w = part_weight(mlc.x, cm);
        if (w != 0.f) {
          cl_ += mlc.y * w;
          const float4* src = reinterpret_cast<const float4*>(st_o + ((cc - 8) * 8 + fj) * D + fd);
#pragma unroll
          for (int u = 0; u < DT / 4; ++u) {
            const float4 vv = src[u];
            co[4 * u + 0] += vv.x * w;
            co[4 * u + 1] += vv.y * w;
            co[4 * u + 2] += vv.z * w;
            co[4 * u + 3] += vv.w * w;
          }
        }
      }
      break;
    }
    if (c0 > 0) load8(c0);
#pragma unroll
    for (int u8 = 0; u8 < 8; ++u8)
      if (c0 + u8 < n_chunks) {
        const float w = part_weight(ml[u8].x, cm);
        if (w != 0.f) {
          cl_ += ml[u8].y * w;
#pragma unroll
          for (int u = 0; u < DT / 4; ++u) {
            co[4 * u + 0] += v[u8][u].x * w;
            co[4 * u + 1] += v[u8][u].y * w;
            co[4 * u + 2] += v[u8][u].z * w;
            co[4 * u + 3] += v[u8][u].w * w;
          }
        }
      }
  }
  write_out(co, cl_);
}

template <int D, bool NARROW, bool PAIR>
__global__ void __launch_bounds__(128, NARROW ? 3 : 2)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                   const __grid_constant__ AttnArgs a) {
  constexpr int NR = D / 64;          // 64-column regions of a K / V tile
  constexpr uint32_t K_BYTES = NR * kRegion;            // one K or V tile
  constexpr uint32_t TMEM_COLS = NARROW ? 128 : 256;   // narrow: O over S
  constexpr uint32_t Q_BYTES = 2u * kQT * D * 2;
  constexpr int DH = D / 2;           // dims each thread of a hi/lo pair keeps
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* R0 = sm;            // Q image -> P image
  uint8_t* R1 = sm + 32768;    // K tile -> the partials received from the cluster
  uint8_t* R2 = NARROW ? R1 : sm + 65536;  // V tile (narrow: over K, after the first product)
  float* recv = reinterpret_cast<float*>(R1);  // [8 tiles][8 rows][D] received
  // [tiles of the cluster][rows folded here] (max, sum): [8][8], pair [16][4]
  float2* s_rml = reinterpret_cast<float2*>(sm + (NARROW ? 2 : 3) * 32768);
  float* s_x = reinterpret_cast<float*>(s_rml + 64);      // [8] scratch
  uint64_t* bars = reinterpret_cast<uint64_t*>(s_x + 8);  // q, k (wide: and v), mma1, mma2, v
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bars + 5);
  int* s_flag = reinterpret_cast<int*>(tslot + 1);

  const int tid = threadIdx.x, warp = tid >> 5;
  // a cluster covers HALVES chunks of 8 tiles; half: this CTA's chunk of
  // them, rank: its tile within the chunk
  constexpr int HALVES = PAIR ? 2 : 1;
  const uint32_t crank = ptx::cluster_rank();
  const int half = (int)(crank >> 3);
  const uint32_t rank = crank & 7u;
  const int cl = (int)(blockIdx.x / (kCluster * HALVES)), g = blockIdx.y;
  int b = 0;
  while (b + 1 < a.rm.batch && a.cl_start[b + 1] <= cl) ++b;
  const int ci = cl - a.cl_start[b];
  const int ncl = (a.n_ch[b] + HALVES - 1) / HALVES;  // clusters per query tile
  const int qt = ci / ncl, c2 = ci - qt * ncl;
  const int c = c2 * HALVES + half;  // this CTA's chunk
  const int t = c * kCluster + (int)rank, p0 = t * kTile;
  const int r0 = a.rm.start[b], M = a.rm.start[b + 1] - r0;
  const int G = a.nq / a.nkv, qn = M * G;
  const int L = a.len[b];
  const bool fits = rows_fit(L, M, a.cap);
  const int kend = L + M;
  const int n_tiles = fits ? (kend + kTile - 1) / kTile : 0;
  const int n_chunks = (n_tiles + kCluster - 1) / kCluster;
  const bool active = t < n_tiles;      // this CTA's tile holds keys
  const bool cl_active = c2 * HALVES < n_chunks;  // uniform over the cluster
  if (!cl_active) return;               // the whole cluster holds no keys of this request
  const int z = (a.layer * a.batch + b) * a.nkv + g;
  const uint8_t* qsrc = a.qimg + ((size_t)(b * a.nkv + g) * a.qt_max + qt) * (size_t)Q_BYTES;

  if (tid == 0) {
    for (int i = 0; i < 5; ++i) ptx::mbar_init(&bars[i], 1);
    ptx::fence_mbar_init();
  }
  if (warp == 0) ptx::tmem_alloc(tslot, TMEM_COLS);
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = *tslot;
  const uint32_t lane_base = (uint32_t)(32 * warp) << 16;

  // a tile of entries older than this call does not depend on the finishing
  // kernel: request it before the wait
  const bool early = active && p0 + kTile <= L;
  const uint64_t pol = ptx::policy_evict_first();
  auto load_kv = [&]() {
    ptx::mbar_arrive_expect_tx(&bars[1], NARROW ? K_BYTES : 2 * K_BYTES);
#pragma unroll
    for (int h = 0; h < NR; ++h) {
      ptx::tma_load_3d(R1 + h * kRegion, &tmK, &bars[1], 64 * h, p0, z, pol);
      // narrow: V is loaded once the first product has consumed the keys;
      // in launches of a few waves it is brought into L2 now
      if (!NARROW)
        ptx::tma_load_3d(R2 + h * kRegion, &tmV, &bars[1], 64 * h, p0, z, pol);
      else if (a.v_prefetch)
        ptx::tma_prefetch_3d(&tmV, 64 * h, p0, z);
    }
  };
  auto load_v = [&]() {  // narrow: into the K image, once the first product is done
    ptx::mbar_arrive_expect_tx(&bars[4], K_BYTES);
#pragma unroll
    for (int h = 0; h < NR; ++h) ptx::tma_load_3d(R2 + h * kRegion, &tmV, &bars[4], 64 * h, p0, z, pol);
  };
  if (tid == 0 && early) {
    ptx::prefetch_tmap(&tmK);
    ptx::prefetch_tmap(&tmV);
    load_kv();
  }
  ptx::griddep_wait();
  if (tid == 0 && active) {
    if (!early) load_kv();
    ptx::mbar_arrive_expect_tx(&bars[0], Q_BYTES);
    ptx::bulk_load(R0, qsrc, Q_BYTES, &bars[0], ptx::policy_evict_last());
  }

  // Thread tid reads TMEM lane tid: query q = tid / 2, its hi part (pt = 0)
  // or lo part (pt = 1).  After the exchange with its partner lane it keeps
  // keys [64 pt, 64 pt + 64) of S and dims [DH pt, DH pt + DH) of O.
  const int q = tid >> 1, pt = tid & 1;
  const int qg = qt * kQT + q;
  const int lim = qg < qn ? L + qg / G : -1;  // the query's last visible key
  float m = -INFINITY, l = 0.f;               // the tile partial of query q
  float o[DH];
#pragma unroll
  for (int j = 0; j < DH; ++j) o[j] = 0.f;
  bool ok = true;
  if (active) {
    ok = ptx::mbar_wait(&bars[0], 0, a.timeout_ns) && ptx::mbar_wait(&bars[1], 0, a.timeout_ns);
    ok = ptx::group_all(ok, 1, 128);
    if (!ok) {
      if (tid == 0) {
        atomicOr(a.err, kErrTimeout);
        // the copies may still be in flight: wait for them before the CTA ends
        ptx::mbar_wait(&bars[0], 0, ptx::kDrainNs);
        ptx::mbar_wait(&bars[1], 0, ptx::kDrainNs);
      }
      __syncthreads();
    }
  }
  // values past the call's last key (stale entries, or NaN in a poisoned
  // cache) would reach O through 0 * V: those rows of the V tile are zeroed
  auto zero_v_tail = [&]() {
    const int z0 = kend - p0;
    if (z0 < kTile) {
      for (int idx = tid; idx < (kTile - z0) * NR * 8; idx += 128) {
        const int r = z0 + idx / (NR * 8), rest = idx - (idx / (NR * 8)) * (NR * 8);
        *reinterpret_cast<uint4*>(R2 + (rest >> 3) * kRegion + r * 128 + (rest & 7) * 16) =
            make_uint4(0, 0, 0, 0);
      }
      ptx::fence_proxy_async_smem();
    }
  };
  // Every thread arrives once at the split cluster barrier, when its CTA no
  // longer reads the image the cluster's partials are received into (the K
  // image: wide after the first product, narrow after the second, V being
  // loaded there): the product's completion, observed on its mbarrier, means
  // its operand reads are done, so the arrival needs no release.  The others
  // wait for the arrival only when they push.
  if (active && ok) {
    if (tid == 0) {
      ptx::tc_fence_after();
      constexpr uint32_t IDESC1 = ptx::idesc_bf16_f32(128, kTile);
#pragma unroll
      for (int kk = 0; kk < D / 16; ++kk) {
        const uint64_t ad = ptx::sdesc_sw128(ptx::smem_u32(R0 + (kk >> 2) * kRegion)) + 2 * (kk & 3);
        const uint64_t bd = ptx::sdesc_sw128(ptx::smem_u32(R1 + (kk >> 2) * kRegion)) + 2 * (kk & 3);
        ptx::mma_bf16(tmem, ad, bd, IDESC1, kk > 0 ? 1u : 0u);
      }
      ptx::mma_commit(&bars[2]);
    }
    if (!NARROW) zero_v_tail();  // while the first product runs
    const bool ok1 = ptx::group_all(ptx::mbar_wait(&bars[2], 0, a.timeout_ns), 1, 128);
    // (after a timeout: once the product has drained)
    if (!ok1 && tid == 0) ptx::mbar_wait(&bars[2], 0, ptx::kDrainNs);
    if (!NARROW || !ok1) ptx::cluster_arrive_relaxed();
    // narrow: the keys are consumed; V comes into their image during the softmax
    if (NARROW && ok1 && tid == 0) load_v();
    ptx::tc_fence_after();
    bool ok2 = ok1, vok = ok1;
    if (ok1) {
      // S = hi + lo of this thread's keys, masked; the tile's maximum and
      // P = 2^(S - m) with the partner lane
      float sv[64];
      {
        float v0[64], v1[64];
        tmem_ld128(tmem + lane_base, v0, v1);
#pragma unroll
        for (int j = 0; j < 64; ++j) {
          const float mine = pt ? v1[j] : v0[j], other = pt ? v0[j] : v1[j];
          sv[j] = mine + __shfl_xor_sync(0xFFFFFFFFu, other, 1);
        }
      }
      softmax_tail(sv, pt, p0 + 64 * pt, lim, m, l);
      // P as bf16 hi (row 2q) and lo (row 2q + 1) parts: hi = P with its low
      // 16 bits cleared, lo = bf16(P - hi).  Wide: into TMEM over S (the
      // second product's A operand, lane 2q + pt its row, two keys per
      // column), each lane completing its row with the partner's half of the
      // keys.  Narrow: into the operand image in shared memory, K-major by key.
      if (!NARROW) {
        uint32_t hw[32], lw[32], row[64];
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          const uint32_t b0 = __float_as_uint(sv[2 * j]), b1 = __float_as_uint(sv[2 * j + 1]);
          hw[j] = (b0 >> 16) | (b1 & 0xFFFF0000u);
          const __nv_bfloat162 lv =
              __floats2bfloat162_rn(sv[2 * j] - __uint_as_float(b0 & 0xFFFF0000u),
                                    sv[2 * j + 1] - __uint_as_float(b1 & 0xFFFF0000u));
          lw[j] = *reinterpret_cast<const uint32_t*>(&lv);
        }
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          // the hi lane takes the partner's hi words (keys 64..127), the lo
          // lane the partner's lo words (keys 0..63)
          const uint32_t got = __shfl_xor_sync(0xFFFFFFFFu, pt ? hw[j] : lw[j], 1);
          row[j] = pt ? got : hw[j];
          row[32 + j] = pt ? lw[j] : got;
        }
        ptx::tmem_st_x64(tmem + lane_base, row);
        ptx::tmem_st_wait();
      } else {
#pragma unroll
        for (int ch = 0; ch < 8; ++ch) put_hilo8(R0, q, pt, 64 * pt + 8 * ch, sv + 8 * ch);
      }
      if (NARROW) {
        vok = ptx::group_all(ptx::mbar_wait(&bars[4], 0, a.timeout_ns), 1, 128);
        if (vok) zero_v_tail();
      }
      ptx::fence_proxy_async_smem();
      // (narrow: the second product writes O over S, read out above)
      ptx::tc_fence_before();
      __syncthreads();
      if (tid == 0 && vok) {
        ptx::tc_fence_after();
        constexpr uint32_t IDESC2 = ptx::idesc_bf16_f32(128, D, true);
#pragma unroll
        for (int kk = 0; kk < kTile / 16; ++kk) {
          const uint64_t bd = ptx::sdesc_sw128_mn(ptx::smem_u32(R2) + kk * 2048u, kRegion, 1024u);
          if (NARROW) {
            const uint64_t ad = ptx::sdesc_sw128(ptx::smem_u32(R0 + (kk >> 2) * kRegion)) + 2 * (kk & 3);
            ptx::mma_bf16(tmem, ad, bd, IDESC2, kk > 0 ? 1u : 0u);
          } else {
            // A: 16 keys = 8 columns per k-step
            ptx::mma_bf16_ta(tmem + 128, tmem + 8u * kk, bd, IDESC2, kk > 0 ? 1u : 0u);
          }
        }
        ptx::mma_commit(&bars[3]);
      }
      ok2 = vok && ptx::group_all(ptx::mbar_wait(&bars[3], 0, a.timeout_ns), 1, 128);
      if (NARROW) {
        // (after a timeout: once the copy and the product have drained)
        if (!ok2 && tid == 0) {
          ptx::mbar_wait(&bars[4], 0, ptx::kDrainNs);
          if (vok) ptx::mbar_wait(&bars[3], 0, ptx::kDrainNs);
        }
        ptx::cluster_arrive_relaxed();
      }
      ptx::tc_fence_after();
      if (ok2) {
        // O = hi + lo of this thread's dims
#pragma unroll
        for (int c0 = 0; c0 < D; c0 += 64) {
          float v[64];
          tmem_ld64(tmem + lane_base + (NARROW ? 0 : 128) + c0, v);
#pragma unroll
          for (int j = 0; j < 64; ++j) {
            const int d = c0 + j;  // compile-time after unrolling
            const bool mine = (d / DH) == pt;
            const float x = __shfl_xor_sync(0xFFFFFFFFu, v[j], 1);
            if (mine) o[d - pt * DH] = v[j] + x;
          }
        }
      }
    }
    if (!(ok1 && ok2)) {
      if (tid == 0) {
        atomicOr(a.err, kErrTimeout);
        // no MMA may still run when TMEM is freed
        ptx::mbar_wait(&bars[2], 0, ptx::kDrainNs);
        if (vok) ptx::mbar_wait(&bars[3], 0, ptx::kDrainNs);
      }
      m = -INFINITY;  // nothing of this tile is passed on
    }
  } else {
    ptx::cluster_arrive_relaxed();  // no keys of this CTA's tile are read
  }
  // the tile's products are done: the next kernel (the O projection) may
  // start and stream its first weight tiles now (earlier, they would compete
  // with this kernel's own loads)
  ptx::griddep_launch_dependents();
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 0) ptx::tmem_dealloc(tmem, TMEM_COLS);

  // ---- the cluster's tile partials, pushed to the CTA that folds them ----
  // CTA r folds query rows RPC r .. RPC r + RPC - 1 (RPC: 8 in a cluster of
  // 8, 4 in a cluster of 16); it receives, from the CTA of every tile i of
  // the cluster, rows (max, sum) into s_rml[i][row] and O into
  // recv[i][row][d], over its K image (every CTA's is consumed once all have
  // arrived)
  constexpr int RPC = PAIR ? 4 : 8;
  ptx::cluster_wait();
  if (active) {
    const uint32_t dst_rank = (uint32_t)(q / RPC), row = (uint32_t)(q % RPC);
    if (pt == 0)
      dsmem_st_f2(ptx::dsmem_map(ptx::smem_u32(s_rml + crank * RPC + row), dst_rank), make_float2(m, l));
    if (m != -INFINITY) {
      const uint32_t dst =
          ptx::dsmem_map(ptx::smem_u32(recv + (crank * RPC + row) * D + pt * DH), dst_rank);
#pragma unroll
      for (int u = 0; u < DH / 4; ++u)
        dsmem_st_f4(dst + 16u * u, make_float4(o[4 * u], o[4 * u + 1], o[4 * u + 2], o[4 * u + 3]));
    }
  }
  ptx::cluster_sync();

  if (PAIR) {
    // ---- two chunks in one cluster: CTA r folds rows 4r..4r+3, each
    // chunk's 8 tiles in tile order, then the two chunk partials in chunk
    // order: the arithmetic of the one-chunk fold and of the fold through
    // memory below (thread: row fj, dims [fd, fd + 4))
    constexpr int TPR = D / 4 < 32 ? D / 4 : 32;  // threads per row
    if (tid < 4 * TPR) {
      const int fj = tid / TPR, fr = 4 * (int)crank + fj, fd = 4 * (tid % TPR);
      float cmx[2], cls[2], cfo[2][4];
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int nh = min(kCluster, n_tiles - (c2 * 2 + h) * kCluster);  // may be <= 0
        float fm = -INFINITY;
        float2 pml[kCluster];
#pragma unroll
        for (int i = 0; i < kCluster; ++i) {
          pml[i] = (i < nh) ? s_rml[(h * kCluster + i) * 4 + fj] : make_float2(-INFINITY, 0.f);
          fm = fmaxf(fm, pml[i].x);
        }
        float fl = 0.f, fo[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int i = 0; i < kCluster; ++i) {
          const float w = part_weight(pml[i].x, fm);
          if (w != 0.f) {
            fl += pml[i].y * w;
            const float4 v = *reinterpret_cast<const float4*>(recv + ((h * kCluster + i) * 4 + fj) * D + fd);
            fo[0] += v.x * w;
            fo[1] += v.y * w;
            fo[2] += v.z * w;
            fo[3] += v.w * w;
          }
        }
        cmx[h] = fm;
        cls[h] = fl;
#pragma unroll
        for (int e = 0; e < 4; ++e) cfo[h][e] = fo[e];
      }
      if (n_chunks == 1) {
        write_rows<D, 4>(a, cfo[0], cls[0], fr, fd, qt, qn, G, g, r0);
      } else {
        float cm = -INFINITY;
#pragma unroll
        for (int cc = 0; cc < 2; ++cc) cm = fmaxf(cm, cmx[cc]);
        float cl_ = 0.f, co[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int cc = 0; cc < 2; ++cc) {
          const float w = part_weight(cmx[cc], cm);
          if (w != 0.f) {
            cl_ += cls[cc] * w;
#pragma unroll
            for (int e = 0; e < 4; ++e) co[e] += cfo[cc][e] * w;
          }
        }
        write_rows<D, 4>(a, co, cl_, fr, fd, qt, qn, G, g, r0);
      }
    }
    return;
  }

  fold_chunk8<D>(a, recv, s_rml, s_flag, sm, kStage, rank, c, n_tiles, n_chunks, b, g, qt, qn, G,
                 r0);
}

// Four CTAs per SM (QUAD), for launches of more clusters than the narrow
// layout keeps resident: the narrow layout's tiles, arithmetic and fold in
// 48 KB of shared memory, 128 TMEM columns and at most 128 registers a
// thread.  The first product runs in halves of d (the whole Q image, one
// 16 KB region of the K tile at a time); V is loaded over Q; P goes to TMEM
// over S, and the second product runs in 64-dim halves of O over S's second
// half, each read out before the next.  S is read and P written in 16-key
// chunks, so that no thread holds a whole row of either.
constexpr uint32_t attn4_smem() { return 32768 + 16384 + 64 * 8 + 8 * 8 + 4 + 16 + 1024; }
static_assert(4 * (attn4_smem() + 1024) <= 228 * 1024, "four CTAs per SM");
// chunks the last arriver stages in shared memory: [11][8 rows][128] floats
// and [11][8] (max, sum) within the Q and K images
constexpr int kStage4 = 11;
static_assert(kStage4 * 8 * 128 * 4 + kStage4 * 8 * 8 <= 32768 + 16384, "staging fits");

template <int D>
__global__ void __launch_bounds__(128, 4)
    attn_tc4_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                    const __grid_constant__ AttnArgs a) {
  constexpr int NR = D / 64;          // 64-column regions of a K / V tile
  constexpr uint32_t Q_BYTES = 2u * kQT * D * 2;
  constexpr int DH = D / 2;           // dims each thread of a hi/lo pair keeps
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* R0 = sm;            // Q image -> V tile -> the partials received from the cluster
  uint8_t* RK = sm + 32768;    // one 64-column region of the K tile
  float* recv = reinterpret_cast<float*>(R0);                // [8 tiles][8 rows][D]
  float2* s_rml = reinterpret_cast<float2*>(sm + 49152);    // [8][8] (max, sum)
  uint64_t* bars = reinterpret_cast<uint64_t*>(s_rml + 64);  // q, k0, s0, k1, s1, v, o0, o1
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bars + 8);
  int* s_flag = reinterpret_cast<int*>(tslot + 1);

  const int tid = threadIdx.x, warp = tid >> 5;
  const uint32_t rank = ptx::cluster_rank();
  const int cl = (int)(blockIdx.x / kCluster), g = blockIdx.y;
  int b = 0;
  while (b + 1 < a.rm.batch && a.cl_start[b + 1] <= cl) ++b;
  const int ci = cl - a.cl_start[b];
  const int ncl = a.n_ch[b];  // clusters per query tile
  const int qt = ci / ncl, c = ci - qt * ncl;
  const int t = c * kCluster + (int)rank, p0 = t * kTile;
  const int r0 = a.rm.start[b], M = a.rm.start[b + 1] - r0;
  const int G = a.nq / a.nkv, qn = M * G;
  const int L = a.len[b];
  const bool fits = rows_fit(L, M, a.cap);
  const int kend = L + M;
  const int n_tiles = fits ? (kend + kTile - 1) / kTile : 0;
  const int n_chunks = (n_tiles + kCluster - 1) / kCluster;
  const bool active = t < n_tiles;
  if (c >= n_chunks) return;  // the whole cluster holds no keys of this request
  const int z = (a.layer * a.batch + b) * a.nkv + g;
  const uint8_t* qsrc = a.qimg + ((size_t)(b * a.nkv + g) * a.qt_max + qt) * (size_t)Q_BYTES;

  if (tid == 0) {
    for (int i = 0; i < 8; ++i) ptx::mbar_init(&bars[i], 1);
    ptx::fence_mbar_init();
  }
  if (warp == 0) ptx::tmem_alloc(tslot, 128);
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = *tslot;
  const uint32_t lane_base = (uint32_t)(32 * warp) << 16;

  const uint64_t pol = ptx::policy_evict_first();
  uint32_t issued = 0;  // (thread 0) barriers with a copy or product outstanding
  auto load_k = [&](int h, int bar) {  // region h of the K tile into RK
    ptx::mbar_arrive_expect_tx(&bars[bar], kRegion);
    ptx::tma_load_3d(RK, &tmK, &bars[bar], 64 * h, p0, z, pol);
    issued |= 1u << bar;
  };
  auto prefetch_rest = [&]() {  // the other K regions (and V, in launches of a few waves) into L2
#pragma unroll
    for (int h = 1; h < NR; ++h) ptx::tma_prefetch_3d(&tmK, 64 * h, p0, z);
    if (a.v_prefetch)
      for (int h = 0; h < NR; ++h) ptx::tma_prefetch_3d(&tmV, 64 * h, p0, z);
  };
  // a tile of entries older than this call does not depend on the finishing
  // kernel: request it before the wait
  const bool early = active && p0 + kTile <= L;
  if (tid == 0 && early) {
    ptx::prefetch_tmap(&tmK);
    ptx::prefetch_tmap(&tmV);
    load_k(0, 1);
    prefetch_rest();
  }
  ptx::griddep_wait();
  if (tid == 0 && active) {
    if (!early) {
      load_k(0, 1);
      prefetch_rest();
    }
    ptx::mbar_arrive_expect_tx(&bars[0], Q_BYTES);
    ptx::bulk_load(R0, qsrc, Q_BYTES, &bars[0], ptx::policy_evict_last());
    issued |= 1u;
  }

  // Thread tid reads TMEM lane tid: query q = tid / 2, its hi part (pt = 0)
  // or lo part (pt = 1); it keeps keys [64 pt, 64 pt + 64) of S and dims
  // [DH pt, DH pt + DH) of O.
  const int q = tid >> 1, pt = tid & 1;
  const int qg = qt * kQT + q;
  const int lim = qg < qn ? L + qg / G : -1;
  float m = -INFINITY, l = 0.f;
  float o[DH];  // written by the second product's read-out; pushed only then
  auto wait_all = [&](bool ok, int bar) {
    return ptx::group_all(ok && ptx::mbar_wait(&bars[bar], 0, a.timeout_ns), 1, 128);
  };
  bool ok = true;
  if (active) {
    ok = wait_all(wait_all(true, 0), 1);
    // S = Q K^T in halves of d: region h of Q and of K, one accumulation chain
#pragma unroll
    for (int h = 0; h < NR; ++h) {
      if (h > 0) {
        if (ok && tid == 0) load_k(h, 3);  // over the region the first half consumed
        ok = wait_all(ok, 3);
      }
      if (ok && tid == 0) {
        ptx::tc_fence_after();
        constexpr uint32_t IDESC1 = ptx::idesc_bf16_f32(128, kTile);
#pragma unroll
        for (int k4 = 0; k4 < 4; ++k4) {
          const int kk = 4 * h + k4;
          const uint64_t ad = ptx::sdesc_sw128(ptx::smem_u32(R0 + h * kRegion)) + 2 * k4;
          const uint64_t bd = ptx::sdesc_sw128(ptx::smem_u32(RK)) + 2 * k4;
          ptx::mma_bf16(tmem, ad, bd, IDESC1, kk > 0 ? 1u : 0u);
        }
        ptx::mma_commit(&bars[2 + 2 * h]);
        issued |= 1u << (2 + 2 * h);
      }
      ok = wait_all(ok, 2 + 2 * h);
    }
    // Q and K are consumed: V comes over Q (from L2) during the softmax
    if (ok && tid == 0) {
      ptx::mbar_arrive_expect_tx(&bars[5], NR * kRegion);
#pragma unroll
      for (int h = 0; h < NR; ++h) ptx::tma_load_3d(R0 + h * kRegion, &tmV, &bars[5], 64 * h, p0, z, pol);
      issued |= 1u << 5;
    }
    ptx::tc_fence_after();
    if (ok) {
      // S = hi + lo of this thread's keys, 16 keys of each half at a time
      float sv[64];
#pragma unroll
      for (int cc = 0; cc < 4; ++cc) {
        uint32_t k0[16], k1[16];  // keys 16 cc + j and 64 + 16 cc + j
        ptx::tmem_ld16(tmem + lane_base + 16 * cc, k0);
        ptx::tmem_ld16(tmem + lane_base + 64 + 16 * cc, k1);
        ptx::tmem_ld_wait();
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const float v0 = __uint_as_float(k0[j]), v1 = __uint_as_float(k1[j]);
          const float mine = pt ? v1 : v0, other = pt ? v0 : v1;
          sv[16 * cc + j] = mine + __shfl_xor_sync(0xFFFFFFFFu, other, 1);
        }
      }
      softmax_tail(sv, pt, p0 + 64 * pt, lim, m, l);
      // P as bf16 hi (row 2q) and lo (row 2q + 1) parts into TMEM over S, two
      // keys per column, 16 keys (8 columns of each half of the row) at a
      // time; each lane completes its row with the partner's half of the keys
#pragma unroll
      for (int cc = 0; cc < 4; ++cc) {
        uint32_t hw[8], lw[8], first[8], second[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const float x0 = sv[16 * cc + 2 * j], x1 = sv[16 * cc + 2 * j + 1];
          const uint32_t b0 = __float_as_uint(x0), b1 = __float_as_uint(x1);
          hw[j] = (b0 >> 16) | (b1 & 0xFFFF0000u);
          const __nv_bfloat162 lv = __floats2bfloat162_rn(x0 - __uint_as_float(b0 & 0xFFFF0000u),
                                                          x1 - __uint_as_float(b1 & 0xFFFF0000u));
          lw[j] = *reinterpret_cast<const uint32_t*>(&lv);
        }
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          // the hi lane takes the partner's hi words (keys 64..127), the lo
          // lane the partner's lo words (keys 0..63)
          const uint32_t got = __shfl_xor_sync(0xFFFFFFFFu, pt ? hw[j] : lw[j], 1);
          first[j] = pt ? got : hw[j];
          second[j] = pt ? lw[j] : got;
        }
        ptx::tmem_st_x8(tmem + lane_base + 8 * cc, first);
        ptx::tmem_st_x8(tmem + lane_base + 32 + 8 * cc, second);
      }
      ptx::tmem_st_wait();
    }
    ok = wait_all(ok, 5);
    // values past the call's last key would reach O through 0 * V
    if (ok) {
      const int z0 = kend - p0;
      if (z0 < kTile) {
        for (int idx = tid; idx < (kTile - z0) * NR * 8; idx += 128) {
          const int r = z0 + idx / (NR * 8), rest = idx - (idx / (NR * 8)) * (NR * 8);
          *reinterpret_cast<uint4*>(R0 + (rest >> 3) * kRegion + r * 128 + (rest & 7) * 16) =
              make_uint4(0, 0, 0, 0);
        }
      }
    }
    ptx::fence_proxy_async_smem();
    // O = P V in 64-dim halves into TMEM columns 64..127 (S's second half,
    // read out above), each read out before the next is written
#pragma unroll
    for (int h = 0; h < NR; ++h) {
      ptx::tc_fence_before();
      __syncthreads();
      if (ok && tid == 0) {
        ptx::tc_fence_after();
        constexpr uint32_t IDESC2 = ptx::idesc_bf16_f32(128, 64, true);
#pragma unroll
        for (int kk = 0; kk < kTile / 16; ++kk) {
          const uint64_t bd =
              ptx::sdesc_sw128_mn(ptx::smem_u32(R0 + h * kRegion) + kk * 2048u, kRegion, 1024u);
          ptx::mma_bf16_ta(tmem + 64, tmem + 8u * kk, bd, IDESC2, kk > 0 ? 1u : 0u);
        }
        ptx::mma_commit(&bars[6 + h]);
        issued |= 1u << (6 + h);
      }
      ok = wait_all(ok, 6 + h);
      ptx::tc_fence_after();
      if (ok) {
#pragma unroll
        for (int cc = 0; cc < 4; ++cc) {
          uint32_t v16[16];
          ptx::tmem_ld16(tmem + lane_base + 64 + 16 * cc, v16);
          ptx::tmem_ld_wait();
          const int d0 = 64 * h + 16 * cc, owner = d0 / DH;  // compile-time after unrolling
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            const float v = __uint_as_float(v16[j]);
            const float x = __shfl_xor_sync(0xFFFFFFFFu, v, 1);
            if (pt == owner) o[d0 - owner * DH + j] = v + x;
          }
        }
      }
    }
    if (!ok) {
      if (tid == 0) {
        atomicOr(a.err, kErrTimeout);
        // no copy or product may still run when TMEM is freed and the CTA ends
        for (int i = 0; i < 8; ++i)
          if (issued & (1u << i)) ptx::mbar_wait(&bars[i], 0, ptx::kDrainNs);
      }
      m = -INFINITY;  // nothing of this tile is passed on
    }
  }
  // the V image is consumed: the cluster's partials may come into it
  ptx::cluster_arrive_relaxed();
  ptx::griddep_launch_dependents();
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 0) ptx::tmem_dealloc(tmem, 128);

  // ---- the tile partials, pushed to the CTA that folds their rows ----------
  ptx::cluster_wait();
  if (active) {
    const uint32_t dst_rank = (uint32_t)(q >> 3), row = (uint32_t)(q & 7);
    if (pt == 0)
      dsmem_st_f2(ptx::dsmem_map(ptx::smem_u32(s_rml + rank * 8 + row), dst_rank), make_float2(m, l));
    if (m != -INFINITY) {
      const uint32_t dst =
          ptx::dsmem_map(ptx::smem_u32(recv + (rank * 8 + row) * D + pt * DH), dst_rank);
#pragma unroll
      for (int u = 0; u < DH / 4; ++u)
        dsmem_st_f4(dst + 16u * u, make_float4(o[4 * u], o[4 * u + 1], o[4 * u + 2], o[4 * u + 3]));
    }
  }
  ptx::cluster_sync();
  fold_chunk8<D>(a, recv, s_rml, s_flag, sm, kStage4, rank, c, n_tiles, n_chunks, b, g, qt, qn, G,
                 r0);
}

// Clusters of 16 resident at once, two CTAs per SM: 14 in a residency probe
// (the occupancy calculator reports 7).
constexpr int kPairClusters = 14;

// How many clusters of 16 of the pair kernel the occupancy calculator allows
// (0 if none fits, or the launch attributes are refused); queried once per
// head size.
template <int D>
int pair_clusters_max() {
  static const int n = [] {
    constexpr uint32_t smem = attn_smem<false, true>();
    if (cudaFuncSetAttribute(attn_tc_kernel<D, false, true>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess ||
        cudaFuncSetAttribute(attn_tc_kernel<D, false, true>,
                             cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess)
      return 0;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(16 * 16, 1);
    cfg.blockDim = dim3(128);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = 16;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    int nc = 0;
    if (cudaOccupancyMaxActiveClusters(&nc, attn_tc_kernel<D, false, true>, &cfg) != cudaSuccess) {
      (void)cudaGetLastError();
      return 0;
    }
    return nc;
  }();
  return n;
}

template <int D, bool NARROW, bool PAIR>
cudaError_t launch_attn(const CUtensorMap& tk, const CUtensorMap& tv, const AttnArgs& a,
                        int clusters, cudaStream_t st) {
  constexpr uint32_t smem = attn_smem<NARROW, PAIR>();
  constexpr int CL = PAIR ? 2 * kCluster : kCluster;
  static const cudaError_t attr = cudaFuncSetAttribute(
      attn_tc_kernel<D, NARROW, PAIR>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (attr != cudaSuccess) return attr;
  // clusters of 16 are beyond the portable size of 8
  static const cudaError_t attr16 =
      PAIR ? cudaFuncSetAttribute(attn_tc_kernel<D, NARROW, PAIR>,
                                  cudaFuncAttributeNonPortableClusterSizeAllowed, 1)
           : cudaSuccess;
  if (attr16 != cudaSuccess) return attr16;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(clusters * CL, a.nkv);
  cfg.blockDim = dim3(128);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr2[2];
  attr2[0].id = cudaLaunchAttributeClusterDimension;
  attr2[0].val.clusterDim.x = CL;
  attr2[0].val.clusterDim.y = 1;
  attr2[0].val.clusterDim.z = 1;
  attr2[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr2[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr2;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, attn_tc_kernel<D, NARROW, PAIR>, tk, tv, a);
}

template <int D>
cudaError_t launch_attn4(const CUtensorMap& tk, const CUtensorMap& tv, const AttnArgs& a,
                         int clusters, cudaStream_t st) {
  constexpr uint32_t smem = attn4_smem();
  static const cudaError_t attr = cudaFuncSetAttribute(
      attn_tc4_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (attr != cudaSuccess) return attr;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(clusters * kCluster, a.nkv);
  cfg.blockDim = dim3(128);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr2[2];
  attr2[0].id = cudaLaunchAttributeClusterDimension;
  attr2[0].val.clusterDim.x = kCluster;
  attr2[0].val.clusterDim.y = 1;
  attr2[0].val.clusterDim.z = 1;
  attr2[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr2[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr2;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, attn_tc4_kernel<D>, tk, tv, a);
}

}  // namespace

int attn_q_tiles(int rows_per_request, int group) {
  return (rows_per_request * group + kQT - 1) / kQT;
}
int attn_chunks(int capacity) { return (capacity + kChunk - 1) / kChunk; }
size_t attn_qimg_bytes(int head_dim) { return (size_t)256 * head_dim; }

cudaError_t launch_attention_split(const RowMap& m, const Model& md, KvState& kv, int layer,
                                   cudaStream_t st) {
  const as2d_config& c = md.cfg;
  AttnArgs a;
  a.rm = m;
  a.len = kv.d_len;
  a.layer = layer;
  a.batch = kv.batch;
  a.cap = kv.capacity;
  a.nq = c.n_q_heads;
  a.nkv = c.n_kv_heads;
  a.qscale = 1.4426950408889634f / sqrtf((float)c.head_dim);
  a.qkv_part = kv.qkv_part;
  a.qkv_rinv = kv.qkv_rinv;
  a.rope = kv.rope;
  a.qkv_split = kv.qkv_split;
  a.qkv_ld = kv.rows_alloc;
  a.kc = kv.k_cache;
  a.vc = kv.v_cache;
  a.qimg = kv.qimg;
  a.qt_max = kv.attn_qt;
  a.ws_o = kv.attn_o;
  a.ws_ml = kv.attn_ml;
  a.chunks_max = kv.attn_chunks;
  a.cnt = kv.attn_cnt;
  a.ao = kv.ao;
  a.lo_row = kv.rows_alloc;
  a.err = kv.d_err;
  a.timeout_ns = kv.wait_ns;
  const int G = c.n_q_heads / c.n_kv_heads;
  int clusters8 = 0, max_nch = 0;
  for (int b = 0; b < kv.batch; ++b) {
    const int rows = m.start[b + 1] - m.start[b];
    const int64_t keys = kv.len_upper[b] + rows;
    int nch = (int)((keys + kChunk - 1) / kChunk);
    if (nch > kv.attn_chunks) nch = kv.attn_chunks;
    a.n_ch[b] = nch;
    if (nch > max_nch) max_nch = nch;
    clusters8 += attn_q_tiles(rows, G) * nch;
  }
  // The same arithmetic whichever way the launch runs; the layout decides
  // how many CTAs an SM holds and whether two chunks fold in one cluster.
  // Narrow: more than kWideClusters clusters of 8.  Pair: every request has
  // at most two chunks, and the clusters of 16 run at once.
  const bool narrow = clusters8 * c.n_kv_heads > kWideClusters;
  const bool quad = clusters8 * c.n_kv_heads > kNarrowClusters;
  // Measured: the prefetch of V takes 32 µs off a 7B block at L = 15128 (60
  // clusters of 8) and 12 µs at k = 16 (120), but adds 100 µs to a ragged
  // round of 16 requests (about 440 clusters, some nine waves).
  a.v_prefetch = clusters8 * c.n_kv_heads <= 128;
  int clusters16 = 0;
  for (int b = 0; b < kv.batch; ++b)
    clusters16 += attn_q_tiles(m.start[b + 1] - m.start[b], G) * ((a.n_ch[b] + 1) / 2);
  const bool pair_fits =
      (c.head_dim == 128 ? pair_clusters_max<128>() : pair_clusters_max<64>()) > 0;
  const bool pair = !narrow && pair_fits && max_nch == 2 && clusters16 * c.n_kv_heads <= kPairClusters;
  const int halves = pair ? 2 : 1;
  a.cl_start[0] = 0;
  for (int b = 0; b < kv.batch; ++b)
    a.cl_start[b + 1] = a.cl_start[b] + attn_q_tiles(m.start[b + 1] - m.start[b], G) *
                                            ((a.n_ch[b] + halves - 1) / halves);
  const int clusters = a.cl_start[kv.batch];
  const dim3 gf(m.rows, c.n_q_heads + 2 * c.n_kv_heads);
  cudaError_t e;
  kv.launches += 2;
  if (c.head_dim == 128) {
    e = launch_pdl(qkv_finish_kernel<128>, gf, dim3(64), 0, st, a);
    if (e == cudaSuccess)
      e = quad     ? launch_attn4<128>(kv.tm_kc, kv.tm_vc, a, clusters, st)
          : narrow ? launch_attn<128, true, false>(kv.tm_kc, kv.tm_vc, a, clusters, st)
          : pair ? launch_attn<128, false, true>(kv.tm_kc, kv.tm_vc, a, clusters, st)
                 : launch_attn<128, false, false>(kv.tm_kc, kv.tm_vc, a, clusters, st);
  } else {
    e = launch_pdl(qkv_finish_kernel<64>, gf, dim3(32), 0, st, a);
    if (e == cudaSuccess)
      e = quad     ? launch_attn4<64>(kv.tm_kc, kv.tm_vc, a, clusters, st)
          : narrow ? launch_attn<64, true, false>(kv.tm_kc, kv.tm_vc, a, clusters, st)
          : pair ? launch_attn<64, false, true>(kv.tm_kc, kv.tm_vc, a, clusters, st)
                 : launch_attn<64, false, false>(kv.tm_kc, kv.tm_vc, a, clusters, st);
  }
  return e;
}

}  // namespace as2d
