// gemm_tc.cuh -- skinny GEMM on the 5th-generation tensor cores for the
// verification pass: D[n][m] = sum_k W[n][k] X[m][k] for the k + 1 token rows
// m of a block (a handful) and every output feature n of a weight matrix W.
//
// Design (weights streamed once per block from HBM):
//   * swap-AB: the 128-row weight tile is the MMA's M operand (tcgen05.mma
//     kind::f16, M = 128), the token rows, padded to NB in {16..256}, are its
//     N operand, so no tensor-core work is spent on padding weight rows;
//   * activations are kept as two bf16 parts, hi = bf16(x) and lo =
//     bf16(x - hi), stored as two row blocks of the operand buffer; each
//     k-step issues one MMA per part into the same fp32 accumulator, so the
//     bf16 weights multiply x to about 16 significant bits (single bf16
//     operands cost ~5e-2 in the logits of a 28-layer model) at no extra
//     weight traffic;
//   * weights are stored tile-major at load time (k_pack.cu): every 128 x 64
//     weight tile is one contiguous, pre-swizzled 16 KB block, fetched with a
//     single bulk copy (cp.async.bulk), so each SM streams one contiguous
//     region; the NB x 64 activation tiles come by TMA (cp.async.bulk.tensor,
//     128-byte swizzle).  An S-deep shared-memory ring guarded by mbarriers;
//     one thread issues loads, one thread issues MMAs, four warps drain the
//     fp32 accumulator from TMEM (double-buffered);
//   * stream-K: the (tile, 64-column k-block) units are split evenly over a
//     persistent grid of one CTA per SM, so every SM streams the same number
//     of weight bytes whatever N is.  A CTA that holds a whole tile applies
//     the epilogue itself; each CTA that holds part of a tile cut between
//     CTAs stores its partial tile, and the last of them to arrive (an atomic
//     count per tile) adds the parts in CTA order and applies the epilogue:
//     the sum order depends on (N, K, grid) only, never on the number of
//     token rows or on arrival order, so results are batch invariant;
//   * the epilogue is fused: residual add (O, down), SwiGLU (gate/up), and
//     logits + argmax (LM head).  The QKV projection (TC_PART) instead splits
//     K evenly over a fixed number of CTAs per tile and stores each CTA's
//     unscaled sums: the attention's first kernel adds them, applies RoPE and
//     appends the keys and values, so no CTA of this kernel waits for
//     another's part at its end.
// Every mbarrier wait is bounded in time; on expiry the kernel records an
// error bit, drains its own outstanding copies and MMAs, frees TMEM and exits.
#pragma once

#include "as2d_internal.h"
#include "ptx_sm100.cuh"

#ifndef AS2D_RING16
#define AS2D_RING16 6
#endif

namespace as2d {

// Weight-ring depth for a token-row padding: as many 16 KB weight tiles in
// flight as the stage size (weights + the hi and lo activation tiles) allows.
constexpr int tc_ring_depth(int nb) {
  return nb <= 32 ? AS2D_RING16 : nb <= 64 ? 5 : nb <= 96 ? 4 : nb <= 192 ? 3 : 2;
}

template <int NB>
struct TcShape {
  static constexpr int S = tc_ring_depth(NB);  // weight-ring depth
  static constexpr uint32_t A_BYTES = 128 * 64 * 2;
  static constexpr uint32_t B_BYTES = NB * 64 * 2;   // one of the hi / lo operand tiles
  static constexpr uint32_t STAGE_B = 2 * B_BYTES;   // hi tile, then lo tile
  static constexpr int CH = 16;       // epilogue column chunk
  static constexpr int SP = CH + 1;   // padded shared-memory row
  // hi and lo results accumulate in separate TMEM columns, [0, NB) and
  // [NB, 2 NB), and are added in the epilogue (hi + lo) -- the same
  // arithmetic for every NB, so results stay batch invariant.  NB <= 128: one
  // MMA of N = 2 NB covers the hi and lo rows (adjacent in shared memory) and
  // reads the weight tile once; wider paddings: two MMAs of N = NB.
  // Accumulators are double-buffered while 2 x 2 NB columns fit in TMEM's 512.
  static constexpr bool ONE_MMA = NB <= 128;
  static constexpr int ACC_COLS = 2 * NB;
  static constexpr int NBUF = 2 * ACC_COLS <= 512 ? 2 : 1;
  static constexpr uint32_t TMEM_COLS = NBUF * ACC_COLS <= 32    ? 32
                                        : NBUF * ACC_COLS <= 64  ? 64
                                        : NBUF * ACC_COLS <= 128 ? 128
                                        : NBUF * ACC_COLS <= 256 ? 256
                                                                 : 512;
  static constexpr uint32_t SMEM =
      1024 + S * (A_BYTES + STAGE_B) + 128 * SP * 4 + (3 * NB + 64) * 4 + (2 * S + 5) * 8 + 16;
  static_assert(SMEM <= 232448, "shared memory of one CTA");
  static_assert(NB % 16 == 0 && NB >= 16 && NB <= 256, "MMA N of M = 128");
};

__device__ __forceinline__ float tc_silu(float x) { return x / (1.0f + expf(-x)); }

__device__ __forceinline__ unsigned long long tc_pack_best(float v, int idx) {
  uint32_t u = __float_as_uint(v);
  uint32_t key = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  return ((unsigned long long)key << 32) | (unsigned long long)(0xFFFFFFFFu - (uint32_t)idx);
}

// TC_PART: CTA c takes k-blocks [r kb / split, (r + 1) kb / split) of tile
// c / split (r = c mod split); otherwise the stream-K range of tc_start.
// Either way the decomposition depends on (N, K, the device) only, never on
// the number of token rows.
__device__ __forceinline__ long long tc_start(int c, const TcParams& p);
__device__ __forceinline__ void tc_range(int c, const TcParams& p, long long& u0, long long& u1) {
  if (p.split > 1) {
    const int tile = c / p.split, r = c - tile * p.split;
    u0 = (long long)tile * p.kb + (long long)r * p.kb / p.split;
    u1 = (long long)tile * p.kb + (long long)(r + 1) * p.kb / p.split;
  } else if (p.split == 1) {
    // whole tiles [c T / grid, (c + 1) T / grid)
    u0 = ((long long)c * p.n_tiles / p.grid) * p.kb;
    u1 = ((long long)(c + 1) * p.n_tiles / p.grid) * p.kb;
  } else {
    u0 = tc_start(c, p);
    u1 = tc_start(c + 1, p);
  }
}

__device__ __forceinline__ long long tc_start(int c, const TcParams& p) {
  return (long long)c * p.units / p.grid;
}
__device__ __forceinline__ int tc_owner(long long u, const TcParams& p) {
  return (int)(((u + 1) * (long long)p.grid - 1) / p.units);
}

// Operands of one 16-row epilogue chunk that come from memory (the residual
// and the norm gain for RESID), fetched by tc_epilogue_load before they are
// needed so that their loads overlap other loads of the caller.
struct TcEpiIn {
  float hv[16];
  float gn;
};

template <int NB, int EPI>
__device__ __forceinline__ void tc_epilogue_load(const TcParams& p, TcEpiIn& in, int tile, int m0,
                                                 int et) {
  constexpr int CH = TcShape<NB>::CH;
  const int n = et, col = tile * 128 + n;
  if (EPI == TC_RESID) {
    in.gn = p.g_next[col];
#pragma unroll
    for (int j = 0; j < CH; ++j)
      if (m0 + j < p.rows) in.hv[j] = p.h[(size_t)(p.row0 + m0 + j) * p.N + col];
  }
}

// Fused epilogue of one 16-row chunk: sC[n * SP + j] holds D for tile row n
// and token row row0 + m0 + j; `in` holds the chunk's tc_epilogue_load.  Runs
// on the 128 epilogue threads (et).
template <int NB, int EPI>
__device__ __forceinline__ void tc_epilogue_apply(const TcParams& p, const TcEpiIn& in,
                                                  const float* sC, float* red, const int* s_pos,
                                                  const int* s_req, int tile, int m0, int et) {
  constexpr int SP = TcShape<NB>::SP;
  constexpr int CH = TcShape<NB>::CH;
  if (EPI == TC_RESID) {
    // thread et owns tile row n = et for the chunk's 16 token rows.  The new
    // residual also yields the next projection's operand and its share of
    // the row's sum of squares (warp butterflies, then warps in order).
    const int n = et, col = tile * 128 + n;
    const float gn = in.gn;
    float hv[CH];
#pragma unroll
    for (int j = 0; j < CH; ++j) hv[j] = in.hv[j];
#pragma unroll
    for (int j = 0; j < CH; ++j) {
      if (m0 + j < p.rows) {
        const size_t at = (size_t)(p.row0 + m0 + j) * p.N + col;
        const float hn = hv[j] + sC[n * SP + j];
        p.h[at] = hn;
        const float xv = hn * gn;
        const bf16 xh = __float2bfloat16_rn(xv);
        p.xn[at] = xh;
        p.xn[at + (size_t)p.lo_row * p.N] = __float2bfloat16_rn(xv - __bfloat162float(xh));
        hv[j] = hn * hn;
      } else {
        hv[j] = 0.f;
      }
    }
#pragma unroll
    for (int j = 0; j < CH; ++j) {
      float v = hv[j];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
      if ((et & 31) == 0) red[(et >> 5) * CH + j] = v;
    }
    ptx::named_bar_sync(1, 128);
    if (et < CH && m0 + et < p.rows)
      p.ss[(size_t)tile * p.ss_ld + p.row0 + m0 + et] =
          ((red[et] + red[CH + et]) + red[2 * CH + et]) + red[3 * CH + et];
  } else if (EPI == TC_SWIGLU) {
    const int F = p.N >> 1;
    for (int idx = et; idx < 64 * CH; idx += 128) {
      const int j = idx >> 6, i = idx & 63, m = m0 + j;
      if (m >= p.rows) break;
      const float g = sC[i * SP + j], up = sC[(64 + i) * SP + j];
      const float uv = tc_silu(g) * up;
      const bf16 uh = __float2bfloat16_rn(uv);
      const size_t at = (size_t)(p.row0 + m) * F + (size_t)tile * 64 + i;
      p.u[at] = uh;
      p.u[at + (size_t)p.lo_row * F] = __float2bfloat16_rn(uv - __bfloat162float(uh));
    }
  } else {  // TC_LOGITS
    if (p.logits) {
      for (int idx = et; idx < 128 * CH; idx += 128) {
        const int j = idx >> 7, n = idx & 127, m = m0 + j;
        if (m >= p.rows) break;
        const int col = tile * 128 + n;
        if (col < p.N) p.logits[(size_t)(p.row0 + m) * p.N + col] = sC[n * SP + j];
      }
    }
    const int ew = et >> 5, el = et & 31;
    for (int j = ew; j < CH; j += 4) {
      const int m = m0 + j;
      if (m >= p.rows) break;
      unsigned long long best = 0ull;
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        const int n = el + 32 * t, col = tile * 128 + n;
        if (col < p.N) {
          const unsigned long long key = tc_pack_best(sC[n * SP + j], col);
          best = key > best ? key : best;
        }
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const unsigned long long other = __shfl_xor_sync(0xFFFFFFFFu, best, o);
        best = other > best ? other : best;
      }
      if (el == 0) atomicMax(&p.best[p.row0 + m], best);
    }
  }
}

template <int NB, int EPI>
__device__ __forceinline__ void tc_epilogue_chunk(const TcParams& p, const float* sC, float* red,
                                                  const int* s_pos, const int* s_req, int tile,
                                                  int m0, int et) {
  TcEpiIn in;
  tc_epilogue_load<NB, EPI>(p, in, tile, m0, et);
  tc_epilogue_apply<NB, EPI>(p, in, sC, red, s_pos, s_req, tile, m0, et);
}

// 16 accumulator columns of chunk ch for this thread's TMEM lane: the hi and
// lo results are added here (hi + lo, fixed order).
template <int NB>
__device__ __forceinline__ void tc_load_acc(uint32_t tbase, int ch, uint32_t (&v)[16]) {
  uint32_t w[16];
  ptx::tmem_ld16(tbase + ch * 16, v);
  ptx::tmem_ld16(tbase + NB + ch * 16, w);
  ptx::tmem_ld_wait();
#pragma unroll
  for (int j = 0; j < 16; ++j) v[j] = __float_as_uint(__uint_as_float(v[j]) + __uint_as_float(w[j]));
}

// Per-row values the epilogue needs, for the launch's token rows: 1 / rms of
// each row from the producer's per-tile sums of squares (in tile order), and
// for QKV the request and cache position of each row.  Run by the 128
// epilogue threads (et), ends with their named barrier.
template <int NB, int EPI>
__device__ __forceinline__ void tc_row_prologue(const TcParams& p, float* s_rinv, int* s_pos,
                                                int* s_req, int et) {
    // every load below is issued before any result is used: one memory
    // round trip for up to 32 tiles' sums (hidden <= 4096)
    for (int m = et; m < p.rows; m += 128) {
      const int gm = p.row0 + m;
      if (EPI != TC_RESID) {
        // 1 / rms of the token row from the producer's per-tile sums (in order)
        const float* src = p.ss + gm;
        float tot = 0.f;
        for (int t0 = 0; t0 < p.n_htiles; t0 += 32) {
          float v[32];
#pragma unroll
          for (int u = 0; u < 32; ++u)
            v[u] = (t0 + u < p.n_htiles) ? src[(size_t)(t0 + u) * p.ss_ld] : 0.f;
#pragma unroll
          for (int u = 0; u < 32; ++u) tot += v[u];
        }
        s_rinv[m] = rsqrtf(tot / (float)p.hidden + p.eps);
        // TC_PART leaves the scaling to the kernel that finishes its sums
        if (EPI == TC_PART && blockIdx.x == 0) p.part_rinv[gm] = s_rinv[m];
      }
    }
    if (EPI != TC_RESID) ptx::named_bar_sync(1, 128);
}

// Adds the partial tiles of a split tile (parts c_first .. c_first + nparts - 1
// in CTA order, all parts' loads issued at once), scales like the GEMM's own
// epilogue and applies the fused epilogue.  128 threads (nl = tile row, et),
// named barrier 1; sC, s_rinv, red, s_pos, s_req as in the GEMM epilogue;
// PROLOGUE: also fills s_rinv, s_pos, s_req (tc_row_prologue), its loads
// overlapping the parts' loads.
template <int NB, int EPI, int MAXP = 8, bool PROLOGUE = false>
__device__ __forceinline__ void tc_reduce_tile(const TcParams& p, float* sC, float* s_rinv,
                                               float* red, int* s_pos, int* s_req,
                                               int tile, int c_first, int nparts, int nl, int et) {
  // MAXP parts are in flight at a time; the parts are added in CTA order
  // whatever MAXP is, so it does not change the result.  The first parts, the
  // epilogue's operands and (PROLOGUE) the row prologue's loads are all
  // issued before any of them is used.
  using Sh = TcShape<NB>;
  constexpr int CH = Sh::CH, SP = Sh::SP;
  const int nchunks = (p.rows + CH - 1) / CH;
  // slot 1 holds a CTA's last segment when it began in an earlier tile: only
  // the first part can be one
  const int sl0 = (int)(tc_start(c_first, p) / p.kb) != tile ? 1 : 0;
  for (int ch = 0; ch < nchunks; ++ch) {
    const int live = p.rows - ch * CH;
    float acc[CH];
#pragma unroll
    for (int j = 0; j < CH; ++j) acc[j] = 0.f;
    TcEpiIn in;
    for (int part0 = 0; part0 < nparts; part0 += MAXP) {
      float4 v[MAXP][4];
#pragma unroll
      for (int pp = 0; pp < MAXP; ++pp) {
        if (part0 + pp < nparts) {
          const int cp = c_first + part0 + pp;
          const int sl = (part0 + pp == 0) ? sl0 : 0;
          const float* src = p.ws + ((size_t)(cp * 2 + sl) * NB + ch * CH) * 128 + nl;
#pragma unroll
          for (int q = 0; q < 4; ++q)
            if (4 * q < live)
              v[pp][q] = make_float4(__ldcg(src + (4 * q) * 128), __ldcg(src + (4 * q + 1) * 128),
                                     __ldcg(src + (4 * q + 2) * 128), __ldcg(src + (4 * q + 3) * 128));
        }
      }
      if (part0 == 0) {
        tc_epilogue_load<NB, EPI>(p, in, tile, ch * CH, et);
        if (PROLOGUE && ch == 0) tc_row_prologue<NB, EPI>(p, s_rinv, s_pos, s_req, et);
      }
#pragma unroll
      for (int pp = 0; pp < MAXP; ++pp) {
        if (part0 + pp < nparts) {
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            if (4 * q < live) {
              acc[4 * q] += v[pp][q].x;
              acc[4 * q + 1] += v[pp][q].y;
              acc[4 * q + 2] += v[pp][q].z;
              acc[4 * q + 3] += v[pp][q].w;
            }
          }
        }
      }
    }
    ptx::named_bar_sync(1, 128);
#pragma unroll
    for (int j = 0; j < CH; ++j)
      sC[nl * SP + j] = (EPI == TC_RESID) ? acc[j] : acc[j] * s_rinv[ch * CH + j];
    ptx::named_bar_sync(1, 128);
    tc_epilogue_apply<NB, EPI>(p, in, sC, red, s_pos, s_req, tile, ch * CH, et);
  }
}

template <int NB, int EPI>
__global__ void __launch_bounds__(192, 1)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ TcParams p) {
  using Sh = TcShape<NB>;
  constexpr int S = Sh::S;
  constexpr uint32_t A_BYTES = Sh::A_BYTES, B_BYTES = Sh::B_BYTES, STAGE_B = Sh::STAGE_B;
  constexpr int CH = Sh::CH, SP = Sh::SP;
  constexpr bool ONE_MMA = Sh::ONE_MMA;
  constexpr int ACC_COLS = Sh::ACC_COLS;
  constexpr int NBUF = Sh::NBUF;
  constexpr uint32_t IDESC = ptx::idesc_bf16_f32(128, ONE_MMA ? 2 * NB : NB);

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = sA + S * A_BYTES;
  float* sC = reinterpret_cast<float*>(sB + S * STAGE_B);
  float* s_rinv = sC + 128 * SP;  // [NB] 1 / rms of each token row (normed inputs)
  float* red = s_rinv + NB;       // [64] cross-warp reduction scratch
  int* s_pos = reinterpret_cast<int*>(red + 64);  // [NB] cache position of each token row
  int* s_req = s_pos + NB;                        // [NB] request of each token row
  uint64_t* full = reinterpret_cast<uint64_t*>(s_req + NB);
  uint64_t* empty = full + S;
  uint64_t* acc_full = empty + S;   // [2]
  uint64_t* acc_empty = acc_full + 2;  // [2]
  uint64_t* drain = acc_empty + 2;     // [1]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  int* flags = reinterpret_cast<int*>(tmem_slot + 2);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int c = blockIdx.x;
  long long u0, u1;
  tc_range(c, p, u0, u1);

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      ptx::mbar_init(&full[s], 1);
      ptx::mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      ptx::mbar_init(&acc_full[b], 1);
      ptx::mbar_init(&acc_empty[b], 4);
    }
    ptx::mbar_init(drain, 1);
    flags[0] = 0;
    flags[1] = 0;
    ptx::fence_mbar_init();
  }
  if (warp == 1) ptx::tmem_alloc(tmem_slot, Sh::TMEM_COLS);
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  ptx::griddep_launch_dependents();

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      ptx::prefetch_tmap(&tmX);
      const uint64_t pol_w = ptx::policy_evict_first();
      const uint64_t pol_x = ptx::policy_evict_last();
      // Weight tiles do not depend on earlier kernels: the first ring's worth
      // is requested before waiting for the predecessor, the activation tiles
      // after it.
      const long long npre_ll = (u1 - u0) < S ? (u1 - u0) : S;
      const int npre = (int)npre_ll;
      for (int it = 0; it < npre; ++it) {
        const long long u = u0 + it;
        ptx::mbar_arrive_expect_tx(&full[it], A_BYTES + STAGE_B);
        ptx::bulk_load(sA + it * A_BYTES, p.w + (size_t)u * (128 * 64), A_BYTES, &full[it], pol_w);
      }
      // k-block of each unit, stepped (no division after the wait)
      int kb = (int)(u0 - (u0 / p.kb) * (long long)p.kb);
      ptx::griddep_wait();
      for (int it = 0; it < npre; ++it) {
        ptx::tma_load_2d(sB + it * STAGE_B, &tmX, &full[it], kb * 64, p.row0, pol_x);
        ptx::tma_load_2d(sB + it * STAGE_B + B_BYTES, &tmX, &full[it], kb * 64,
                         p.lo_row + p.row0, pol_x);
        kb = (kb + 1 == p.kb) ? 0 : kb + 1;
      }
      int it = npre;
      bool ok = true;
      for (long long u = u0 + npre; u < u1; ++u, ++it) {
        const int s = it % S;
        const uint32_t ph = (uint32_t)(it / S) & 1u;
        if (!ptx::mbar_wait(&empty[s], ph ^ 1u, p.timeout_ns)) {
          ok = false;
          break;
        }
        ptx::mbar_arrive_expect_tx(&full[s], A_BYTES + STAGE_B);
        ptx::bulk_load(sA + s * A_BYTES, p.w + (size_t)u * (128 * 64), A_BYTES, &full[s], pol_w);
        ptx::tma_load_2d(sB + s * STAGE_B, &tmX, &full[s], kb * 64, p.row0, pol_x);
        ptx::tma_load_2d(sB + s * STAGE_B + B_BYTES, &tmX, &full[s], kb * 64, p.lo_row + p.row0,
                         pol_x);
        kb = (kb + 1 == p.kb) ? 0 : kb + 1;
      }
      if (!ok) {
        atomicOr(p.err, kErrTimeout);
        flags[0] = 1;
      }
      // every copy this CTA issued has landed before the CTA may exit
      for (int j = (it > S ? it - S : 0); j < it; ++j)
        ptx::mbar_wait(&full[j % S], (uint32_t)(j / S) & 1u, ptx::kDrainNs);
    }
    __syncwarp();  // lanes 1..31 wait for lane 0: the warp reaches the barrier converged
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      int it = 0, seg = 0;
      bool ok = true;
      for (long long u = u0; u < u1 && ok; ++seg) {
        const int tile = (int)(u / p.kb);
        const long long tend = (long long)(tile + 1) * p.kb;
        const long long send = u1 < tend ? u1 : tend;
        const int buf = seg % NBUF;
        const uint32_t bph = (uint32_t)(seg / NBUF) & 1u;
        if (!ptx::mbar_wait(&acc_empty[buf], bph ^ 1u, p.timeout_ns)) {
          ok = false;
          break;
        }
        ptx::tc_fence_after();
        const uint32_t dt = tmem + (uint32_t)(buf * ACC_COLS);
        for (long long v = u; v < send; ++v, ++it) {
          const int s = it % S;
          const uint32_t ph = (uint32_t)(it / S) & 1u;
          if (!ptx::mbar_wait(&full[s], ph, p.timeout_ns)) {
            ok = false;
            break;
          }
          ptx::tc_fence_after();
          const uint64_t ad = ptx::sdesc_sw128(ptx::smem_u32(sA + s * A_BYTES));
          const uint64_t bh = ptx::sdesc_sw128(ptx::smem_u32(sB + s * STAGE_B));
          const uint64_t bl = ptx::sdesc_sw128(ptx::smem_u32(sB + s * STAGE_B + B_BYTES));
          // the operand is x = hi + lo (two bf16 parts), so the weights see x
          // to about 16 significant bits
#pragma unroll
          for (int kk = 0; kk < 4; ++kk) {
            const uint32_t acc = (v > u || kk > 0) ? 1u : 0u;
            if (ONE_MMA) {
              ptx::mma_bf16(dt, ad + 2 * kk, bh + 2 * kk, IDESC, acc);
            } else {
              ptx::mma_bf16(dt, ad + 2 * kk, bh + 2 * kk, IDESC, acc);
              ptx::mma_bf16(dt + NB, ad + 2 * kk, bl + 2 * kk, IDESC, acc);
            }
          }
          ptx::mma_commit(&empty[s]);
        }
        if (!ok) break;
        ptx::mma_commit(&acc_full[buf]);
        u = send;
      }
      if (!ok) {
        atomicOr(p.err, kErrTimeout);
        flags[0] = 1;
      }
      // every MMA this thread issued has completed before TMEM is freed
      ptx::mma_commit(drain);
      ptx::mbar_wait(drain, 0, ptx::kDrainNs);
    }
    __syncwarp();
  } else {
    // ---------------- epilogue: warps 2..5, one TMEM lane each ----------------
    ptx::griddep_wait();  // the epilogue reads and writes the predecessors' outputs
    const int q4 = warp & 3;
    const int nl = q4 * 32 + lane;  // tile row this thread drains
    const int et = threadIdx.x - 64;
    tc_row_prologue<NB, EPI>(p, s_rinv, s_pos, s_req, et);
    const int nchunks = (p.rows + CH - 1) / CH;
    const int first_tile = (int)(u0 / p.kb);
    int seg = 0;
    for (long long u = u0; u < u1; ++seg) {
      const int tile = (int)(u / p.kb);
      const long long tstart = (long long)tile * p.kb, tend = tstart + p.kb;
      const long long send = u1 < tend ? u1 : tend;
      const bool whole = (u == tstart && send == tend);
      const int buf = seg % NBUF;
      const uint32_t bph = (uint32_t)(seg / NBUF) & 1u;
      if (!ptx::group_all(ptx::mbar_wait(&acc_full[buf], bph, p.timeout_ns), 1, 128)) {
        if (et == 0) atomicOr(p.err, kErrTimeout);
        break;  // every epilogue thread leaves together
      }
      ptx::tc_fence_after();
      const uint32_t tbase = tmem + (uint32_t)(buf * ACC_COLS) + ((uint32_t)(q4 * 32) << 16);
      if (EPI == TC_PART) {
        // this CTA's k-block sums for its tile, unscaled, [row][tile row]
        float* dst = p.part + ((size_t)c * p.part_ld + p.row0) * 128 + nl;
        for (int ch = 0; ch < nchunks; ++ch) {
          uint32_t v[16];
          tc_load_acc<NB>(tbase, ch, v);
#pragma unroll
          for (int j = 0; j < CH; ++j)
            if (ch * CH + j < p.rows) dst[(size_t)(ch * CH + j) * 128] = __uint_as_float(v[j]);
        }
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(&acc_empty[buf]);
      } else if (whole) {
        for (int ch = 0; ch < nchunks; ++ch) {
          uint32_t v[16];
          tc_load_acc<NB>(tbase, ch, v);
          ptx::named_bar_sync(1, 128);
#pragma unroll
          for (int j = 0; j < CH; ++j)
            sC[nl * SP + j] = (EPI == TC_RESID) ? __uint_as_float(v[j])
                                                : __uint_as_float(v[j]) * s_rinv[ch * CH + j];
          ptx::named_bar_sync(1, 128);
          tc_epilogue_chunk<NB, EPI>(p, sC, red, s_pos, s_req, tile, ch * CH, et);
        }
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(&acc_empty[buf]);
      } else {
        const int slot = (tile == first_tile) ? 0 : 1;
        // partial tile, laid out [NB][128]: a warp's stores of one token row
        // are 32 consecutive floats, and so are the finishing loads
        float* wsp = p.ws + (size_t)(c * 2 + slot) * NB * 128 + nl;
        for (int ch = 0; ch < nchunks; ++ch) {
          uint32_t v[16];
          tc_load_acc<NB>(tbase, ch, v);
#pragma unroll
          for (int j = 0; j < 16; ++j) wsp[(size_t)(ch * CH + j) * 128] = __uint_as_float(v[j]);
        }
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(&acc_empty[buf]);
        if (p.defer) {  // finished by tc_resid_finish_kernel, launched next
          u = send;
          continue;
        }
        // the last CTA to store a part of this tile adds the parts, in CTA
        // order whichever CTA that is, and applies the epilogue
        __threadfence();
        ptx::named_bar_sync(1, 128);
        const int c_first = tc_owner(tstart, p), c_last = tc_owner(tend - 1, p);
        const int nparts = c_last - c_first + 1;
        if (et == 0) flags[1] = (atomicAdd(&p.counters[tile], 1) == nparts - 1) ? 1 : 0;
        ptx::named_bar_sync(1, 128);
        const int last = flags[1];
        ptx::named_bar_sync(1, 128);
        if (last) {
          __threadfence();
          tc_reduce_tile<NB, EPI, 6>(p, sC, s_rinv, red, s_pos, s_req, tile, c_first, nparts, nl, et);
          if (et == 0) p.counters[tile] = 0;  // ready for the next launch
        }
      }
      u = send;
    }
  }

  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, Sh::TMEM_COLS);
  }
}

// The residual epilogue of a stream-K launch's split tiles, one CTA of 128
// threads per (tile, token row): thread n adds the parts of tile row n in CTA
// order, adds the residual, writes h and the next operand (hi, lo) and takes
// its share of the row's sum of squares -- the arithmetic of
// tc_reduce_tile + TC_RESID, with every load of a thread issued first.
template <int NB>
__global__ void __launch_bounds__(128) tc_resid_finish_kernel(const __grid_constant__ TcParams p) {
  __shared__ float red[4];
  const int tile = blockIdx.x, m = blockIdx.y, n = threadIdx.x;
  const long long tstart = (long long)tile * p.kb, tend = tstart + p.kb;
  const int c_first = tc_owner(tstart, p), c_last = tc_owner(tend - 1, p);
  // slot 1 holds a CTA's last segment when it began in an earlier tile: only
  // the first part can be one
  const int sl0 = (int)(tc_start(c_first, p) / p.kb) != tile ? 1 : 0;
  const int col = tile * 128 + n;
  // the next norm's gain is a weight, written by no kernel: its load (often
  // from HBM, busy with the next projection's weight stream) overlaps the wait
  const float gn = c_last != c_first ? __ldg(p.g_next + col) : 0.f;
  ptx::griddep_wait();
  ptx::griddep_launch_dependents();
  if (c_last == c_first) return;  // a whole tile, finished by its GEMM CTA
  const int nparts = c_last - c_first + 1;
  const size_t at = (size_t)(p.row0 + m) * p.N + col;
  const float h0 = p.h[at];
  const float* src = p.ws + (size_t)m * 128 + n;
  float acc = 0.f;
  for (int part0 = 0; part0 < nparts; part0 += 16) {
    float v[16];
#pragma unroll
    for (int pp = 0; pp < 16; ++pp) {
      v[pp] = 0.f;
      if (part0 + pp < nparts) {
        const int cp = c_first + part0 + pp;
        const int sl = (part0 + pp == 0) ? sl0 : 0;
        v[pp] = __ldcg(src + (size_t)(cp * 2 + sl) * NB * 128);
      }
    }
#pragma unroll
    for (int pp = 0; pp < 16; ++pp)
      if (part0 + pp < nparts) acc += v[pp];
  }
  const float hn = h0 + acc;
  p.h[at] = hn;
  const float xv = hn * gn;
  const bf16 xh = __float2bfloat16_rn(xv);
  p.xn[at] = xh;
  p.xn[at + (size_t)p.lo_row * p.N] = __float2bfloat16_rn(xv - __bfloat162float(xh));
  float sq = hn * hn;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xFFFFFFFFu, sq, o);
  if ((n & 31) == 0) red[n >> 5] = sq;
  __syncthreads();
  if (n == 0) p.ss[(size_t)tile * p.ss_ld + p.row0 + m] = ((red[0] + red[1]) + red[2]) + red[3];
}

template <int NB, int EPI>
cudaError_t tc_gemm_launch(const CUtensorMap& x, const TcParams& p, cudaStream_t st) {
  constexpr uint32_t smem = TcShape<NB>::SMEM;
  // set once per instantiation; a function-local static is initialised
  // exactly once even when several host threads launch at the same time
  static const cudaError_t attr = cudaFuncSetAttribute(
      tc_gemm_kernel<NB, EPI>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (attr != cudaSuccess) return attr;
  cudaError_t e = launch_pdl(tc_gemm_kernel<NB, EPI>, dim3(p.grid), dim3(192), smem, st, x, p);
  if (e != cudaSuccess || !p.defer || p.grid < 2) return e;
  // only the residual projections leave their split tiles to a finishing kernel
  if (EPI != TC_RESID) return cudaErrorInvalidValue;
  return launch_pdl(tc_resid_finish_kernel<NB>, dim3(p.n_tiles, p.rows), dim3(128), 0, st, p);
}

template <int EPI>
cudaError_t tc_gemm_dispatch(int nb, const CUtensorMap& x, const TcParams& p, cudaStream_t st) {
  switch (nb) {
    case 16: return tc_gemm_launch<16, EPI>(x, p, st);
    case 32: return tc_gemm_launch<32, EPI>(x, p, st);
    case 48: return tc_gemm_launch<48, EPI>(x, p, st);
    case 64: return tc_gemm_launch<64, EPI>(x, p, st);
    case 96: return tc_gemm_launch<96, EPI>(x, p, st);
    case 128: return tc_gemm_launch<128, EPI>(x, p, st);
    case 160: return tc_gemm_launch<160, EPI>(x, p, st);
    case 192: return tc_gemm_launch<192, EPI>(x, p, st);
    case 224: return tc_gemm_launch<224, EPI>(x, p, st);
    case 256: return tc_gemm_launch<256, EPI>(x, p, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace as2d
