// k_mk.cu -- the whole verification pass as one persistent, cooperative
// kernel (one CTA per SM) for calls of at most 32 token rows.  Opt-in
// (AS2D_PERSISTENT=1 in the environment when the state is created): on the
// 7B-class workload it is currently slower than the kernel sequence.
//
// The pass is a fixed list of phases: embedding; per layer QKV + RoPE + KV
// append, split-KV attention, merge, O + residual, gate/up + SwiGLU, down +
// residual; LM head + argmax; accept scan.  Every CTA walks the list in order.
//   warp 0  streams the weight tiles of every projection phase, one after the
//           other, into a shared-memory ring; weights never depend on earlier
//           phases, so this stream never waits on other CTAs and runs ahead
//           into the next projection while the current one finishes;
//   warp 6  loads a projection's activation tiles once every CTA has finished
//           the phase that produced them (per-phase arrival counters);
//   warp 1  issues the tcgen05 MMAs (accumulators in TMEM);
//   warps 2-5 run the fused epilogues and the non-projection phases, then
//           mark the phase done for this CTA.
// The kernels' arithmetic is shared with the multi-kernel path (same device
// functions, same stream-K partition per projection), so results do not
// depend on which path ran them.  All waits are bounded in time.
#include "attn_dev.cuh"
#include "gemm_tc.cuh"
#include "small_dev.cuh"

#include <cstdlib>
#include <vector>

namespace as2d {

enum MkKind : int { MK_EMBED = 0, MK_GEMM = 1, MK_ATTN = 2, MK_MERGE = 3, MK_ACCEPT = 4 };

// One phase of the pass (built once per state, read by every CTA).
struct MkPhase {
  int kind, epi, xmap, layer;
  const bf16* w;          // packed weights (projection phases)
  int N, K, n_tiles, kb;
  long long units;
  int grid;               // CTAs that share the units (the multi-kernel grid)
  const float* g_next;    // residual phases: gain of the next norm
};

struct MkMaps {
  CUtensorMap m[3];       // activation operands: xn, ao, u
};

struct MkArgs {
  RowMap rm;
  const MkPhase* phases;
  int n_phases;
  unsigned int* bar;       // per-phase arrival counters (monotonic over calls)
  unsigned int bar_target; // grid x call number
  unsigned long long timeout_ns;
  TcParams tp;             // fields shared by every projection phase
  attn::AttnArgs attn;     // fields shared by every attention phase
  int attn_parts, nkv, nq;
  AcceptArgs acc;
  const bf16* embed;
  const float* g0;
  const int32_t* cand;
  const int32_t* root;
  const int32_t* len;
  int32_t* err;            // [0] error bits, [1 + b] bad-token flags
  float2* rope;
  float* h;
  bf16* xn;
  float* ss;
  int rows_alloc, hidden, head_dim, vocab;
  double theta;
};

namespace {

template <int NB>
__device__ __forceinline__ void mk_epilogue_chunk(int epi, const TcParams& p, const float* sC,
                                                  float* red, const int* s_pos, const int* s_req,
                                                  int tile, int m0, int et) {
  switch (epi) {
    case TC_QKV: tc_epilogue_chunk<NB, TC_QKV>(p, sC, red, s_pos, s_req, tile, m0, et); break;
    case TC_RESID: tc_epilogue_chunk<NB, TC_RESID>(p, sC, red, s_pos, s_req, tile, m0, et); break;
    case TC_SWIGLU: tc_epilogue_chunk<NB, TC_SWIGLU>(p, sC, red, s_pos, s_req, tile, m0, et); break;
    default: tc_epilogue_chunk<NB, TC_LOGITS>(p, sC, red, s_pos, s_req, tile, m0, et); break;
  }
}

template <int NB>
__device__ __forceinline__ void mk_finish_tile(int epi, const TcParams& p, float* sC,
                                               float* s_rinv, float* red, int* s_pos,
                                               int* s_req, int tile, int c_first,
                                               int nparts, int nl, int et) {
  switch (epi) {
    case TC_QKV:
      tc_reduce_tile<NB, TC_QKV, 4>(p, sC, s_rinv, red, s_pos, s_req, tile, c_first, nparts, nl, et);
      break;
    case TC_RESID:
      tc_reduce_tile<NB, TC_RESID, 4>(p, sC, s_rinv, red, s_pos, s_req, tile, c_first, nparts, nl, et);
      break;
    case TC_SWIGLU:
      tc_reduce_tile<NB, TC_SWIGLU, 4>(p, sC, s_rinv, red, s_pos, s_req, tile, c_first, nparts, nl, et);
      break;
    default:
      tc_reduce_tile<NB, TC_LOGITS, 4>(p, sC, s_rinv, red, s_pos, s_req, tile, c_first, nparts, nl, et);
      break;
  }
}

constexpr int kMkThreads = 224;  // 7 warps

template <int NB>
struct MkShape {
  static constexpr int SW = NB == 16 ? 8 : 7;          // weight ring (16 KB stages)
  static constexpr int SX = NB == 16 ? 8 : 6;          // activation ring (hi + lo tiles)
  static constexpr uint32_t W_BYTES = 128 * 64 * 2;
  static constexpr uint32_t X_HALF = NB * 64 * 2;
  static constexpr uint32_t X_BYTES = 2 * X_HALF;
  static constexpr int CH = 16, SP = 17;
  static constexpr int ACC_COLS = 2 * NB;              // hi, lo results
  static constexpr uint32_t TMEM_COLS = 2 * ACC_COLS < 32 ? 32 : 2 * ACC_COLS;
  // byte offsets in dynamic shared memory (after 1024-byte alignment)
  static constexpr uint32_t OFF_W = 0;
  static constexpr uint32_t OFF_X = OFF_W + SW * W_BYTES;
  static constexpr uint32_t OFF_C = OFF_X + SX * X_BYTES;
  static constexpr uint32_t OFF_RINV = OFF_C + 128 * SP * 4;
  static constexpr uint32_t OFF_RED = OFF_RINV + NB * 4;
  static constexpr uint32_t OFF_POS = OFF_RED + 64 * 4;
  static constexpr uint32_t OFF_REQ = OFF_POS + NB * 4;
  static constexpr uint32_t OFF_K = (OFF_REQ + NB * 4 + 15) / 16 * 16;
  static constexpr uint32_t OFF_V = OFF_K + 64 * attn::kPitch * 2;
  static constexpr uint32_t OFF_MW = OFF_V + 64 * attn::kPitch * 2;
  static constexpr uint32_t OFF_ML = OFF_MW + attn::kMaxParts * 4;
  static constexpr uint32_t OFF_P = (OFF_ML + 16 + 63) / 64 * 64;
  static constexpr uint32_t OFF_BAR = (OFF_P + sizeof(TcParams) + 7) / 8 * 8;
  static constexpr uint32_t N_BARS = 2 * SW + 2 * SX + 5;
  static constexpr uint32_t OFF_TMEM = OFF_BAR + N_BARS * 8;  // TMEM address, then a flag
  static constexpr uint32_t SMEM = 1024 + OFF_TMEM + 16;
};

__device__ __forceinline__ long long mk_start(int c, long long units, int grid) {
  return c < grid ? (long long)c * units / grid : units;
}

// Wait until every CTA has finished phase `ph` of this call.
__device__ __forceinline__ bool mk_wait(const unsigned int* bar, int ph, unsigned int target,
                                        unsigned long long limit_ns) {
  if (ph < 0) return true;
  unsigned int v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(bar + ph) : "memory");
  if ((int)(v - target) >= 0) return true;
  const unsigned long long t0 = ptx::globaltimer_ns();
  for (;;) {
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(bar + ph) : "memory");
    if ((int)(v - target) >= 0) return true;
    if (ptx::globaltimer_ns() - t0 > limit_ns) return false;
    __nanosleep(64);
  }
}

__device__ __forceinline__ void fence_proxy_async() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

// Embedding row r by 128 threads: the same arithmetic as embed_kernel.
__device__ __forceinline__ void mk_embed_row(const MkArgs& a, int r, int et, float* red) {
  const RowMap& m = a.rm;
  const int b = row_request(m, r);
  const int i = r - m.start[b];
  const int H = a.hidden, d = a.head_dim;
  if (et < d / 2) {
    const double ang = (double)(a.len[b] + i) * pow(a.theta, -2.0 * (double)et / (double)d);
    double sn, cs;
    sincos(ang, &sn, &cs);
    a.rope[(size_t)r * (d / 2) + et] = make_float2((float)cs, (float)sn);
  }
  int tok = (i == 0) ? a.root[b] : a.cand[m.start[b] - b + i - 1];
  if (tok < 0 || tok >= a.vocab) {
    if (et == 0) {
      atomicOr(a.err, kErrBadToken);
      a.err[1 + b] = 1;
    }
    tok = 0;
  }
  embed_row_body(a.embed + (size_t)tok * H, a.g0, H, r, a.rows_alloc, a.h, a.xn, a.ss, et, 128,
                 red, 1);
}

}  // namespace

template <int NB, int D>
__global__ void __launch_bounds__(kMkThreads, 1)
    mk_kernel(const __grid_constant__ MkMaps maps, const __grid_constant__ MkArgs a) {
  using Sh = MkShape<NB>;
  constexpr int SW = Sh::SW, SX = Sh::SX, CH = Sh::CH, SP = Sh::SP;
  constexpr uint32_t IDESC = ptx::idesc_bf16_f32(128, 2 * NB);

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* sW = smem + Sh::OFF_W;
  uint8_t* sX = smem + Sh::OFF_X;
  float* sC = reinterpret_cast<float*>(smem + Sh::OFF_C);
  float* s_rinv = reinterpret_cast<float*>(smem + Sh::OFF_RINV);
  float* red = reinterpret_cast<float*>(smem + Sh::OFF_RED);
  int* s_pos = reinterpret_cast<int*>(smem + Sh::OFF_POS);
  int* s_req = reinterpret_cast<int*>(smem + Sh::OFF_REQ);
  auto sK = reinterpret_cast<bf16(*)[attn::kPitch]>(smem + Sh::OFF_K);
  auto sV = reinterpret_cast<bf16(*)[attn::kPitch]>(smem + Sh::OFF_V);
  float* mw = reinterpret_cast<float*>(smem + Sh::OFF_MW);
  float* ml = reinterpret_cast<float*>(smem + Sh::OFF_ML);
  TcParams* sP = reinterpret_cast<TcParams*>(smem + Sh::OFF_P);
  uint64_t* wfull = reinterpret_cast<uint64_t*>(smem + Sh::OFF_BAR);
  uint64_t* wempty = wfull + SW;
  uint64_t* xfull = wempty + SW;
  uint64_t* xempty = xfull + SX;
  uint64_t* acc_full = xempty + SX;   // [2]
  uint64_t* acc_empty = acc_full + 2;  // [2]
  uint64_t* drain = acc_empty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + Sh::OFF_TMEM);
  int* s_last = reinterpret_cast<int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int c = blockIdx.x, G = gridDim.x;
  const unsigned long long tmo = a.timeout_ns;

  if (threadIdx.x == 0) {
    for (int s = 0; s < SW; ++s) {
      ptx::mbar_init(&wfull[s], 1);
      ptx::mbar_init(&wempty[s], 1);
    }
    for (int s = 0; s < SX; ++s) {
      ptx::mbar_init(&xfull[s], 1);
      ptx::mbar_init(&xempty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      ptx::mbar_init(&acc_full[b], 1);
      ptx::mbar_init(&acc_empty[b], 4);
    }
    ptx::mbar_init(drain, 1);
    ptx::fence_mbar_init();
  }
  if (warp == 1) ptx::tmem_alloc(tmem_slot, Sh::TMEM_COLS);
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ---------------- weight stream, all projections in order ----------------
    if (lane == 0) {
      const uint64_t pol = ptx::policy_evict_first();
      int wit = 0;
      bool ok = true;
      for (int ph = 0; ph < a.n_phases && ok; ++ph) {
        const MkPhase& P = a.phases[ph];
        if (P.kind != MK_GEMM) continue;
        const long long u0 = mk_start(c, P.units, P.grid), u1 = mk_start(c + 1, P.units, P.grid);
        for (long long u = u0; u < u1; ++u, ++wit) {
          const int s = wit % SW;
          if (!ptx::mbar_wait(&wempty[s], ((uint32_t)(wit / SW) & 1u) ^ 1u, tmo)) {
            ok = false;
            break;
          }
          ptx::mbar_arrive_expect_tx(&wfull[s], Sh::W_BYTES);
          ptx::bulk_load(sW + s * Sh::W_BYTES, P.w + (size_t)u * (128 * 64), Sh::W_BYTES, &wfull[s],
                         pol);
        }
      }
      if (!ok) atomicOr(a.err, kErrTimeout);
      for (int j = (wit > SW ? wit - SW : 0); j < wit; ++j)
        ptx::mbar_wait(&wfull[j % SW], (uint32_t)(j / SW) & 1u, tmo);
    }
    __syncwarp();
  } else if (warp == 6) {
    // ---------------- activation tiles, after their producing phase ----------------
    if (lane == 0) {
      const uint64_t pol = ptx::policy_evict_last();
      int xit = 0;
      bool ok = true;
      for (int ph = 0; ph < a.n_phases && ok; ++ph) {
        const MkPhase& P = a.phases[ph];
        if (P.kind != MK_GEMM) continue;
        const long long u0 = mk_start(c, P.units, P.grid), u1 = mk_start(c + 1, P.units, P.grid);
        if (u0 == u1) continue;
        if (!mk_wait(a.bar, ph - 1, a.bar_target, tmo)) {
          ok = false;
          break;
        }
        fence_proxy_async();
        const CUtensorMap* xm = &maps.m[P.xmap];
        for (long long u = u0; u < u1; ++u, ++xit) {
          const int s = xit % SX;
          if (!ptx::mbar_wait(&xempty[s], ((uint32_t)(xit / SX) & 1u) ^ 1u, tmo)) {
            ok = false;
            break;
          }
          const int kb = (int)(u % P.kb);
          ptx::mbar_arrive_expect_tx(&xfull[s], Sh::X_BYTES);
          ptx::tma_load_2d(sX + s * Sh::X_BYTES, xm, &xfull[s], kb * 64, 0, pol);
          ptx::tma_load_2d(sX + s * Sh::X_BYTES + Sh::X_HALF, xm, &xfull[s], kb * 64, a.rows_alloc,
                           pol);
        }
      }
      if (!ok) atomicOr(a.err, kErrTimeout);
      for (int j = (xit > SX ? xit - SX : 0); j < xit; ++j)
        ptx::mbar_wait(&xfull[j % SX], (uint32_t)(j / SX) & 1u, tmo);
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      int wit = 0, xit = 0, seg = 0;
      bool ok = true;
      for (int ph = 0; ph < a.n_phases && ok; ++ph) {
        const MkPhase& P = a.phases[ph];
        if (P.kind != MK_GEMM) continue;
        const long long u0 = mk_start(c, P.units, P.grid), u1 = mk_start(c + 1, P.units, P.grid);
        for (long long u = u0; u < u1 && ok; ++seg) {
          const int tile = (int)(u / P.kb);
          const long long tend = (long long)(tile + 1) * P.kb;
          const long long send = u1 < tend ? u1 : tend;
          const int buf = seg & 1;
          if (!ptx::mbar_wait(&acc_empty[buf], ((uint32_t)(seg >> 1) & 1u) ^ 1u, tmo)) {
            ok = false;
            break;
          }
          ptx::tc_fence_after();
          const uint32_t dt = tmem + (uint32_t)(buf * Sh::ACC_COLS);
          for (long long v = u; v < send; ++v, ++wit, ++xit) {
            const int sw = wit % SW, sx = xit % SX;
            if (!ptx::mbar_wait(&wfull[sw], (uint32_t)(wit / SW) & 1u, tmo) ||
                !ptx::mbar_wait(&xfull[sx], (uint32_t)(xit / SX) & 1u, tmo)) {
              ok = false;
              break;
            }
            ptx::tc_fence_after();
            const uint64_t ad = ptx::sdesc_sw128(ptx::smem_u32(sW + sw * Sh::W_BYTES));
            const uint64_t bd = ptx::sdesc_sw128(ptx::smem_u32(sX + sx * Sh::X_BYTES));
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              ptx::mma_bf16(dt, ad + 2 * kk, bd + 2 * kk, IDESC, (v > u || kk > 0) ? 1u : 0u);
            ptx::mma_commit(&wempty[sw]);
            ptx::mma_commit(&xempty[sx]);
          }
          if (!ok) break;
          ptx::mma_commit(&acc_full[buf]);
          u = send;
        }
      }
      if (!ok) atomicOr(a.err, kErrTimeout);
      ptx::mma_commit(drain);
      ptx::mbar_wait(drain, 0, tmo);
    }
    __syncwarp();
  } else {
    // ---------------- epilogue and the other phases: warps 2..5 ----------------
    const int et = threadIdx.x - 64;
    const int q4 = warp & 3;
    const int nl = q4 * 32 + lane;
    int seg = 0;
    bool ok = true;
    for (int ph = 0; ph < a.n_phases && ok; ++ph) {
      const MkPhase& P = a.phases[ph];
      // one thread waits for the previous phase; the outcome is shared so that
      // the whole group continues or stops together
      if (et == 0) *s_last = mk_wait(a.bar, ph - 1, a.bar_target, tmo) ? 1 : 0;
      ptx::named_bar_sync(1, 128);
      if (!*s_last) {
        ok = false;
        break;
      }
      __threadfence();
      if (P.kind == MK_EMBED) {
        for (int r = c; r < a.rm.rows; r += G) mk_embed_row(a, r, et, red);
      } else if (P.kind == MK_GEMM) {
        {
          // the shared projection fields, copied by the group, then this phase's
          static_assert(sizeof(TcParams) % 4 == 0, "copied in 4-byte words");
          const int* src = reinterpret_cast<const int*>(&a.tp);
          int* dst = reinterpret_cast<int*>(sP);
          for (int i = et; i < (int)(sizeof(TcParams) / 4); i += 128) dst[i] = src[i];
          ptx::named_bar_sync(1, 128);
          if (et == 0) {
            sP->w = P.w;
            sP->N = P.N;
            sP->K = P.K;
            sP->n_tiles = P.n_tiles;
            sP->kb = P.kb;
            sP->units = P.units;
            sP->grid = P.grid;
            sP->layer = P.layer;
            sP->g_next = P.g_next;
          }
        }
        ptx::named_bar_sync(1, 128);
        const TcParams& p = *sP;
        switch (P.epi) {
          case TC_QKV: tc_row_prologue<NB, TC_QKV>(p, s_rinv, s_pos, s_req, et); break;
          case TC_SWIGLU: tc_row_prologue<NB, TC_SWIGLU>(p, s_rinv, s_pos, s_req, et); break;
          case TC_LOGITS: tc_row_prologue<NB, TC_LOGITS>(p, s_rinv, s_pos, s_req, et); break;
          default: break;
        }
        const long long u0 = mk_start(c, P.units, P.grid), u1 = mk_start(c + 1, P.units, P.grid);
        const int nchunks = (p.rows + CH - 1) / CH;
        const int first_tile = (int)(u0 / P.kb);
        for (long long u = u0; u < u1; ++seg) {
          const int tile = (int)(u / P.kb);
          const long long tstart = (long long)tile * P.kb, tend = tstart + P.kb;
          const long long send = u1 < tend ? u1 : tend;
          const bool whole = (u == tstart && send == tend);
          const int buf = seg & 1;
          if (!ptx::group_all(ptx::mbar_wait(&acc_full[buf], (uint32_t)(seg >> 1) & 1u, tmo), 1,
                              128)) {
            ok = false;
            break;
          }
          ptx::tc_fence_after();
          const uint32_t tbase = tmem + (uint32_t)(buf * Sh::ACC_COLS) + ((uint32_t)(q4 * 32) << 16);
          if (whole) {
            for (int ch = 0; ch < nchunks; ++ch) {
              uint32_t v[16];
              tc_load_acc<NB>(tbase, ch, v);
              ptx::named_bar_sync(1, 128);
#pragma unroll
              for (int j = 0; j < CH; ++j)
                sC[nl * SP + j] = (P.epi == TC_RESID) ? __uint_as_float(v[j])
                                                      : __uint_as_float(v[j]) * s_rinv[ch * CH + j];
              ptx::named_bar_sync(1, 128);
              mk_epilogue_chunk<NB>(P.epi, p, sC, red, s_pos, s_req, tile, ch * CH, et);
            }
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&acc_empty[buf]);
          } else {
            const int slot = (tile == first_tile) ? 0 : 1;
            float* wsp = p.ws + (size_t)(c * 2 + slot) * NB * 128 + nl;  // [NB][128]
            for (int ch = 0; ch < nchunks; ++ch) {
              uint32_t v[16];
              tc_load_acc<NB>(tbase, ch, v);
#pragma unroll
              for (int j = 0; j < 16; ++j) wsp[(size_t)(ch * CH + j) * 128] = __uint_as_float(v[j]);
            }
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&acc_empty[buf]);
            // the last CTA to finish a part of this tile adds the parts (in
            // CTA order, as the GEMM kernel does) and applies the epilogue
            __threadfence();
            ptx::named_bar_sync(1, 128);
            const int c_first = tc_owner(tstart, p), c_last = tc_owner(tend - 1, p);
            const int nparts = c_last - c_first + 1;
            if (et == 0) *s_last = (atomicAdd(&p.counters[tile], 1) == nparts - 1) ? 1 : 0;
            ptx::named_bar_sync(1, 128);
            const int last = *s_last;
            ptx::named_bar_sync(1, 128);
            if (last) {
              __threadfence();
              mk_finish_tile<NB>(P.epi, p, sC, s_rinv, red, s_pos, s_req, tile, c_first, nparts,
                                 nl, et);
              if (et == 0) p.counters[tile] = 0;
            }
          }
          u = send;
        }
      } else if (P.kind == MK_ATTN) {
        const int items = a.attn_parts * a.nkv * a.rm.batch;
        for (int it = c; it < items; it += G) {
          const int part = it % a.attn_parts, rest = it / a.attn_parts;
          attn::part_item<D>(a.attn, P.layer, part, rest % a.nkv, rest / a.nkv, sK, sV, et, 128, 1);
        }
      } else if (P.kind == MK_MERGE) {
        const int items = a.rm.rows * a.nq;
        for (int it = c; it < items; it += G)
          attn::merge_item<D, 16>(a.attn, it / a.nq, it % a.nq, mw, ml, et, 128, 1);
      } else if (P.kind == MK_ACCEPT) {
        if (c == 0)
          for (int b = et >> 5; b < a.rm.batch; b += 4) accept_request(a.acc, b, lane);
      }
      // this CTA is done with phase ph
      ptx::named_bar_sync(1, 128);
      if (et == 0) {
        __threadfence();
        fence_proxy_async();
        atomicAdd(a.bar + ph, 1u);
      }
    }
    if (!ok && et == 0) atomicOr(a.err, kErrTimeout);
  }

  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, Sh::TMEM_COLS);
  }
}

// ---- host side ----------------------------------------------------------------

namespace {

bool mk_enabled() {
  static const bool v = [] {
    const char* e = getenv("AS2D_PERSISTENT");
    return e && e[0] == '1';
  }();
  return v;
}

template <int NB, int D>
cudaError_t mk_launch_t(const MkMaps& maps, const MkArgs& a, int grid, cudaStream_t st) {
  constexpr uint32_t smem = MkShape<NB>::SMEM;
  static const cudaError_t attr_e =
      cudaFuncSetAttribute(mk_kernel<NB, D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (attr_e != cudaSuccess) return attr_e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kMkThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, mk_kernel<NB, D>, maps, a);
}

template <int NB, int D>
bool mk_fits(int sm_count) {
  constexpr uint32_t smem = MkShape<NB>::SMEM;
  if (cudaFuncSetAttribute(mk_kernel<NB, D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)smem) != cudaSuccess)
    return false;
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, mk_kernel<NB, D>, kMkThreads, smem) !=
      cudaSuccess)
    return false;
  return per_sm >= 1 && sm_count > 0;
}

}  // namespace

cudaError_t mk_prepare(const Model& m, KvState& kv) {
  kv.mk_ok = false;
  if (!mk_enabled()) return cudaSuccess;
  const as2d_config& c = m.cfg;
  const bool d128 = c.head_dim == 128;
  const bool fits = d128 ? (mk_fits<16, 128>(m.sm_count) && mk_fits<32, 128>(m.sm_count))
                         : (mk_fits<16, 64>(m.sm_count) && mk_fits<32, 64>(m.sm_count));
  cudaGetLastError();
  if (!fits) return cudaSuccess;  // the multi-kernel path serves every call
  const int G = m.sm_count;
  std::vector<MkPhase> ph;
  auto gemm = [&](int epi, int xmap, int layer, const bf16* w, int N, int K, const float* gn) {
    MkPhase p{};
    p.kind = MK_GEMM;
    p.epi = epi;
    p.xmap = xmap;
    p.layer = layer;
    p.w = w;
    p.N = N;
    p.K = K;
    p.n_tiles = (N + 127) / 128;
    p.kb = (K + 63) / 64;
    p.units = (long long)p.n_tiles * p.kb;
    p.grid = (int)(p.units < G ? p.units : G);
    p.g_next = gn;
    ph.push_back(p);
  };
  auto other = [&](int kind, int layer) {
    MkPhase p{};
    p.kind = kind;
    p.layer = layer;
    ph.push_back(p);
  };
  other(MK_EMBED, 0);
  for (int l = 0; l < c.n_layers; ++l) {
    gemm(TC_QKV, 0, l, m.w_qkv[l], m.qkv_rows, c.hidden, nullptr);
    other(MK_ATTN, l);
    other(MK_MERGE, l);
    gemm(TC_RESID, 1, l, m.w_o[l], c.hidden, m.q_dim, m.mlp_norm[l]);
    gemm(TC_SWIGLU, 0, l, m.w_gu[l], 2 * c.ffn, c.hidden, nullptr);
    gemm(TC_RESID, 2, l, m.w_down[l], c.hidden, c.ffn,
         l + 1 < c.n_layers ? m.attn_norm[l + 1] : m.final_norm);
  }
  gemm(TC_LOGITS, 0, c.n_layers, m.lm_head, c.vocab, c.hidden, nullptr);
  other(MK_ACCEPT, 0);
  const size_t bytes = ph.size() * sizeof(MkPhase) + ph.size() * 4 + 256;
  cudaError_t e = cudaMalloc(&kv.mk_mem, bytes);
  if (e != cudaSuccess) return e;
  e = cudaMemcpy(kv.mk_mem, ph.data(), ph.size() * sizeof(MkPhase), cudaMemcpyHostToDevice);
  kv.mk_bar = reinterpret_cast<unsigned int*>((char*)kv.mk_mem + (ph.size() * sizeof(MkPhase) + 255) / 256 * 256);
  if (e == cudaSuccess) e = cudaMemset(kv.mk_bar, 0, ph.size() * 4);
  if (e != cudaSuccess) return e;
  kv.mk_n_phases = (int)ph.size();
  kv.mk_gen = 0;
  kv.mk_ok = true;
  return cudaSuccess;
}

bool mk_usable(const KvState& kv, int rows) { return kv.mk_ok && rows <= 32; }

cudaError_t launch_mk(const RowMap& rm, const Model& m, KvState& kv, const int32_t* cand,
                      const as2d_verify_out& out, cudaStream_t st) {
  const as2d_config& c = m.cfg;
  const int G = m.sm_count;
  MkArgs a{};
  a.rm = rm;
  a.phases = reinterpret_cast<const MkPhase*>(kv.mk_mem);
  a.n_phases = kv.mk_n_phases;
  a.bar = kv.mk_bar;
  a.bar_target = (unsigned int)G * (++kv.mk_gen);
  a.timeout_ns = 2000000000ull;
  TcParams& tp = a.tp;
  tp.h = kv.h;
  tp.u = kv.u;
  tp.q = kv.q;
  tp.kc = kv.k_cache;
  tp.vc = kv.v_cache;
  tp.rope = kv.rope;
  tp.len = kv.d_len;
  tp.batch = kv.batch;
  tp.cap = kv.capacity;
  tp.nq = c.n_q_heads;
  tp.nkv = c.n_kv_heads;
  tp.d = c.head_dim;
  tp.logits = out.logits;
  tp.best = kv.best;
  tp.xn = kv.xn;
  tp.ss = kv.ss;
  tp.ss_ld = kv.rows_alloc;
  tp.lo_row = kv.rows_alloc;
  tp.n_htiles = c.hidden / 128;
  tp.eps = c.rms_eps;
  tp.hidden = c.hidden;
  tp.rm = rm;
  tp.ws = kv.ws;
  tp.counters = kv.counters;
  tp.err = kv.d_err;
  tp.timeout_ns = a.timeout_ns;
  tp.row0 = 0;
  tp.rows = rm.rows;
  attn::AttnArgs& aa = a.attn;
  aa.rm = rm;
  aa.q = kv.q;
  aa.len = kv.d_len;
  aa.kc = kv.k_cache;
  aa.vc = kv.v_cache;
  aa.batch = kv.batch;
  aa.cap = kv.capacity;
  aa.nq = c.n_q_heads;
  aa.nkv = c.n_kv_heads;
  aa.qscale = 1.4426950408889634f / sqrtf((float)c.head_dim);
  aa.ws_o = kv.attn_o;
  aa.ws_ml = kv.attn_ml;
  aa.parts_max = kv.attn_parts;
  aa.qmax = kv.attn_qmax;
  aa.ao = kv.ao;
  aa.lo_row = kv.rows_alloc;
  int64_t max_len = 0;
  for (int b = 0; b < kv.batch; ++b) {
    const int64_t e = kv.len_upper[b] + (rm.start[b + 1] - rm.start[b]);
    max_len = e > max_len ? e : max_len;
  }
  a.attn_parts = (int)((max_len + 63) / 64);
  a.nkv = c.n_kv_heads;
  a.nq = c.n_q_heads;
  a.acc = AcceptArgs{rm, cand, kv.best, kv.d_len, kv.d_root, kv.d_err + 1, out.n_accepted,
                     out.correction_token, out.greedy};
  a.embed = m.embed;
  a.g0 = m.attn_norm[0];
  a.cand = cand;
  a.root = kv.d_root;
  a.len = kv.d_len;
  a.err = kv.d_err;
  a.rope = kv.rope;
  a.h = kv.h;
  a.xn = kv.xn;
  a.ss = kv.ss;
  a.rows_alloc = kv.rows_alloc;
  a.hidden = c.hidden;
  a.head_dim = c.head_dim;
  a.vocab = c.vocab;
  a.theta = (double)c.rope_theta;
  const int nb = nb_for_rows(rm.rows);
  MkMaps maps;
  maps.m[0] = kv.tm_xn[nb_index(nb)];
  maps.m[1] = kv.tm_ao[nb_index(nb)];
  maps.m[2] = kv.tm_u[nb_index(nb)];
  ++kv.launches;
  if (c.head_dim == 128)
    return nb == 16 ? mk_launch_t<16, 128>(maps, a, G, st) : mk_launch_t<32, 128>(maps, a, G, st);
  return nb == 16 ? mk_launch_t<16, 64>(maps, a, G, st) : mk_launch_t<32, 64>(maps, a, G, st);
}

}  // namespace as2d
