// k_pack.cu -- load-time re-layout of the weight matrices into the
// tile-major form the tensor-core GEMM streams.
//
// A logical matrix W [N][K] (N padded up to a multiple of 128 with zero rows,
// K a multiple of 64) is stored as N/128 x K/64 blocks in (tile, k-block)
// order; block (t, kb) holds rows [128 t, 128 t + 128) and columns
// [64 kb, 64 kb + 64) as 128 rows of 128 bytes, with the 16-byte chunk j of
// row r placed at chunk j ^ (r mod 8).  That is byte for byte the shared-memory
// image that a 128-byte-swizzled TMA tile load would produce, so a GEMM unit
// is one contiguous 16 KB bulk copy, and the units a CTA streams are
// consecutive in memory.
#include "as2d_internal.h"

namespace as2d {
namespace {

// Row sources of one packed matrix: plain concatenation of up to three
// segments (e.g. q, k, v projections), or gate/up interleaving (tile rows
// 0..63 from gate rows 64t.., 64..127 from up rows 64t..).
struct PackSrc {
  const bf16* seg[3];
  int seg_rows[3];
  int nseg;
  int interleave;  // 1: gate (seg 0) / up (seg 1) in blocks of 64 rows
  int n_rows;      // logical rows
  int K;
};

__global__ void __launch_bounds__(256) pack_kernel(PackSrc s, bf16* __restrict__ dst, int kb_count) {
  const int tile = blockIdx.x / kb_count, kb = blockIdx.x - tile * kb_count;
  bf16* blk = dst + (size_t)blockIdx.x * (128 * 64);
  for (int idx = threadIdx.x; idx < 128 * 8; idx += blockDim.x) {
    const int r = idx >> 3, j = idx & 7;
    const int R = tile * 128 + r;
    const bf16* src = nullptr;
    if (s.interleave) {
      const int f = (R >> 7) * 64 + (R & 63);
      if (f < s.seg_rows[0]) src = s.seg[(R & 64) ? 1 : 0] + (size_t)f * s.K;
    } else if (R < s.n_rows) {
      int rr = R, q = 0;
      while (q < s.nseg - 1 && rr >= s.seg_rows[q]) rr -= s.seg_rows[q++];
      src = s.seg[q] + (size_t)rr * s.K;
    }
    uint4 v = make_uint4(0, 0, 0, 0);
    if (src) v = *reinterpret_cast<const uint4*>(src + kb * 64 + j * 8);
    *reinterpret_cast<uint4*>(blk + r * 64 + ((j ^ (r & 7)) * 8)) = v;
  }
}

}  // namespace

size_t packed_elems(int n_rows, int K) { return (size_t)((n_rows + 127) / 128) * 128 * K; }

cudaError_t pack_weights(bf16* dst, int n_rows, int K, const void* const* segs,
                         const int* seg_rows, int nseg, bool interleave, cudaStream_t st) {
  PackSrc s{};
  for (int i = 0; i < nseg; ++i) {
    s.seg[i] = (const bf16*)segs[i];
    s.seg_rows[i] = seg_rows[i];
  }
  s.nseg = nseg;
  s.interleave = interleave ? 1 : 0;
  s.n_rows = n_rows;
  s.K = K;
  const int tiles = (n_rows + 127) / 128, kbs = K / 64;
  pack_kernel<<<tiles * kbs, 256, 0, st>>>(s, dst, kbs);
  return cudaGetLastError();
}

}  // namespace as2d
