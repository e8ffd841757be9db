// as2d_internal.h -- structures shared by the library's translation units.
// Not part of the C-ABI (include/as2d.h is).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <string>
#include <vector>

#include "as2d.h"

namespace as2d {

constexpr int kMaxBatch = AS2D_MAX_BATCH;
constexpr int kMaxK = AS2D_MAX_K;
constexpr int kMaxRows = kMaxBatch * (kMaxK + 1);
constexpr int kPrefillRows = 64;  // token rows of one prefill pass

typedef __nv_bfloat16 bf16;

// Row layout of one call: request b owns rows [start[b], start[b+1]); its
// candidates start at index start[b] - b of the packed candidate array.
// Passed by value to every kernel, so a call needs no host-to-device copy.
struct RowMap {
  int32_t batch;
  int32_t rows;
  int32_t start[kMaxBatch + 1];
};

__host__ __device__ inline int row_request(const RowMap& m, int r) {
  int b = 0;
  while (b + 1 < m.batch && m.start[b + 1] <= r) ++b;
  return b;
}

// Device error bits (ORed into KvState::d_err); the values of include/as2d.h's
// AS2D_DEVERR_* bits.
enum : int32_t {
  kErrBadToken = AS2D_DEVERR_BAD_TOKEN,
  kErrRollback = AS2D_DEVERR_ROLLBACK,
  kErrTimeout = AS2D_DEVERR_TIMEOUT,
  kErrCapacity = AS2D_DEVERR_CAPACITY,
};

// Whether a request of device-side length `len` has room for `rows` more
// cache entries.  A request that does not is skipped by every kernel that
// indexes the cache or the rotary table with its length (no key/value append,
// no attention, zero attention output); the embedding kernel flags it
// (kErrCapacity and the request's bad flag), and the accept scan then reports
// n_accepted = correction = -1 and leaves its length and root unchanged.
__host__ __device__ inline bool rows_fit(int len, int rows, int cap) {
  return len >= 0 && len <= cap - rows;
}

enum TcEpi { TC_RESID = 1, TC_SWIGLU = 2, TC_LOGITS = 3, TC_PART = 4 };

struct TcParams {
  const bf16* w;         // packed weight blocks (k_pack.cu), unit u at u * 8192
  int lo_row;            // operand buffers hold hi rows [0, R), lo rows [R, 2R): R
  int N, K;              // logical W is [N][K]
  int n_tiles, kb;       // 128-row tiles, 64-column k-blocks
  long long units;       // n_tiles * kb
  int grid;              // CTAs
  int split;             // TC_PART: CTAs per tile (K split), else 0 (stream-K)
  int defer;             // stream-K: split tiles are finished by tc_resid_finish_kernel
  float* part;           // TC_PART: [tile][split][part_ld][128] fp32 sums
  float* part_rinv;      // TC_PART: [part_ld] 1 / rms of each token row
  int part_ld;           // rows_alloc
  int rows;              // token rows handled by this launch
  int row0;              // first token row of this launch
  float* ws;             // [grid][2][NB][128] partial tiles
  int* counters;         // [n_tiles] arrivals; zero between launches
  int* err;
  unsigned long long timeout_ns;
  // epilogue operands
  float* h;              // RESID: h[m][n] += D (ld = N)
  bf16* u;               // SWIGLU: u[m][j], ld = N / 2
  float* logits;         // LOGITS (nullable), ld = N
  unsigned long long* best;
  // RMSNorm folded into the GEMMs: a RESID epilogue leaves, for the next
  // projection, xn = bf16(h * g_next) and per-128-column sums of h^2; the
  // next projection scales its accumulator by 1 / rms of its row.
  const float* g_next;   // RESID: gain of the norm that consumes h next
  bf16* xn;              // RESID: [rows][N] next operand
  float* ss;             // [N / 128][rows_alloc] partial sums of squares
  int ss_ld;             // rows_alloc
  int n_htiles;          // hidden / 128 (consumer side)
  float eps;
  int hidden;
  RowMap rm;
};

// Launch with programmatic stream serialization: the kernel may be scheduled
// while its predecessor in the stream is still running; every kernel of the
// library calls griddepcontrol.wait before it touches memory that an earlier
// kernel of the stream wrote.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t st, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, args...);
}

struct Model {
  as2d_config cfg;
  int qkv_rows;      // (n_q + 2 n_kv) * head_dim
  int q_dim;         // n_q * head_dim
  int kv_dim;        // n_kv * head_dim
  int sm_count;      // SMs the grids are sized for (the device's, or a budget)
  int device_sm_count;
  void* arena = nullptr;  // every weight below lives here
  size_t arena_bytes = 0;
  const bf16* embed = nullptr;    // [V][H]
  const bf16* lm_head = nullptr;  // logical [V][H], packed tile-major
  const float* final_norm = nullptr;
  // projection weights, packed tile-major (k_pack.cu)
  std::vector<const bf16*> w_qkv;   // logical [(nq + 2 nkv) d][H]: q rows, k rows, v rows
  std::vector<const bf16*> w_o;     // logical [H][nq d]
  std::vector<const bf16*> w_gu;    // logical [2F][H]: per 128 rows, 64 gate then 64 up
  std::vector<const bf16*> w_down;  // logical [H][F]
  std::vector<const float*> attn_norm, mlp_norm;  // fp32 gains [H]
};

// Token-row paddings of the tensor-core projections (the MMA's N): a call of
// `rows` token rows runs at the smallest one that holds them (at most 256 per
// launch).  A row's arithmetic does not depend on the padding.
constexpr int kNbCount = 10;
constexpr int kNbSet[kNbCount] = {16, 32, 48, 64, 96, 128, 160, 192, 224, 256};
inline int nb_index(int nb) {
  int i = 0;
  while (i + 1 < kNbCount && kNbSet[i] != nb) ++i;
  return i;
}
inline int nb_for_rows(int rows) {
  int i = 0;
  while (i + 1 < kNbCount && kNbSet[i] < rows) ++i;
  return kNbSet[i];
}

struct KvState {
  Model* model = nullptr;
  int batch = 0;
  int capacity = 0;
  bf16* k_cache = nullptr;  // [layers][batch][n_kv][cap][d]
  bf16* v_cache = nullptr;
  std::vector<int64_t> len_upper;  // host bound of each request's length
  // device state
  int32_t* d_len = nullptr;   // [batch]
  int32_t* d_root = nullptr;  // [batch]
  int32_t* d_err = nullptr;   // [1]
  // working memory, sized for batch * (max_k + 1) rows
  int max_k = kMaxK;         // most candidates (rows - 1) of one request in a call
  int max_rows = 0;
  void* work = nullptr;
  size_t work_bytes = 0;
  float* h = nullptr;        // [rows][H] residual stream, fp32
  // bf16 operand buffers hold hi rows [0, rows_alloc) then lo rows
  bf16* xn = nullptr;        // [2 rows][H] next projection's operand bf16(h * g)
  bf16* ao = nullptr;        // [2 rows][nq d] attention output
  bf16* u = nullptr;         // [2 rows][F] SwiGLU output
  unsigned long long* best = nullptr;  // [rows] packed (logit, index) maxima
  float2* rope = nullptr;    // [rows][d/2] (cos, sin) at each row's position
  float2* rope_full = nullptr;  // [capacity][d/2] (cos, sin) of every position (own allocation)
  int rows_alloc = 0;        // activation rows allocated (>= every NB used)
  int nb_max = 16;
  float* ws = nullptr;       // [ws_sms][2][nb_max][128] partial GEMM tiles
  int ws_sms = 0;            // the model's SM budget when ws was sized
  float* qkv_part = nullptr;   // [qkv tiles][qkv_split][rows_alloc][128] split-K sums
  float* qkv_rinv = nullptr;   // [rows_alloc] 1 / rms of each row at the QKV projection
  int qkv_split = 1;
  int* counters = nullptr;   // [max tiles] stream-K arrival counters
  int n_counters = 0;
  float* ss = nullptr;       // [hidden / 128][rows_alloc] partial sums of h^2
  // attention (k_attn.cu): per (request, kv head, 64-query tile)
  uint8_t* qimg = nullptr;   // query operand images, attn_qimg_bytes(d) each
  int attn_qt = 0;           // query tiles of the widest request
  int attn_chunks = 0;       // 1024-key chunks of the capacity
  float* attn_o = nullptr;   // [batch][n_kv][qt][chunks][64][d] chunk partials
  float2* attn_ml = nullptr; // [batch][n_kv][qt][chunks][64] (max, sum) base 2
  int* attn_cnt = nullptr;   // [batch][n_kv][qt][8] chunks arrived per 8-row group; zero between launches
  int n_attn_cnt = 0;
  // TMA descriptors of the activation operands, per token-row padding
  CUtensorMap tm_xn[kNbCount], tm_ao[kNbCount], tm_u[kNbCount];
  // TMA descriptors of the caches: [n_layers * batch * n_kv][capacity][d]
  CUtensorMap tm_kc, tm_vc;
  // limit of the kernels' pipeline waits (as2d_kv_set_wait_limit)
  unsigned long long wait_ns = 2000000000ull;
  // measurement support
  int prof_class = -1;
  std::vector<cudaEvent_t> prof_events;  // pairs
  int prof_used = 0;                     // pairs recorded since the last read
  int64_t launches = 0;                  // kernels launched since the last read
  // staging of as2d_verify_from_buffers (cand_buffer.cu), allocated on first use:
  // candidates [batch][kMaxK], then n_accepted [batch] and correction [batch]
  int32_t* cb_dev = nullptr;
  int32_t* cb_host = nullptr;            // pinned, same layout
  int32_t* pf_out = nullptr;             // [2] n_accepted, root of as2d_prefill chunks
  // as2d_prefill's working state (batch 1, kPrefillRows rows per pass), made
  // on first use; shares this state's cache, lengths, roots, error flags and
  // rotary table
  KvState* pf = nullptr;
};

// Error reporting shared by the translation units of the C-ABI: records the
// thread-local message returned by as2d_last_error and passes `st` through.
as2d_status report_error(as2d_status st, const std::string& msg);
void clear_error();

// Launchers (k_basic.cu).  All enqueue on `st` and return cudaGetLastError().
cudaError_t launch_embed(const RowMap& m, const Model& md, KvState& kv,
                         const int32_t* cand, cudaStream_t st,
                         const int32_t* root_override = nullptr);
cudaError_t launch_accept(const RowMap& m, const Model& md, KvState& kv,
                          const int32_t* cand, const as2d_verify_out& out,
                          cudaStream_t st, bool force = false);
cudaError_t launch_rollback(KvState& kv, const int32_t* new_len,
                            const int32_t* new_root, cudaStream_t st);
// Fills kv.rope_full for positions [0, capacity).
cudaError_t launch_rope_table(const Model& md, KvState& kv, cudaStream_t st);
// Load-time weight re-layout (k_pack.cu).
size_t packed_elems(int n_rows, int K);
cudaError_t pack_weights(bf16* dst, int n_rows, int K, const void* const* segs,
                         const int* seg_rows, int nseg, bool interleave, cudaStream_t st);

// Attention on the tensor cores (k_attn.cu): query tiles of a request of
// `rows` rows, 1024-key chunks of a capacity, bytes of one query image.
int attn_q_tiles(int rows_per_request, int group);
int attn_chunks(int capacity);
size_t attn_qimg_bytes(int head_dim);
// The cache [n_layers][batch][n_kv][capacity][head_dim] bf16 as the 3D tensor
// map the attention kernel loads key/value tiles through.
bool encode_cache_map(CUtensorMap* map, const void* cache, int head_dim, int capacity,
                      int64_t heads);
cudaError_t launch_attention_split(const RowMap& m, const Model& md, KvState& kv, int layer,
                                   cudaStream_t st);

// Tensor-core GEMM launchers (k_tc_*.cu), one per fused epilogue.
int qkv_split_for(const Model& m);
cudaError_t tc_gemm_part(int nb, const CUtensorMap& x, const TcParams& p, cudaStream_t st);
cudaError_t tc_gemm_resid(int nb, const CUtensorMap& x, const TcParams& p,
                          cudaStream_t st);
cudaError_t tc_gemm_swiglu(int nb, const CUtensorMap& x, const TcParams& p,
                           cudaStream_t st);
cudaError_t tc_gemm_logits(int nb, const CUtensorMap& x, const TcParams& p,
                           cudaStream_t st);

cudaError_t launch_f32_from_bf16(float* dst, const void* src, int64_t n,
                                 cudaStream_t st);

}  // namespace as2d

// Handle types of the C-ABI.
struct as2d_model {
  as2d::Model m;
};
struct as2d_kv {
  as2d::KvState s;
};
