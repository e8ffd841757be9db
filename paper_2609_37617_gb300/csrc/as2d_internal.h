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

// Device error bits (ORed into KvState::d_err).
enum : int32_t {
  kErrBadToken = 1,
  kErrRollback = 2,
  kErrTimeout = 4,
};

struct Model {
  as2d_config cfg;
  int qkv_rows;      // (n_q + 2 n_kv) * head_dim
  int q_dim;         // n_q * head_dim
  int kv_dim;        // n_kv * head_dim
  int sm_count;
  void* arena = nullptr;  // every weight below lives here
  size_t arena_bytes = 0;
  const bf16* embed = nullptr;    // [V][H]
  const bf16* lm_head = nullptr;  // [V][H]
  const float* final_norm = nullptr;
  std::vector<const bf16*> w_qkv;   // [(nq + 2 nkv) d][H]: q rows, k rows, v rows
  std::vector<const bf16*> w_o;     // [H][nq d]
  std::vector<const bf16*> w_gu;    // [2F][H]: blocks of 64 gate rows, 64 up rows
  std::vector<const bf16*> w_down;  // [H][F]
  std::vector<const float*> attn_norm, mlp_norm;  // fp32 gains [H]
};

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
  // working memory, sized for batch * (kMaxK + 1) rows
  int max_rows = 0;
  void* work = nullptr;
  size_t work_bytes = 0;
  float* h = nullptr;        // [rows][H] residual stream, fp32
  bf16* xn = nullptr;        // [rows][H] normalised activations
  float* qkv = nullptr;      // [rows][qkv_rows]
  float* q = nullptr;        // [rows][nq][d] rotated queries
  bf16* ao = nullptr;        // [rows][nq d] attention output
  bf16* u = nullptr;         // [rows][F] SwiGLU output
  unsigned long long* best = nullptr;  // [rows] packed (logit, index) maxima
  // measurement support
  int prof_class = -1;
  std::vector<cudaEvent_t> prof_events;  // pairs
  int prof_used = 0;                     // pairs recorded since the last read
  int64_t launches = 0;                  // kernels launched since the last read
};

// Launchers (k_basic.cu).  All enqueue on `st` and return cudaGetLastError().
cudaError_t launch_embed(const RowMap& m, const Model& md, KvState& kv,
                         const int32_t* cand, cudaStream_t st);
cudaError_t launch_rmsnorm(const RowMap& m, const Model& md, KvState& kv,
                           const float* gain, cudaStream_t st);
cudaError_t launch_gemv_qkv(const RowMap& m, const Model& md, KvState& kv,
                            int layer, cudaStream_t st);
cudaError_t launch_rope_append(const RowMap& m, const Model& md, KvState& kv,
                               int layer, cudaStream_t st);
cudaError_t launch_attention(const RowMap& m, const Model& md, KvState& kv,
                             int layer, cudaStream_t st);
cudaError_t launch_gemv_o(const RowMap& m, const Model& md, KvState& kv,
                          int layer, cudaStream_t st);
cudaError_t launch_gemv_gate_up(const RowMap& m, const Model& md, KvState& kv,
                                int layer, cudaStream_t st);
cudaError_t launch_gemv_down(const RowMap& m, const Model& md, KvState& kv,
                             int layer, cudaStream_t st);
cudaError_t launch_lm_head(const RowMap& m, const Model& md, KvState& kv,
                           float* logits, cudaStream_t st);
cudaError_t launch_accept(const RowMap& m, const Model& md, KvState& kv,
                          const int32_t* cand, const as2d_verify_out& out,
                          cudaStream_t st);
cudaError_t launch_rollback(KvState& kv, const int32_t* new_len,
                            const int32_t* new_root, cudaStream_t st);
cudaError_t launch_f32_from_bf16(float* dst, const void* src, int64_t n,
                                 cudaStream_t st);

}  // namespace as2d
