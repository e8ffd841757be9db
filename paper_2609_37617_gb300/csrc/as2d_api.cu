// as2d_api.cu -- the C-ABI of include/as2d.h: argument checking, ownership,
// weight re-layout at load time, and the per-call launch sequence of the
// verification pass (Section 3.2; App. C.2).
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <string>

#include "as2d_internal.h"

using namespace as2d;

namespace {

thread_local std::string g_err;

as2d_status fail(as2d_status st, const std::string& msg) {
  g_err = msg;
  return st;
}

#define CUDA_TRY(expr)                                                      \
  do {                                                                      \
    cudaError_t e_ = (expr);                                                \
    if (e_ != cudaSuccess)                                                  \
      return fail(AS2D_ERR_CUDA, std::string(#expr) + ": " +                \
                                     cudaGetErrorString(e_));               \
  } while (0)

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Carves consecutive 256-byte-aligned pieces out of one allocation.
struct Carver {
  char* base;
  size_t off = 0;
  template <typename T>
  T* take(size_t count) {
    off = align_up(off, 256);
    T* p = reinterpret_cast<T*>(base + off);
    off += count * sizeof(T);
    return p;
  }
};

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static const EncodeTiledFn fn = [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      return (EncodeTiledFn)ptr;
    return (EncodeTiledFn) nullptr;
  }();
  return fn;
}

// Row-major bf16 matrix [outer][inner] viewed by TMA in boxes of
// box_inner x box_outer elements with 128-byte swizzling.
bool encode_2d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t outer,
               uint32_t box_inner, uint32_t box_outer) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {inner * 2};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

bool as2d::encode_cache_map(CUtensorMap* map, const void* cache, int head_dim, int capacity,
                            int64_t heads) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[3] = {(cuuint64_t)head_dim, (cuuint64_t)capacity, (cuuint64_t)heads};
  cuuint64_t strides[2] = {(cuuint64_t)head_dim * 2, (cuuint64_t)capacity * head_dim * 2};
  cuuint32_t box[3] = {64, 128, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(cache), dims, strides,
            box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

namespace {

as2d_status check_config(const as2d_config* c) {
  if (!c) return fail(AS2D_ERR_INVALID_ARG, "config is NULL");
  if (c->n_layers <= 0 || c->hidden <= 0 || c->n_q_heads <= 0 ||
      c->n_kv_heads <= 0 || c->head_dim <= 0 || c->ffn <= 0 || c->vocab <= 1)
    return fail(AS2D_ERR_INVALID_ARG, "config sizes must be positive");
  if (!(c->rope_theta > 0.f) || !(c->rms_eps >= 0.f))
    return fail(AS2D_ERR_INVALID_ARG, "rope_theta must be > 0 and rms_eps >= 0");
  if (c->n_q_heads % c->n_kv_heads != 0)
    return fail(AS2D_ERR_INVALID_ARG, "n_q_heads must be a multiple of n_kv_heads");
  if (c->head_dim != 64 && c->head_dim != 128)
    return fail(AS2D_ERR_UNSUPPORTED, "head_dim must be 64 or 128");
  if (c->hidden % 128 != 0 || (c->n_q_heads * c->head_dim) % 128 != 0 ||
      (c->n_kv_heads * c->head_dim) % 128 != 0)
    return fail(AS2D_ERR_UNSUPPORTED,
                "hidden, n_q*head_dim and n_kv*head_dim must be multiples of 128");
  if (c->ffn % 64 != 0) return fail(AS2D_ERR_UNSUPPORTED, "ffn must be a multiple of 64");
  if (c->vocab % 8 != 0) return fail(AS2D_ERR_UNSUPPORTED, "vocab must be a multiple of 8");
  return AS2D_OK;
}

}  // namespace

as2d_status as2d::report_error(as2d_status st, const std::string& msg) { return fail(st, msg); }
void as2d::clear_error() { g_err.clear(); }

extern "C" const char* as2d_last_error(void) { return g_err.c_str(); }

extern "C" as2d_status as2d_model_load(const as2d_config* cfg,
                                       const as2d_weights* w,
                                       as2d_model** out) {
  g_err.clear();
  as2d_status st = check_config(cfg);
  if (st != AS2D_OK) return st;
  if (!w || !out) return fail(AS2D_ERR_INVALID_ARG, "weights or out is NULL");
  if (!w->embed || !w->final_norm || !w->lm_head || !w->attn_norm || !w->w_q ||
      !w->w_k || !w->w_v || !w->w_o || !w->mlp_norm || !w->w_gate ||
      !w->w_up || !w->w_down)
    return fail(AS2D_ERR_INVALID_ARG, "a weight pointer is NULL");
  const int L = cfg->n_layers;
  for (int l = 0; l < L; ++l)
    if (!w->attn_norm[l] || !w->w_q[l] || !w->w_k[l] || !w->w_v[l] ||
        !w->w_o[l] || !w->mlp_norm[l] || !w->w_gate[l] || !w->w_up[l] ||
        !w->w_down[l])
      return fail(AS2D_ERR_INVALID_ARG, "a per-layer weight pointer is NULL");

  as2d_model* mh = new as2d_model();
  Model& m = mh->m;
  m.cfg = *cfg;
  const size_t H = cfg->hidden, F = cfg->ffn, V = cfg->vocab, d = cfg->head_dim;
  m.q_dim = cfg->n_q_heads * cfg->head_dim;
  m.kv_dim = cfg->n_kv_heads * cfg->head_dim;
  m.qkv_rows = m.q_dim + 2 * m.kv_dim;
  int dev = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&m.sm_count, cudaDevAttrMultiProcessorCount, dev);
  m.device_sm_count = m.sm_count;
  (void)d;

  const size_t qkv_packed = packed_elems(m.qkv_rows, (int)H);
  const size_t o_packed = packed_elems((int)H, m.q_dim);
  const size_t gu_packed = packed_elems((int)(2 * F), (int)H);
  const size_t down_packed = packed_elems((int)H, (int)F);
  const size_t lm_packed = packed_elems((int)V, (int)H);
  size_t bytes = align_up(V * H * 2, 256) + align_up(lm_packed * 2, 256);
  bytes += L * (align_up(qkv_packed * 2, 256) + align_up(o_packed * 2, 256) +
                align_up(gu_packed * 2, 256) + align_up(down_packed * 2, 256) +
                2 * align_up(H * 4, 256));
  bytes += align_up(H * 4, 256) + 4096;
  cudaError_t e = cudaMalloc(&m.arena, bytes);
  if (e != cudaSuccess) {
    delete mh;
    return fail(AS2D_ERR_CUDA, std::string("cudaMalloc of the weight arena: ") + cudaGetErrorString(e));
  }
  m.arena_bytes = bytes;
  Carver cv{(char*)m.arena};
  auto fail_free = [&](const std::string& msg) {
    cudaFree(m.arena);
    delete mh;
    return fail(AS2D_ERR_CUDA, msg);
  };
#define LOAD_TRY(expr)                                                        \
  do {                                                                        \
    cudaError_t e_ = (expr);                                                  \
    if (e_ != cudaSuccess)                                                    \
      return fail_free(std::string(#expr) + ": " + cudaGetErrorString(e_));   \
  } while (0)

  bf16* embed = cv.take<bf16>(V * H);
  bf16* lm = cv.take<bf16>(lm_packed);
  float* fnorm = cv.take<float>(H);
  LOAD_TRY(cudaMemcpy(embed, w->embed, V * H * 2, cudaMemcpyDeviceToDevice));
  {
    const void* segs[1] = {w->lm_head};
    const int rows[1] = {(int)V};
    LOAD_TRY(pack_weights(lm, (int)V, (int)H, segs, rows, 1, false, 0));
  }
  LOAD_TRY(launch_f32_from_bf16(fnorm, w->final_norm, H, 0));
  m.embed = embed;
  m.lm_head = lm;
  m.final_norm = fnorm;
  for (int l = 0; l < L; ++l) {
    bf16* qkv = cv.take<bf16>(qkv_packed);
    bf16* wo = cv.take<bf16>(o_packed);
    bf16* gu = cv.take<bf16>(gu_packed);
    bf16* wd = cv.take<bf16>(down_packed);
    float* an = cv.take<float>(H);
    float* mn = cv.take<float>(H);
    {
      const void* segs[3] = {w->w_q[l], w->w_k[l], w->w_v[l]};
      const int rows[3] = {m.q_dim, m.kv_dim, m.kv_dim};
      LOAD_TRY(pack_weights(qkv, m.qkv_rows, (int)H, segs, rows, 3, false, 0));
    }
    {
      const void* segs[1] = {w->w_o[l]};
      const int rows[1] = {(int)H};
      LOAD_TRY(pack_weights(wo, (int)H, m.q_dim, segs, rows, 1, false, 0));
    }
    {
      const void* segs[2] = {w->w_gate[l], w->w_up[l]};
      const int rows[2] = {(int)F, (int)F};
      LOAD_TRY(pack_weights(gu, (int)(2 * F), (int)H, segs, rows, 2, true, 0));
    }
    {
      const void* segs[1] = {w->w_down[l]};
      const int rows[1] = {(int)H};
      LOAD_TRY(pack_weights(wd, (int)H, (int)F, segs, rows, 1, false, 0));
    }
    LOAD_TRY(launch_f32_from_bf16(an, w->attn_norm[l], H, 0));
    LOAD_TRY(launch_f32_from_bf16(mn, w->mlp_norm[l], H, 0));
    m.w_qkv.push_back(qkv);
    m.w_o.push_back(wo);
    m.w_gu.push_back(gu);
    m.w_down.push_back(wd);
    m.attn_norm.push_back(an);
    m.mlp_norm.push_back(mn);
  }
  LOAD_TRY(cudaDeviceSynchronize());
#undef LOAD_TRY
  *out = mh;
  return AS2D_OK;
}

extern "C" as2d_status as2d_model_set_sm_budget(as2d_model* mh, int32_t n_sms) {
  g_err.clear();
  if (!mh) return fail(AS2D_ERR_INVALID_ARG, "model is NULL");
  if (n_sms < 1 || n_sms > mh->m.device_sm_count)
    return fail(AS2D_ERR_INVALID_ARG, "n_sms must be in [1, the device's SM count]");
  mh->m.sm_count = n_sms;
  return AS2D_OK;
}

extern "C" void as2d_model_free(as2d_model* mh) {
  if (!mh) return;
  cudaFree(mh->m.arena);
  delete mh;
}

namespace {

// Sizes, allocates and carves the working memory of a state of `batch`
// requests with up to `rows_per_request` rows each, and encodes the
// activation descriptors.  Leaves s.work null on failure.
as2d_status alloc_work(KvState& s, const Model& m, int batch, int capacity,
                       int rows_per_request) {
  s.max_k = rows_per_request - 1;
  s.max_rows = batch * rows_per_request;
  s.nb_max = nb_for_rows(s.max_rows);
  s.rows_alloc = s.max_rows > s.nb_max ? s.max_rows : s.nb_max;
  const size_t R = s.rows_alloc, H = m.cfg.hidden, F = m.cfg.ffn;
  const size_t max_tiles = ((size_t)(m.cfg.vocab > 2 * F ? m.cfg.vocab : 2 * F) + 127) / 128 + 64;
  size_t bytes = 4096 + 3 * align_up((size_t)(batch + 1) * 4, 256);
  bytes += align_up(R * H * 4, 256) + align_up(2 * R * H * 2, 256) +
           align_up(2 * R * m.q_dim * 2, 256) + align_up(2 * R * F * 2, 256) + align_up(R * 8, 256) +
           align_up(R * (m.cfg.head_dim / 2) * 8, 256) + align_up(R * (H / 128) * 4, 256) +
           align_up((size_t)m.sm_count * 2 * s.nb_max * 128 * 4, 256) + align_up(max_tiles * 4, 256);
  s.qkv_split = qkv_split_for(m);
  const size_t qkv_tiles = (size_t)(m.qkv_rows + 127) / 128;
  bytes += align_up(qkv_tiles * s.qkv_split * R * 128 * 4, 256) + align_up(R * 4, 256);
  const int group = m.cfg.n_q_heads / m.cfg.n_kv_heads;
  s.attn_qt = attn_q_tiles(rows_per_request, group);
  s.attn_chunks = attn_chunks(capacity);
  const size_t attn_items = (size_t)batch * m.cfg.n_kv_heads * s.attn_qt;
  const size_t attn_rows = attn_items * s.attn_chunks * 64;
  bytes += align_up(attn_items * attn_qimg_bytes(m.cfg.head_dim), 256) +
           align_up(attn_rows * m.cfg.head_dim * 4, 256) + align_up(attn_rows * 8, 256) +
           align_up(attn_items * 8 * 4, 256);
  cudaError_t e = cudaMalloc(&s.work, bytes);
  if (e != cudaSuccess) {
    s.work = nullptr;
    return fail(AS2D_ERR_CUDA, std::string("cudaMalloc of the working memory: ") + cudaGetErrorString(e));
  }
  s.work_bytes = bytes;
  Carver cv{(char*)s.work};
  s.d_len = cv.take<int32_t>(batch);
  s.d_root = cv.take<int32_t>(batch);
  s.d_err = cv.take<int32_t>(batch + 1);
  s.h = cv.take<float>(R * H);
  s.xn = cv.take<bf16>(2 * R * H);
  s.ao = cv.take<bf16>(2 * R * m.q_dim);
  s.u = cv.take<bf16>(2 * R * F);
  s.best = cv.take<unsigned long long>(R);
  s.rope = cv.take<float2>(R * (m.cfg.head_dim / 2));
  s.ss = cv.take<float>(R * (H / 128));
  s.ws = cv.take<float>((size_t)m.sm_count * 2 * s.nb_max * 128);
  s.ws_sms = m.sm_count;
  s.counters = cv.take<int>(max_tiles);
  s.n_counters = (int)max_tiles;
  s.qkv_part = cv.take<float>(qkv_tiles * s.qkv_split * R * 128);
  s.qkv_rinv = cv.take<float>(R);
  s.qimg = cv.take<uint8_t>(attn_items * attn_qimg_bytes(m.cfg.head_dim));
  s.attn_o = cv.take<float>(attn_rows * m.cfg.head_dim);
  s.attn_ml = cv.take<float2>(attn_rows);
  s.attn_cnt = cv.take<int>(attn_items * 8);
  s.n_attn_cnt = (int)attn_items * 8;
  bool ok = encode_cache_map(&s.tm_kc, s.k_cache, m.cfg.head_dim, capacity,
                             (int64_t)m.cfg.n_layers * batch * m.cfg.n_kv_heads) &&
            encode_cache_map(&s.tm_vc, s.v_cache, m.cfg.head_dim, capacity,
                             (int64_t)m.cfg.n_layers * batch * m.cfg.n_kv_heads);
  for (int i = 0; i < kNbCount && ok; ++i) {
    const int nb = kNbSet[i];
    if (nb > s.nb_max) break;
    ok = encode_2d(&s.tm_xn[i], s.xn, H, 2 * R, 64, nb) &&
         encode_2d(&s.tm_ao[i], s.ao, m.q_dim, 2 * R, 64, nb) &&
         encode_2d(&s.tm_u[i], s.u, F, 2 * R, 64, nb);
  }
  if (!ok) {
    cudaFree(s.work);
    s.work = nullptr;
    return fail(AS2D_ERR_CUDA, "cuTensorMapEncodeTiled failed for an activation buffer or a cache");
  }
  return AS2D_OK;
}

}  // namespace

extern "C" as2d_status as2d_kv_init_prefilled(as2d_model* mh, int32_t batch,
                                              const int32_t* kv_len,
                                              int32_t capacity, void* k_cache,
                                              void* v_cache,
                                              const int32_t* root_tokens,
                                              as2d_kv** out) {
  g_err.clear();
  if (!mh || !kv_len || !k_cache || !v_cache || !root_tokens || !out)
    return fail(AS2D_ERR_INVALID_ARG, "a pointer argument is NULL");
  if (batch < 1 || batch > kMaxBatch)
    return fail(AS2D_ERR_INVALID_ARG, "batch must be in [1, AS2D_MAX_BATCH]");
  if (capacity < 1) return fail(AS2D_ERR_INVALID_ARG, "capacity must be positive");
  if (capacity > 65536)
    return fail(AS2D_ERR_UNSUPPORTED, "capacity above 65536 positions is not supported");
  const Model& m = mh->m;
  for (int b = 0; b < batch; ++b) {
    if (kv_len[b] < 0 || kv_len[b] >= capacity)
      return fail(AS2D_ERR_CAPACITY, "kv_len must be in [0, capacity)");
    if (root_tokens[b] < 0 || root_tokens[b] >= m.cfg.vocab)
      return fail(AS2D_ERR_INVALID_ARG, "root token outside [0, vocab)");
  }
  as2d_kv* kh = new as2d_kv();
  KvState& s = kh->s;
  s.model = &mh->m;
  s.batch = batch;
  s.capacity = capacity;
  s.k_cache = (bf16*)k_cache;
  s.v_cache = (bf16*)v_cache;
  s.len_upper.assign(kv_len, kv_len + batch);
  {
    const as2d_status rc = alloc_work(s, m, batch, capacity, kMaxK + 1);
    if (rc != AS2D_OK) {
      delete kh;
      return rc;
    }
  }
  cudaError_t e;
  const size_t bytes = s.work_bytes;
  e = cudaMemset(s.work, 0, bytes);
  if (e == cudaSuccess)
    e = cudaMalloc(&s.rope_full, (size_t)capacity * (m.cfg.head_dim / 2) * sizeof(float2));
  if (e == cudaSuccess) e = launch_rope_table(m, s, 0);
  if (e == cudaSuccess) e = cudaMemcpy(s.d_len, kv_len, batch * 4, cudaMemcpyHostToDevice);
  if (e == cudaSuccess) e = cudaMemcpy(s.d_root, root_tokens, batch * 4, cudaMemcpyHostToDevice);
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  if (e != cudaSuccess) {
    cudaFree(s.rope_full);
    cudaFree(s.work);
    delete kh;
    return fail(AS2D_ERR_CUDA, std::string("initialising the state: ") + cudaGetErrorString(e));
  }
  *out = kh;
  return AS2D_OK;
}

extern "C" void as2d_kv_free(as2d_kv* kh) {
  if (!kh) return;
  for (cudaEvent_t e : kh->s.prof_events) cudaEventDestroy(e);
  cudaFree(kh->s.work);
  cudaFree(kh->s.rope_full);
  cudaFree(kh->s.cb_dev);
  cudaFree(kh->s.pf_out);
  if (kh->s.pf) {
    // the prefill state's lengths, roots, flags and rotary table are this state's
    cudaFree(kh->s.pf->work);
    delete kh->s.pf;
  }
  cudaFreeHost(kh->s.cb_host);
  delete kh;
}

namespace {

// Event pair around the launches of one kernel class in one layer, recorded
// only while that class is being profiled.
struct ProfScope {
  KvState& s;
  cudaStream_t st;
  bool on;
  int idx = -1;
  ProfScope(KvState& s_, int cls, cudaStream_t st_) : s(s_), st(st_), on(s_.prof_class == cls) {
    if (!on) return;
    if ((size_t)(2 * s.prof_used + 2) > s.prof_events.size()) {
      for (int i = 0; i < 64; ++i) {
        cudaEvent_t e;
        if (cudaEventCreate(&e) != cudaSuccess) { on = false; return; }
        s.prof_events.push_back(e);
      }
    }
    idx = s.prof_used++;
    cudaEventRecord(s.prof_events[2 * idx], st);
  }
  ~ProfScope() {
    if (on && idx >= 0) cudaEventRecord(s.prof_events[2 * idx + 1], st);
  }
};

#define LAUNCH(cls, expr)                        \
  do {                                           \
    ProfScope ps_(s, cls, st);                   \
    CUDA_TRY(expr);                              \
  } while (0)

// One projection on the tensor cores: row chunks of at most 256 token rows.
}  // namespace

// CTAs per tile of the QKV projection's K split: as many as fill the SMs
// (at most 8 and at most one per 64-column block).  Depends on the model and
// the device only.
int as2d::qkv_split_for(const Model& m) {
  const int tiles = (m.qkv_rows + 127) / 128, kb = m.cfg.hidden / 64;
  int s = m.sm_count / tiles;
  if (s > 8) s = 8;
  if (s > kb) s = kb;
  return s < 1 ? 1 : s;
}

namespace {

cudaError_t tc_project(int epi, const Model& m, KvState& s, const RowMap& rm, const bf16* w,
                       const CUtensorMap* xmaps, int N, int K, TcParams p, cudaStream_t st) {
  p.w = w;
  p.N = N;
  p.K = K;
  p.n_tiles = (N + 127) / 128;
  p.kb = (K + 63) / 64;
  p.units = (long long)p.n_tiles * p.kb;
  // Work split (all of it a function of N, K and the device only, so a
  // row's sums are added in the same order whatever the number of rows):
  //   QKV (TC_PART): K split evenly over qkv_split CTAs per tile, sums
  //     finished by qkv_finish_kernel;
  //   at least 90% as many tiles as SMs (gate/up): whole tiles per CTA,
  //     as evenly as they go, each finished by its own CTA;
  //   otherwise stream-K over one CTA per SM, with at least four units per
  //     CTA for the residual projections (a small projection spread over
  //     every SM cuts each tile into many parts, and its CTAs on SMs still
  //     held by the attention start late); residual projections leave their
  //     split tiles to tc_resid_finish_kernel, the LM head finishes them in
  //     the GEMM (last CTA of a tile).
  p.grid = (int)(p.units < m.sm_count ? p.units : m.sm_count);
  if (epi == TC_RESID && p.units / 4 < p.grid) p.grid = p.units >= 4 ? (int)(p.units / 4) : 1;
  p.split = 0;
  p.defer = epi == TC_RESID ? 1 : 0;
  if (epi == TC_SWIGLU && p.n_tiles * 10 >= m.sm_count * 9) {
    const int per = (p.n_tiles + m.sm_count - 1) / m.sm_count;
    p.split = 1;
    p.grid = (p.n_tiles + per - 1) / per;
    p.defer = 0;
  }
  if (epi == TC_PART) {
    p.split = s.qkv_split;
    p.grid = p.n_tiles * p.split;
    p.part = s.qkv_part;
    p.part_rinv = s.qkv_rinv;
    p.part_ld = s.rows_alloc;
  }
  p.ws = s.ws;
  p.counters = s.counters;
  p.err = s.d_err;
  p.timeout_ns = s.wait_ns;
  p.rm = rm;
  for (int row0 = 0; row0 < rm.rows; row0 += 256) {
    p.row0 = row0;
    p.rows = rm.rows - row0 < 256 ? rm.rows - row0 : 256;
    const int nb = nb_for_rows(p.rows);
    const CUtensorMap& x = xmaps[nb_index(nb)];
    cudaError_t e;
    switch (epi) {
      case TC_PART: e = tc_gemm_part(nb, x, p, st); break;
      case TC_RESID: e = tc_gemm_resid(nb, x, p, st); break;
      case TC_SWIGLU: e = tc_gemm_swiglu(nb, x, p, st); break;
      default: e = tc_gemm_logits(nb, x, p, st); break;
    }
    if (e != cudaSuccess) return e;
    s.launches += (p.defer && p.grid >= 2) ? 2 : 1;
  }
  return cudaSuccess;
}

// One verification pass.  force: keep every row whatever the greedy tokens
// (prefill); root_override: device int32 [batch], the tokens forwarded in
// place of the pending roots.
as2d_status run_block(KvState& s, const int32_t* cand, const int32_t* k,
                      const as2d_verify_out* out, cudaStream_t st, bool force = false,
                      const int32_t* root_override = nullptr) {
  if (!out || !out->n_accepted || !out->correction_token)
    return fail(AS2D_ERR_INVALID_ARG, "out, out->n_accepted and out->correction_token are required");
  RowMap rm;
  rm.batch = s.batch;
  rm.start[0] = 0;
  int total_k = 0;
  for (int b = 0; b < s.batch; ++b) {
    const int kb = k ? k[b] : 0;
    if (kb < 0 || kb > s.max_k)
      return fail(AS2D_ERR_INVALID_ARG, "k must be in [0, AS2D_MAX_K]");
    if (s.len_upper[b] + kb + 1 > s.capacity)
      return fail(AS2D_ERR_CAPACITY, "length bound + k + 1 exceeds the cache capacity");
    rm.start[b + 1] = rm.start[b] + kb + 1;
    total_k += kb;
  }
  rm.rows = rm.start[s.batch];
  if (total_k > 0 && !cand) return fail(AS2D_ERR_INVALID_ARG, "candidates is NULL");
  const Model& m = *s.model;
  if (m.sm_count > s.ws_sms)
    return fail(AS2D_ERR_INVALID_ARG, "the model's SM budget grew after this state was created");
  const as2d_config& c = m.cfg;

  // One pass of the verification step (Section 3.2; App. C.2): embedding
  // gather, n_layers x {QKV (split-K sums), RoPE + KV append + attention, O + residual,
  // gate/up + SwiGLU, down + residual}, LM head + argmax, accept scan, as a
  // sequence of kernels chained by programmatic dependent launch.
  LAUNCH(AS2D_KERNEL_OTHER, launch_embed(rm, m, s, cand, st, root_override));
  TcParams tp{};
  tp.h = s.h;
  tp.u = s.u;
  tp.logits = out->logits;
  tp.best = s.best;
  tp.xn = s.xn;
  tp.ss = s.ss;
  tp.ss_ld = s.rows_alloc;
  tp.lo_row = s.rows_alloc;
  tp.n_htiles = c.hidden / 128;
  tp.eps = c.rms_eps;
  tp.hidden = c.hidden;
  const int H = c.hidden, F = c.ffn;
  for (int l = 0; l < c.n_layers; ++l) {
    LAUNCH(AS2D_KERNEL_QKV, tc_project(TC_PART, m, s, rm, m.w_qkv[l], s.tm_xn, m.qkv_rows, H, tp, st));
    LAUNCH(AS2D_KERNEL_ATTENTION, launch_attention_split(rm, m, s, l, st));
    tp.g_next = m.mlp_norm[l];
    LAUNCH(AS2D_KERNEL_O, tc_project(TC_RESID, m, s, rm, m.w_o[l], s.tm_ao, H, m.q_dim, tp, st));
    LAUNCH(AS2D_KERNEL_GATE_UP, tc_project(TC_SWIGLU, m, s, rm, m.w_gu[l], s.tm_xn, 2 * F, H, tp, st));
    tp.g_next = (l + 1 < c.n_layers) ? m.attn_norm[l + 1] : m.final_norm;
    LAUNCH(AS2D_KERNEL_DOWN, tc_project(TC_RESID, m, s, rm, m.w_down[l], s.tm_u, H, F, tp, st));
  }
  LAUNCH(AS2D_KERNEL_LM_HEAD, tc_project(TC_LOGITS, m, s, rm, m.lm_head, s.tm_xn, c.vocab, H, tp, st));
  LAUNCH(AS2D_KERNEL_OTHER, launch_accept(rm, m, s, cand, *out, st, force));
  for (int b = 0; b < s.batch; ++b) s.len_upper[b] += (k ? k[b] : 0) + 1;
  return AS2D_OK;
}

}  // namespace

extern "C" as2d_status as2d_prefill(as2d_kv* kh, const int32_t* tokens, int32_t n,
                                    int32_t* first_token, void* stream) {
  g_err.clear();
  if (!kh || !tokens || n < 1) return fail(AS2D_ERR_INVALID_ARG, "kv, tokens and n >= 1 are required");
  KvState& s = kh->s;
  if (s.batch != 1) return fail(AS2D_ERR_UNSUPPORTED, "prefill runs batch-1 states");
  if (s.len_upper[0] + n > s.capacity)
    return fail(AS2D_ERR_CAPACITY, "length bound + n exceeds the cache capacity");
  if (!s.pf_out) {
    const cudaError_t e = cudaMalloc(&s.pf_out, 2 * sizeof(int32_t));
    if (e != cudaSuccess) {
      s.pf_out = nullptr;
      return fail(AS2D_ERR_CUDA, std::string("cudaMalloc: ") + cudaGetErrorString(e));
    }
  }
  if (!s.pf) {
    // a working state for passes of kPrefillRows rows over this state's cache
    KvState* a = new KvState();
    a->model = s.model;
    a->batch = 1;
    a->capacity = s.capacity;
    a->k_cache = s.k_cache;
    a->v_cache = s.v_cache;
    a->len_upper = s.len_upper;
    as2d_status rc = alloc_work(*a, *s.model, 1, s.capacity, kPrefillRows);
    if (rc == AS2D_OK) {
      const cudaError_t e = cudaMemset(a->work, 0, a->work_bytes);
      if (e != cudaSuccess) {
        cudaFree(a->work);
        rc = fail(AS2D_ERR_CUDA, std::string("cudaMemset: ") + cudaGetErrorString(e));
      }
    }
    if (rc != AS2D_OK) {
      delete a;
      return rc;
    }
    a->d_len = s.d_len;
    a->d_root = s.d_root;
    a->d_err = s.d_err;
    a->rope_full = s.rope_full;
    s.pf = a;
  }
  KvState& w = *s.pf;
  w.len_upper = s.len_upper;
  w.wait_ns = s.wait_ns;
  // passes of at most kPrefillRows tokens: the pass's first token stands in
  // for the pending root, the rest are kept as accepted candidates, and the
  // greedy token after the pass's last row becomes the root
  as2d_status rc = AS2D_OK;
  for (int s0 = 0; s0 < n && rc == AS2D_OK; s0 += kPrefillRows) {
    const int rows = (n - s0) < kPrefillRows ? (n - s0) : kPrefillRows;
    const int32_t k = rows - 1;
    const bool last = s0 + rows == n;
    const as2d_verify_out out{s.pf_out, (last && first_token) ? first_token : s.pf_out + 1,
                              nullptr, nullptr};
    rc = run_block(w, tokens + s0 + 1, &k, &out, (cudaStream_t)stream,
                   /*force=*/true, /*root_override=*/tokens + s0);
  }
  s.len_upper = w.len_upper;
  s.launches += w.launches;
  w.launches = 0;
  return rc;
}

extern "C" as2d_status as2d_verify_block(as2d_kv* kh, const int32_t* candidates,
                                         const int32_t* k,
                                         const as2d_verify_out* out,
                                         void* stream) {
  g_err.clear();
  if (!kh || !k) return fail(AS2D_ERR_INVALID_ARG, "kv and k are required");
  return run_block(kh->s, candidates, k, out, (cudaStream_t)stream);
}

extern "C" as2d_status as2d_decode_step(as2d_kv* kh, const as2d_verify_out* out,
                                        void* stream) {
  g_err.clear();
  if (!kh) return fail(AS2D_ERR_INVALID_ARG, "kv is NULL");
  return run_block(kh->s, nullptr, nullptr, out, (cudaStream_t)stream);
}

extern "C" as2d_status as2d_kv_rollback(as2d_kv* kh, const int32_t* new_len,
                                        const int32_t* new_root, void* stream) {
  g_err.clear();
  if (!kh || !new_len || !new_root)
    return fail(AS2D_ERR_INVALID_ARG, "kv, new_len and new_root are required");
  KvState& s = kh->s;
  for (int b = 0; b < s.batch; ++b) {
    if (new_len[b] < 0 || new_len[b] >= s.capacity)
      return fail(AS2D_ERR_INVALID_ARG, "new_len must be in [0, capacity)");
    if (new_root[b] < 0 || new_root[b] >= s.model->cfg.vocab)
      return fail(AS2D_ERR_INVALID_ARG, "new_root outside [0, vocab)");
  }
  CUDA_TRY(launch_rollback(s, new_len, new_root, (cudaStream_t)stream));
  for (int b = 0; b < s.batch; ++b) s.len_upper[b] = new_len[b];
  return AS2D_OK;
}

extern "C" as2d_status as2d_kv_read_state(as2d_kv* kh, int32_t* len,
                                          int32_t* root, void* stream) {
  g_err.clear();
  if (!kh) return fail(AS2D_ERR_INVALID_ARG, "kv is NULL");
  KvState& s = kh->s;
  CUDA_TRY(cudaStreamSynchronize((cudaStream_t)stream));
  int32_t tmp_len[kMaxBatch], tmp_root[kMaxBatch];
  CUDA_TRY(cudaMemcpy(tmp_len, s.d_len, s.batch * 4, cudaMemcpyDeviceToHost));
  CUDA_TRY(cudaMemcpy(tmp_root, s.d_root, s.batch * 4, cudaMemcpyDeviceToHost));
  for (int b = 0; b < s.batch; ++b) {
    s.len_upper[b] = tmp_len[b];
    if (len) len[b] = tmp_len[b];
    if (root) root[b] = tmp_root[b];
  }
  return AS2D_OK;
}

extern "C" as2d_status as2d_kv_device_state(as2d_kv* kh, const int32_t** len,
                                            const int32_t** root) {
  g_err.clear();
  if (!kh) return fail(AS2D_ERR_INVALID_ARG, "kv is NULL");
  if (len) *len = kh->s.d_len;
  if (root) *root = kh->s.d_root;
  return AS2D_OK;
}

extern "C" as2d_status as2d_kv_check(as2d_kv* kh, void* stream) {
  g_err.clear();
  if (!kh) return fail(AS2D_ERR_INVALID_ARG, "kv is NULL");
  CUDA_TRY(cudaStreamSynchronize((cudaStream_t)stream));
  int32_t err = 0;
  CUDA_TRY(cudaMemcpy(&err, kh->s.d_err, 4, cudaMemcpyDeviceToHost));
  if (err != 0) {
    int32_t zero = 0;
    CUDA_TRY(cudaMemcpy(kh->s.d_err, &zero, 4, cudaMemcpyHostToDevice));
    // a kernel that gave up may have left split-tile arrival counts behind
    if (kh->s.counters && kh->s.n_counters > 0)
      CUDA_TRY(cudaMemset(kh->s.counters, 0, (size_t)kh->s.n_counters * 4));
    if (kh->s.attn_cnt && kh->s.n_attn_cnt > 0)
      CUDA_TRY(cudaMemset(kh->s.attn_cnt, 0, (size_t)kh->s.n_attn_cnt * 4));
    std::string msg = "device error:";
    if (err & kErrBadToken) msg += " candidate or root token outside [0, vocab);";
    if (err & kErrRollback) msg += " rollback beyond the committed length;";
    if (err & kErrTimeout) msg += " a kernel wait timed out;";
    if (err & kErrCapacity) msg += " a device-side length left no room for the call's rows;";
    return fail(AS2D_ERR_DEVICE, msg);
  }
  return AS2D_OK;
}

extern "C" as2d_status as2d_kv_set_wait_limit(as2d_kv* kh, uint64_t ns) {
  g_err.clear();
  if (!kh) return fail(AS2D_ERR_INVALID_ARG, "kv is NULL");
  kh->s.wait_ns = ns;
  return AS2D_OK;
}

extern "C" as2d_status as2d_kv_profile(as2d_kv* kh, int32_t kernel_class) {
  g_err.clear();
  if (!kh) return fail(AS2D_ERR_INVALID_ARG, "kv is NULL");
  if (kernel_class < -1 || kernel_class >= AS2D_KERNEL_CLASSES)
    return fail(AS2D_ERR_INVALID_ARG, "kernel_class must be -1 or a class id");
  kh->s.prof_class = kernel_class;
  return AS2D_OK;
}

extern "C" as2d_status as2d_kv_profile_read(as2d_kv* kh, int32_t* launches,
                                            double* total_ms,
                                            int64_t* all_launches) {
  g_err.clear();
  if (!kh) return fail(AS2D_ERR_INVALID_ARG, "kv is NULL");
  KvState& s = kh->s;
  double tot = 0.0;
  for (int i = 0; i < s.prof_used; ++i) {
    CUDA_TRY(cudaEventSynchronize(s.prof_events[2 * i + 1]));
    float ms = 0.f;
    CUDA_TRY(cudaEventElapsedTime(&ms, s.prof_events[2 * i], s.prof_events[2 * i + 1]));
    tot += ms;
  }
  if (launches) *launches = s.prof_used;
  if (total_ms) *total_ms = tot;
  if (all_launches) *all_launches = s.launches;
  s.prof_used = 0;
  s.launches = 0;
  return AS2D_OK;
}

// ---- decode step with no allocation -------------------------------------------
//
// For callers that must not allocate device memory when they decode: for
// example a process whose device memory is handed out by another component
// under a fixed budget, or a real-time loop where the latency or the possible
// failure of an allocation is not acceptable.  The model is loaded once
// beforehand (that allocates, at set-up time); each call then keeps all of its
// working memory in one array compiled into this library, so it calls no
// allocator at all.

namespace {

constexpr int kStaticMaxHidden = 4096;
constexpr int kStaticMaxFfn = 20480;
constexpr int kStaticMaxQDim = 4096;     // n_q * head_dim
constexpr int kStaticMaxKvHeads = 8;
constexpr int kStaticMaxGroup = 16;      // n_q / n_kv
constexpr int kStaticMaxCapacity = 4096;
constexpr int kStaticMaxVocab = 262144;
constexpr int kStaticMaxSms = 192;
constexpr int kStaticRows = 16;          // one token row, padded to a TMA box
constexpr int kStaticChunks = kStaticMaxCapacity / 1024;  // attention chunks

constexpr size_t sa(size_t x) { return (x + 255) / 256 * 256; }
constexpr size_t kOffErr = 0;                                                     // err, bad, n
constexpr size_t kOffH = kOffErr + 256;
constexpr size_t kOffXn = kOffH + sa((size_t)kStaticRows * kStaticMaxHidden * 4);
// one query tile per kv head (a single row of at most 16 query heads per group)
constexpr size_t kOffQ = kOffXn + sa((size_t)2 * kStaticRows * kStaticMaxHidden * 2);
constexpr size_t kOffAo = kOffQ + sa((size_t)kStaticMaxKvHeads * 256 * 128);
constexpr size_t kOffU = kOffAo + sa((size_t)2 * kStaticRows * kStaticMaxQDim * 2);
constexpr size_t kOffBest = kOffU + sa((size_t)2 * kStaticRows * kStaticMaxFfn * 2);
constexpr size_t kOffRope = kOffBest + sa((size_t)kStaticRows * 8);
constexpr size_t kOffSs = kOffRope + sa((size_t)kStaticRows * 64 * 8);
constexpr size_t kOffWs = kOffSs + sa((size_t)(kStaticMaxHidden / 128) * kStaticRows * 4);
constexpr size_t kOffCnt = kOffWs + sa((size_t)kStaticMaxSms * 2 * 16 * 128 * 4);
constexpr size_t kOffAttnO = kOffCnt + sa((size_t)(kStaticMaxVocab / 128 + 64) * 4);
constexpr size_t kOffAttnMl =
    kOffAttnO + sa((size_t)kStaticMaxKvHeads * kStaticChunks * 64 * 128 * 4);
constexpr size_t kStaticMaxQkvTiles = (kStaticMaxQDim + 2 * kStaticMaxKvHeads * 128) / 128;
constexpr size_t kOffAttnCnt = kOffAttnMl + sa((size_t)kStaticMaxKvHeads * kStaticChunks * 64 * 8);
constexpr size_t kOffQkvPart = kOffAttnCnt + sa((size_t)kStaticMaxKvHeads * 8 * 4);
constexpr size_t kOffQkvRinv = kOffQkvPart + sa(kStaticMaxQkvTiles * 8 * kStaticRows * 128 * 4);
constexpr size_t kStaticScratchBytes = kOffQkvRinv + sa((size_t)kStaticRows * 4);

struct StaticDevice {
  bool ready = false;
  char* base = nullptr;
  CUtensorMap tm_xn, tm_ao, tm_u;
  int hidden = 0, q_dim = 0, ffn = 0;
};
constexpr int kStaticMaxDevices = 64;
StaticDevice g_static_dev[kStaticMaxDevices];

// Host-side descriptor of the scratch, built when the library is loaded so
// that no call has to allocate it.
KvState make_static_state() {
  KvState s;
  s.len_upper.assign(1, 0);
  return s;
}
KvState g_static_kv = make_static_state();
// Guards g_static_dev and g_static_kv: calls from several host threads are
// enqueued one at a time (their work on the GPU still shares one array).
std::mutex g_static_mu;

}  // namespace

// Working memory of as2d_decode_step_static, shared by every call on a device.
static __device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

extern "C" as2d_status as2d_decode_step_static(as2d_model* mh, void* k_cache, void* v_cache,
                                               int32_t capacity, int32_t* len, int32_t* root,
                                               int32_t* correction_token, float* logits,
                                               int32_t* error_bits, void* stream) {
  g_err.clear();
  if (!mh || !k_cache || !v_cache || !len || !root || !correction_token)
    return fail(AS2D_ERR_INVALID_ARG, "model, caches, len, root and correction_token are required");
  const Model& m = mh->m;
  const as2d_config& c = m.cfg;
  if (capacity < 1 || capacity > kStaticMaxCapacity)
    return fail(AS2D_ERR_CAPACITY, "as2d_decode_step_static supports capacity in [1, 4096]");
  if (c.hidden > kStaticMaxHidden || c.ffn > kStaticMaxFfn || m.q_dim > kStaticMaxQDim ||
      c.n_kv_heads > kStaticMaxKvHeads || c.n_q_heads / c.n_kv_heads > kStaticMaxGroup ||
      c.vocab > kStaticMaxVocab || m.sm_count > kStaticMaxSms)
    return fail(AS2D_ERR_UNSUPPORTED,
                "model larger than as2d_decode_step_static's fixed working memory (hidden <= "
                "4096, ffn <= 20480, n_q*head_dim <= 4096, n_kv <= 8, group <= 16, vocab <= "
                "262144, <= 192 SMs)");
  int dev = 0;
  CUDA_TRY(cudaGetDevice(&dev));
  if (dev < 0 || dev >= kStaticMaxDevices)
    return fail(AS2D_ERR_UNSUPPORTED, "device ordinal above 63");
  std::lock_guard<std::mutex> lock(g_static_mu);
  StaticDevice& sd = g_static_dev[dev];
  if (!sd.ready || sd.hidden != c.hidden || sd.q_dim != m.q_dim || sd.ffn != c.ffn) {
    // Set-up, once per device (and again only if a model of another shape is
    // used): the array's device address, then TMA descriptors of the operand
    // buffers inside it.  No allocation is involved.
    void* base = nullptr;
    CUDA_TRY(cudaGetSymbolAddress(&base, g_static_scratch));
    char* b = (char*)base;
    if (!encode_2d(&sd.tm_xn, b + kOffXn, c.hidden, 2 * kStaticRows, 64, 16) ||
        !encode_2d(&sd.tm_ao, b + kOffAo, m.q_dim, 2 * kStaticRows, 64, 16) ||
        !encode_2d(&sd.tm_u, b + kOffU, c.ffn, 2 * kStaticRows, 64, 16))
      return fail(AS2D_ERR_CUDA, "cuTensorMapEncodeTiled failed for the fixed working memory");
    sd.base = b;
    sd.hidden = c.hidden;
    sd.q_dim = m.q_dim;
    sd.ffn = c.ffn;
    sd.ready = true;
  }
  cudaStream_t st = (cudaStream_t)stream;
  char* b = sd.base;
  KvState& s = g_static_kv;
  s.model = &mh->m;
  s.batch = 1;
  s.capacity = capacity;
  s.k_cache = (bf16*)k_cache;
  s.v_cache = (bf16*)v_cache;
  s.len_upper[0] = capacity - 1;  // attention grid covers the whole cache
  s.d_len = len;
  s.d_root = root;
  s.d_err = (int32_t*)(b + kOffErr);
  s.max_rows = 1;
  s.rows_alloc = kStaticRows;
  s.nb_max = 16;
  s.h = (float*)(b + kOffH);
  s.xn = (bf16*)(b + kOffXn);
  s.qimg = (uint8_t*)(b + kOffQ);
  s.ao = (bf16*)(b + kOffAo);
  s.u = (bf16*)(b + kOffU);
  s.best = (unsigned long long*)(b + kOffBest);
  s.rope = (float2*)(b + kOffRope);
  s.ss = (float*)(b + kOffSs);
  s.ws = (float*)(b + kOffWs);
  s.counters = (int*)(b + kOffCnt);
  s.attn_o = (float*)(b + kOffAttnO);
  s.attn_ml = (float2*)(b + kOffAttnMl);
  s.attn_cnt = (int*)(b + kOffAttnCnt);
  s.n_attn_cnt = c.n_kv_heads * 8;
  s.qkv_part = (float*)(b + kOffQkvPart);
  s.qkv_rinv = (float*)(b + kOffQkvRinv);
  s.qkv_split = qkv_split_for(m);
  s.attn_qt = 1;
  s.attn_chunks = attn_chunks(capacity);
  if (!encode_cache_map(&s.tm_kc, k_cache, c.head_dim, capacity, (int64_t)c.n_layers * c.n_kv_heads) ||
      !encode_cache_map(&s.tm_vc, v_cache, c.head_dim, capacity, (int64_t)c.n_layers * c.n_kv_heads))
    return fail(AS2D_ERR_CUDA, "cuTensorMapEncodeTiled failed for a cache");
  s.tm_xn[0] = sd.tm_xn;
  s.tm_ao[0] = sd.tm_ao;
  s.tm_u[0] = sd.tm_u;
  s.prof_class = -1;
  // the array keeps the previous call's contents: clear the error words, the
  // argmax slots and the stream-K arrival counters (as many as the largest
  // projection has tiles, as for an allocated state), which must start at zero
  const int wide = c.vocab > 2 * c.ffn ? c.vocab : 2 * c.ffn;
  s.n_counters = (wide + 127) / 128 + 64;
  CUDA_TRY(cudaMemsetAsync(b + kOffErr, 0, 256, st));
  CUDA_TRY(cudaMemsetAsync(b + kOffBest, 0, kStaticRows * 8, st));
  CUDA_TRY(cudaMemsetAsync(b + kOffCnt, 0, (size_t)s.n_counters * 4, st));
  CUDA_TRY(cudaMemsetAsync(b + kOffAttnCnt, 0, (size_t)s.n_attn_cnt * 4, st));

  RowMap rm;
  rm.batch = 1;
  rm.rows = 1;
  rm.start[0] = 0;
  rm.start[1] = 1;
  as2d_verify_out out{(int32_t*)(b + kOffErr + 16), correction_token, nullptr, logits};
  const int H = c.hidden, F = c.ffn;
  LAUNCH(AS2D_KERNEL_OTHER, launch_embed(rm, m, s, nullptr, st));
  TcParams tp{};
  tp.h = s.h;
  tp.u = s.u;
  tp.logits = logits;
  tp.best = s.best;
  tp.xn = s.xn;
  tp.ss = s.ss;
  tp.ss_ld = s.rows_alloc;
  tp.lo_row = s.rows_alloc;
  tp.n_htiles = c.hidden / 128;
  tp.eps = c.rms_eps;
  tp.hidden = c.hidden;
  for (int l = 0; l < c.n_layers; ++l) {
    LAUNCH(AS2D_KERNEL_QKV, tc_project(TC_PART, m, s, rm, m.w_qkv[l], s.tm_xn, m.qkv_rows, H, tp, st));
    LAUNCH(AS2D_KERNEL_ATTENTION, launch_attention_split(rm, m, s, l, st));
    tp.g_next = m.mlp_norm[l];
    LAUNCH(AS2D_KERNEL_O, tc_project(TC_RESID, m, s, rm, m.w_o[l], s.tm_ao, H, m.q_dim, tp, st));
    LAUNCH(AS2D_KERNEL_GATE_UP, tc_project(TC_SWIGLU, m, s, rm, m.w_gu[l], s.tm_xn, 2 * F, H, tp, st));
    tp.g_next = (l + 1 < c.n_layers) ? m.attn_norm[l + 1] : m.final_norm;
    LAUNCH(AS2D_KERNEL_DOWN, tc_project(TC_RESID, m, s, rm, m.w_down[l], s.tm_u, H, F, tp, st));
  }
  LAUNCH(AS2D_KERNEL_LM_HEAD, tc_project(TC_LOGITS, m, s, rm, m.lm_head, s.tm_xn, c.vocab, H, tp, st));
  LAUNCH(AS2D_KERNEL_OTHER, launch_accept(rm, m, s, nullptr, out, st));
  // the call's device error bits, for the caller (a copy, not an allocation)
  if (error_bits)
    CUDA_TRY(cudaMemcpyAsync(error_bits, b + kOffErr, sizeof(int32_t), cudaMemcpyDeviceToDevice, st));
  return AS2D_OK;
}

static_assert(kStaticMaxVocab / 128 + 64 >= (2 * kStaticMaxFfn) / 128 + 64,
              "the counter region covers the largest projection's tiles");
static_assert(kStaticScratchBytes == 9735424, "as2d.h states the fixed working-memory size");
