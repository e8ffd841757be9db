// cpu_drafter.cu -- a small decoder run on the host cores, for a producer
// placed on a different processor than the target (the paper places drafter
// and target on different processors of one device; here the GPU verifies
// while the CPU cores draft).
//
// Host code, fp32, one greedy decode step per call over the decoder's own KV
// cache: RMSNorm, Q/K/V projections, rotate-half RoPE, grouped-query
// attention over the positions so far, output projection with residual,
// SwiGLU MLP with residual, final norm, LM head, argmax (lowest index on
// ties).  Matrix-vector products are split over `threads` OpenMP threads by
// output rows, each row's dot product vectorised (a fixed lane order per
// build).
#include <cmath>
#include <new>
#include <vector>

#include <omp.h>

#include "as2d_internal.h"

using namespace as2d;

struct as2d_cpu_decoder {
  as2d_config c;
  int threads = 1;
  int capacity = 0;
  int len = 0;
  int32_t root = 0;
  std::vector<float> embed, lm_head, final_norm;
  struct Layer {
    std::vector<float> attn_norm, wq, wk, wv, wo, mlp_norm, wg, wu, wd;
  };
  std::vector<Layer> layers;
  std::vector<float> kc, vc;  // [layers][n_kv][capacity][d]
  // scratch
  std::vector<float> x, a, q, k, v, att, o, g, u, logits, sc;
};

namespace {

void copy_in(std::vector<float>& dst, const void* src, size_t n) {
  const float* s = static_cast<const float*>(src);
  dst.assign(s, s + n);
}

// y[r] = W[r] . x for r in [0, rows), W row-major [rows][cols]
void matvec(const float* W, const float* x, float* y, int rows, int cols, int threads) {
#pragma omp parallel for num_threads(threads) schedule(static)
  for (int r = 0; r < rows; ++r) {
    const float* w = W + (size_t)r * cols;
    float acc = 0.f;
#pragma omp simd reduction(+ : acc)
    for (int i = 0; i < cols; ++i) acc += w[i] * x[i];
    y[r] = acc;
  }
}

void rmsnorm(const float* x, const float* g, float* y, int n, float eps) {
  double ss = 0;
  for (int i = 0; i < n; ++i) ss += (double)x[i] * x[i];
  const float r = (float)(1.0 / std::sqrt(ss / n + eps));
  for (int i = 0; i < n; ++i) y[i] = x[i] * r * g[i];
}

void rope(float* v, int pos, int d, float theta) {
  const int h = d / 2;
  for (int e = 0; e < h; ++e) {
    const double ang = (double)pos * std::pow((double)theta, -2.0 * e / d);
    const float c = (float)std::cos(ang), s = (float)std::sin(ang);
    const float x = v[e], y = v[e + h];
    v[e] = x * c - y * s;
    v[e + h] = y * c + x * s;
  }
}

}  // namespace

extern "C" as2d_status as2d_cpu_decoder_create(const as2d_config* cfg, const as2d_weights* w,
                                               int32_t capacity, int32_t threads, int32_t root,
                                               as2d_cpu_decoder** out) {
  clear_error();
  if (!cfg || !w || !out) return report_error(AS2D_ERR_INVALID_ARG, "cfg, weights and out are required");
  *out = nullptr;
  const as2d_config& c = *cfg;
  if (c.n_layers < 1 || c.hidden < 1 || c.n_q_heads < 1 || c.n_kv_heads < 1 || c.head_dim < 2 ||
      c.head_dim % 2 || c.ffn < 1 || c.vocab < 2 || c.n_q_heads % c.n_kv_heads)
    return report_error(AS2D_ERR_INVALID_ARG, "bad decoder shape");
  if (capacity < 1 || threads < 1 || threads > 256 || root < 0 || root >= c.vocab)
    return report_error(AS2D_ERR_INVALID_ARG, "bad capacity, threads or root");
  if (!w->embed || !w->final_norm || !w->lm_head || !w->attn_norm || !w->w_q || !w->w_k ||
      !w->w_v || !w->w_o || !w->mlp_norm || !w->w_gate || !w->w_up || !w->w_down)
    return report_error(AS2D_ERR_INVALID_ARG, "a weight pointer is NULL");
  as2d_cpu_decoder* d = new (std::nothrow) as2d_cpu_decoder();
  if (!d) return report_error(AS2D_ERR_NO_MEMORY, "out of host memory");
  try {
    const size_t H = c.hidden, F = c.ffn, V = c.vocab, D = c.head_dim;
    const size_t QD = (size_t)c.n_q_heads * D, KD = (size_t)c.n_kv_heads * D;
    d->c = c;
    d->threads = threads;
    d->capacity = capacity;
    d->root = root;
    copy_in(d->embed, w->embed, V * H);
    copy_in(d->lm_head, w->lm_head, V * H);
    copy_in(d->final_norm, w->final_norm, H);
    d->layers.resize(c.n_layers);
    for (int l = 0; l < c.n_layers; ++l) {
      auto& L = d->layers[l];
      if (!w->attn_norm[l] || !w->w_q[l] || !w->w_k[l] || !w->w_v[l] || !w->w_o[l] ||
          !w->mlp_norm[l] || !w->w_gate[l] || !w->w_up[l] || !w->w_down[l]) {
        delete d;
        return report_error(AS2D_ERR_INVALID_ARG, "a per-layer weight pointer is NULL");
      }
      copy_in(L.attn_norm, w->attn_norm[l], H);
      copy_in(L.wq, w->w_q[l], QD * H);
      copy_in(L.wk, w->w_k[l], KD * H);
      copy_in(L.wv, w->w_v[l], KD * H);
      copy_in(L.wo, w->w_o[l], H * QD);
      copy_in(L.mlp_norm, w->mlp_norm[l], H);
      copy_in(L.wg, w->w_gate[l], F * H);
      copy_in(L.wu, w->w_up[l], F * H);
      copy_in(L.wd, w->w_down[l], H * F);
    }
    d->kc.assign((size_t)c.n_layers * KD * capacity, 0.f);
    d->vc.assign((size_t)c.n_layers * KD * capacity, 0.f);
    d->x.resize(H);
    d->a.resize(H);
    d->q.resize(QD);
    d->k.resize(KD);
    d->v.resize(KD);
    d->att.resize(QD);
    d->o.resize(H);
    d->g.resize(F);
    d->u.resize(F);
    d->logits.resize(V);
    d->sc.resize(capacity);
  } catch (const std::bad_alloc&) {
    delete d;
    return report_error(AS2D_ERR_NO_MEMORY, "out of host memory");
  }
  *out = d;
  return AS2D_OK;
}

extern "C" as2d_status as2d_cpu_decoder_step(as2d_cpu_decoder* d, int32_t* token_out) {
  clear_error();
  if (!d) return report_error(AS2D_ERR_INVALID_ARG, "decoder is NULL");
  if (d->len >= d->capacity) return report_error(AS2D_ERR_CAPACITY, "the decoder's cache is full");
  const as2d_config& c = d->c;
  const int H = c.hidden, F = c.ffn, V = c.vocab, D = c.head_dim, T = d->threads;
  const int nq = c.n_q_heads, nkv = c.n_kv_heads, G = nq / nkv, pos = d->len;
  const float scale = 1.0f / std::sqrt((float)D);
  const float* e = d->embed.data() + (size_t)d->root * H;
  for (int i = 0; i < H; ++i) d->x[i] = e[i];
  for (int l = 0; l < c.n_layers; ++l) {
    auto& L = d->layers[l];
    rmsnorm(d->x.data(), L.attn_norm.data(), d->a.data(), H, c.rms_eps);
    matvec(L.wq.data(), d->a.data(), d->q.data(), nq * D, H, T);
    matvec(L.wk.data(), d->a.data(), d->k.data(), nkv * D, H, T);
    matvec(L.wv.data(), d->a.data(), d->v.data(), nkv * D, H, T);
    for (int h = 0; h < nq; ++h) rope(d->q.data() + (size_t)h * D, pos, D, c.rope_theta);
    for (int h = 0; h < nkv; ++h) {
      rope(d->k.data() + (size_t)h * D, pos, D, c.rope_theta);
      float* kd = d->kc.data() + (((size_t)l * nkv + h) * d->capacity + pos) * D;
      float* vd = d->vc.data() + (((size_t)l * nkv + h) * d->capacity + pos) * D;
      for (int i = 0; i < D; ++i) {
        kd[i] = d->k[(size_t)h * D + i];
        vd[i] = d->v[(size_t)h * D + i];
      }
    }
#pragma omp parallel for num_threads(T) schedule(static)
    for (int h = 0; h < nq; ++h) {
      const int g = h / G;
      const float* qh = d->q.data() + (size_t)h * D;
      const float* K = d->kc.data() + ((size_t)l * nkv + g) * d->capacity * D;
      const float* Vv = d->vc.data() + ((size_t)l * nkv + g) * d->capacity * D;
      std::vector<float> s(pos + 1);
      float m = -INFINITY;
      for (int t = 0; t <= pos; ++t) {
        float acc = 0.f;
        for (int i = 0; i < D; ++i) acc += qh[i] * K[(size_t)t * D + i];
        s[t] = acc * scale;
        m = s[t] > m ? s[t] : m;
      }
      float sum = 0.f;
      for (int t = 0; t <= pos; ++t) {
        s[t] = std::exp(s[t] - m);
        sum += s[t];
      }
      float* out = d->att.data() + (size_t)h * D;
      for (int i = 0; i < D; ++i) out[i] = 0.f;
      for (int t = 0; t <= pos; ++t) {
        const float p = s[t] / sum;
        for (int i = 0; i < D; ++i) out[i] += p * Vv[(size_t)t * D + i];
      }
    }
    matvec(L.wo.data(), d->att.data(), d->o.data(), H, nq * D, T);
    for (int i = 0; i < H; ++i) d->x[i] += d->o[i];
    rmsnorm(d->x.data(), L.mlp_norm.data(), d->a.data(), H, c.rms_eps);
    matvec(L.wg.data(), d->a.data(), d->g.data(), F, H, T);
    matvec(L.wu.data(), d->a.data(), d->u.data(), F, H, T);
    for (int i = 0; i < F; ++i) {
      const float gv = d->g[i];
      d->u[i] *= gv / (1.0f + std::exp(-gv));
    }
    matvec(L.wd.data(), d->u.data(), d->o.data(), H, F, T);
    for (int i = 0; i < H; ++i) d->x[i] += d->o[i];
  }
  rmsnorm(d->x.data(), d->final_norm.data(), d->a.data(), H, c.rms_eps);
  matvec(d->lm_head.data(), d->a.data(), d->logits.data(), V, H, T);
  int best = 0;
  for (int i = 1; i < V; ++i)
    if (d->logits[i] > d->logits[best]) best = i;
  d->len += 1;
  d->root = best;
  if (token_out) *token_out = best;
  return AS2D_OK;
}

extern "C" as2d_status as2d_cpu_decoder_logits(as2d_cpu_decoder* d, float* logits) {
  clear_error();
  if (!d || !logits) return report_error(AS2D_ERR_INVALID_ARG, "decoder and logits are required");
  for (int i = 0; i < d->c.vocab; ++i) logits[i] = d->logits[i];
  return AS2D_OK;
}

extern "C" as2d_status as2d_cpu_decoder_reset(as2d_cpu_decoder* d, int32_t len, int32_t root) {
  clear_error();
  if (!d) return report_error(AS2D_ERR_INVALID_ARG, "decoder is NULL");
  if (len < 0 || len > d->len || root < 0 || root >= d->c.vocab)
    return report_error(AS2D_ERR_INVALID_ARG, "len must be in [0, current length], root in [0, vocab)");
  d->len = len;
  d->root = root;
  return AS2D_OK;
}

extern "C" void as2d_cpu_decoder_free(as2d_cpu_decoder* d) { delete d; }
