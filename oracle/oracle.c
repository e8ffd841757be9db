/*
 * oracle.c -- plain, slow CPU oracle for AS2D target-side block verification.
 *
 * TEST INFRASTRUCTURE ONLY (see oracle.h): loaded by the tests, the smoke
 * check and the CPU-baseline leg of the benchmark; never by the product path.
 *
 * Every function is the textbook definition written out, in the order the
 * definition states it.  The only parallelism is OpenMP over independent
 * output rows of a matrix-vector product and over attention heads; it does not
 * change any sum's order.  Build with -DORACLE_REAL=float for the fp32
 * self-check build; the default is double.
 */
#include "oracle.h"

#include <math.h>
#include <omp.h>
#include <stdlib.h>
#include <string.h>

#ifndef ORACLE_REAL
#define ORACLE_REAL double
#endif
typedef ORACLE_REAL real;

int32_t oracle_real_bytes(void) { return (int32_t)sizeof(real); }

int32_t oracle_set_threads(int32_t n) {
  if (n > 0) omp_set_num_threads(n);
  return (int32_t)omp_get_max_threads();
}

/* ---- bf16 conversions ------------------------------------------------- */

double oracle_bf16_to_double(uint16_t b) {
  uint32_t u = (uint32_t)b << 16;
  float f;
  memcpy(&f, &u, 4);
  return (double)f;
}

/* Round a double to the nearest bf16 value, ties to even, by scaling to the
   bf16 unit in the last place of |x| and rounding to an integer. */
uint16_t oracle_double_to_bf16(double x) {
  if (isnan(x)) return 0x7FC0;
  uint16_t sign = signbit(x) ? 0x8000 : 0;
  double ax = fabs(x);
  if (ax == 0.0) return sign;
  if (isinf(ax)) return (uint16_t)(sign | 0x7F80);
  int e;
  frexp(ax, &e); /* ax = m * 2^e, m in [0.5, 1) */
  int ulp_exp = (e - 1 < -126) ? -133 : e - 8; /* 7 fraction bits */
  double r = nearbyint(ldexp(ax, -ulp_exp));   /* default mode: ties to even */
  double y = ldexp(r, ulp_exp);
  if (y >= 0x1p128) return (uint16_t)(sign | 0x7F80);
  float f = (float)y; /* exact: y is a bf16 value */
  uint32_t u;
  memcpy(&u, &f, 4);
  return (uint16_t)(sign | (u >> 16));
}

static inline real bf(uint16_t b) { return (real)oracle_bf16_to_double(b); }

/* ---- sub-steps on `real` ------------------------------------------------ */

/* RMSNorm: y = x / sqrt(mean(x^2) + eps) * gain. */
static void rmsnorm_r(int32_t n, const real* x, const uint16_t* gain,
                      double eps, real* y) {
  real ss = 0;
  for (int32_t i = 0; i < n; ++i) ss += x[i] * x[i];
  real inv = (real)1 / (real)sqrt((double)(ss / (real)n) + eps);
  for (int32_t i = 0; i < n; ++i) y[i] = x[i] * inv * bf(gain[i]);
}

/* y = W x with W [n_out][n_in] row-major. */
static void linear_r(int32_t n_out, int32_t n_in, const uint16_t* w,
                     const real* x, real* y) {
#pragma omp parallel for schedule(static)
  for (int32_t i = 0; i < n_out; ++i) {
    const uint16_t* row = w + (int64_t)i * n_in;
    real acc = 0;
    for (int32_t j = 0; j < n_in; ++j) acc += bf(row[j]) * x[j];
    y[i] = acc;
  }
}

/* Rotary position embedding, rotate-half convention: dimension i is paired
   with i + d/2 and turned by the angle pos * theta^(-2i/d). */
static void rope_r(int32_t d, real* v, int64_t pos, double theta) {
  int32_t half = d / 2;
  for (int32_t i = 0; i < half; ++i) {
    double ang = (double)pos * pow(theta, -2.0 * (double)i / (double)d);
    real c = (real)cos(ang), s = (real)sin(ang);
    real a = v[i], b = v[i + half];
    v[i] = a * c - b * s;
    v[i + half] = b * c + a * s;
  }
}

/* Softmax attention of one query over keys [0, n_keys):
   out = sum_t softmax_t(q.K_t / sqrt(d)) V_t. */
static void attend_r(int32_t d, int64_t n_keys, const real* q,
                     const uint16_t* k_rows, const uint16_t* v_rows,
                     real* out) {
  real* s = (real*)malloc(sizeof(real) * (size_t)(n_keys > 0 ? n_keys : 1));
  real scale = (real)(1.0 / sqrt((double)d));
  real mx = -INFINITY;
  for (int64_t t = 0; t < n_keys; ++t) {
    real dot = 0;
    for (int32_t c = 0; c < d; ++c) dot += q[c] * bf(k_rows[t * d + c]);
    s[t] = dot * scale;
    if (s[t] > mx) mx = s[t];
  }
  real z = 0;
  for (int64_t t = 0; t < n_keys; ++t) {
    s[t] = (real)exp((double)(s[t] - mx));
    z += s[t];
  }
  for (int32_t c = 0; c < d; ++c) out[c] = 0;
  for (int64_t t = 0; t < n_keys; ++t) {
    real p = s[t] / z;
    for (int32_t c = 0; c < d; ++c) out[c] += p * bf(v_rows[t * d + c]);
  }
  free(s);
}

static real silu_r(real x) { return x / ((real)1 + (real)exp(-(double)x)); }

/* ---- exported sub-steps (double interface) ------------------------------ */

static real* to_real(int64_t n, const double* x) {
  real* r = (real*)calloc((size_t)(n > 0 ? n : 1), sizeof(real));
  for (int64_t i = 0; i < n; ++i) r[i] = (real)x[i];
  return r;
}
static void from_real(int64_t n, const real* r, double* x) {
  for (int64_t i = 0; i < n; ++i) x[i] = (double)r[i];
}

void oracle_rmsnorm(int32_t n, const double* x, const uint16_t* gain,
                    double eps, double* y) {
  real* xr = to_real(n, x);
  real* yr = (real*)malloc(sizeof(real) * (size_t)(n > 0 ? n : 1));
  rmsnorm_r(n, xr, gain, eps, yr);
  from_real(n, yr, y);
  free(xr);
  free(yr);
}

void oracle_linear(int32_t n_out, int32_t n_in, const uint16_t* w,
                   const double* x, double* y) {
  real* xr = to_real(n_in, x);
  real* yr = (real*)malloc(sizeof(real) * (size_t)(n_out > 0 ? n_out : 1));
  linear_r(n_out, n_in, w, xr, yr);
  from_real(n_out, yr, y);
  free(xr);
  free(yr);
}

void oracle_rope(int32_t d, double* v, int64_t pos, double theta) {
  real* r = to_real(d, v);
  rope_r(d, r, pos, theta);
  from_real(d, r, v);
  free(r);
}

void oracle_attend(int32_t d, int64_t n_keys, const double* q,
                   const uint16_t* k_rows, const uint16_t* v_rows,
                   double* out) {
  real* qr = to_real(d, q);
  real* o = (real*)malloc(sizeof(real) * (size_t)d);
  attend_r(d, n_keys, qr, k_rows, v_rows, o);
  from_real(d, o, out);
  free(qr);
  free(o);
}

double oracle_silu(double x) { return (double)silu_r((real)x); }

/* Greedy token with deterministic tie-breaking: the lowest index among the
   maxima.  margin (optional) = top-1 value minus the largest other value. */
int32_t oracle_argmax(int32_t n, const double* x, double* margin) {
  int32_t best = 0;
  for (int32_t i = 1; i < n; ++i)
    if (x[i] > x[best]) best = i;
  if (margin) {
    double second = -INFINITY;
    for (int32_t i = 0; i < n; ++i)
      if (i != best && x[i] > second) second = x[i];
    *margin = (n > 1) ? x[best] - second : INFINITY;
  }
  return best;
}

/* Greedy verification rule (Section 3.2; App. C.2): candidate c_{i+1}
   (cand[i]) is accepted while every earlier candidate was accepted and it
   equals the greedy token g_i predicted after the row before it.  The
   correction is the greedy token after the accepted prefix, g_n; when all k
   are accepted it is the bonus token g_k. */
void oracle_accept(int32_t k, const int32_t* cand, const int32_t* greedy,
                   int32_t* n_accepted, int32_t* correction) {
  int32_t n = 0;
  while (n < k && cand[n] == greedy[n]) ++n;
  *n_accepted = n;
  *correction = greedy[n];
}

/* ---- one decode step: Eq. 3 ------------------------------------------------ */

static int32_t decode_step_r(const oracle_config* c, const oracle_weights* w,
                             const oracle_kv* kv, int64_t pos, int32_t token,
                             real* logits) {
  const int32_t H = c->hidden, d = c->head_dim, nq = c->n_q, nkv = c->n_kv;
  const int32_t F = c->ffn, V = c->vocab, group = nq / nkv;
  if (pos < 0 || pos >= kv->capacity || token < 0 || token >= V) return -1;
  if (nkv <= 0 || nq % nkv != 0) return -1;

  real* h = (real*)malloc(sizeof(real) * H);
  real* a = (real*)malloc(sizeof(real) * H);
  real* q = (real*)malloc(sizeof(real) * (size_t)nq * d);
  real* kk = (real*)malloc(sizeof(real) * (size_t)nkv * d);
  real* vv = (real*)malloc(sizeof(real) * (size_t)nkv * d);
  real* o = (real*)malloc(sizeof(real) * (size_t)nq * d);
  real* y = (real*)malloc(sizeof(real) * H);
  real* gt = (real*)malloc(sizeof(real) * F);
  real* up = (real*)malloc(sizeof(real) * F);

  for (int32_t i = 0; i < H; ++i) h[i] = bf(w->embed[(int64_t)token * H + i]);

  for (int32_t l = 0; l < c->n_layers; ++l) {
    /* attention block */
    rmsnorm_r(H, h, w->attn_norm[l], c->rms_eps, a);
    linear_r(nq * d, H, w->w_q[l], a, q);
    linear_r(nkv * d, H, w->w_k[l], a, kk);
    linear_r(nkv * d, H, w->w_v[l], a, vv);
    for (int32_t j = 0; j < nq; ++j) rope_r(d, q + (int64_t)j * d, pos, c->rope_theta);
    for (int32_t g = 0; g < nkv; ++g) rope_r(d, kk + (int64_t)g * d, pos, c->rope_theta);
    for (int32_t g = 0; g < nkv; ++g) {
      uint16_t* kr = kv->k[l] + ((int64_t)g * kv->capacity + pos) * d;
      uint16_t* vr = kv->v[l] + ((int64_t)g * kv->capacity + pos) * d;
      for (int32_t e = 0; e < d; ++e) {
        kr[e] = oracle_double_to_bf16((double)kk[(int64_t)g * d + e]);
        vr[e] = oracle_double_to_bf16((double)vv[(int64_t)g * d + e]);
      }
    }
#pragma omp parallel for schedule(static)
    for (int32_t j = 0; j < nq; ++j) {
      int32_t g = j / group; /* query head j reads key/value head j / group */
      const uint16_t* kr = kv->k[l] + (int64_t)g * kv->capacity * d;
      const uint16_t* vr = kv->v[l] + (int64_t)g * kv->capacity * d;
      attend_r(d, pos + 1, q + (int64_t)j * d, kr, vr, o + (int64_t)j * d);
    }
    linear_r(H, nq * d, w->w_o[l], o, y);
    for (int32_t i = 0; i < H; ++i) h[i] += y[i];

    /* MLP block */
    rmsnorm_r(H, h, w->mlp_norm[l], c->rms_eps, a);
    linear_r(F, H, w->w_gate[l], a, gt);
    linear_r(F, H, w->w_up[l], a, up);
    for (int32_t i = 0; i < F; ++i) gt[i] = silu_r(gt[i]) * up[i];
    linear_r(H, F, w->w_down[l], gt, y);
    for (int32_t i = 0; i < H; ++i) h[i] += y[i];
  }
  rmsnorm_r(H, h, w->final_norm, c->rms_eps, a);
  linear_r(V, H, w->lm_head, a, logits);

  free(h); free(a); free(q); free(kk); free(vv); free(o); free(y);
  free(gt); free(up);
  return 0;
}

int32_t oracle_decode_step(const oracle_config* cfg, const oracle_weights* w,
                           const oracle_kv* kv, int64_t pos, int32_t token,
                           double* logits) {
  real* lr = (real*)malloc(sizeof(real) * (size_t)cfg->vocab);
  int32_t rc = decode_step_r(cfg, w, kv, pos, token, lr);
  if (rc == 0) from_real(cfg->vocab, lr, logits);
  free(lr);
  return rc;
}

/* ---- block verification: App. C.2 ----------------------------------------- */

int32_t oracle_verify_block(const oracle_config* cfg, const oracle_weights* w,
                            const oracle_kv* kv, int64_t len, int32_t root,
                            int32_t k, const int32_t* cand,
                            int32_t* n_accepted, int32_t* correction,
                            int32_t* greedy, double* logits, double* margin,
                            int64_t* new_len, int32_t* new_root) {
  const int32_t V = cfg->vocab;
  if (k < 0 || len < 0 || len + k + 1 > kv->capacity) return -1;
  for (int32_t i = 0; i < k; ++i)
    if (cand[i] < 0 || cand[i] >= V) return -1;

  double* row = (double*)malloc(sizeof(double) * (size_t)V);
  /* Row i forwards token t_i (t_0 = the known root, t_i = c_i) at position
     len + i, after rows 0..i-1 appended their keys and values: the block is
     k+1 sequential decode steps on the committed prefix followed by the
     preceding candidates (pathwise equivalence, App. C.4 requirement 1). */
  for (int32_t i = 0; i <= k; ++i) {
    int32_t tok = (i == 0) ? root : cand[i - 1];
    int32_t rc = oracle_decode_step(cfg, w, kv, len + i, tok, row);
    if (rc != 0) {
      free(row);
      return rc;
    }
    greedy[i] = oracle_argmax(V, row, margin ? &margin[i] : NULL);
    if (logits) memcpy(logits + (int64_t)i * V, row, sizeof(double) * (size_t)V);
  }
  free(row);

  oracle_accept(k, cand, greedy, n_accepted, correction);

  /* State repair (App. C.2; App. C.4 requirement 2): the retained state is
     the committed prefix plus the root and the accepted candidates; the
     rejected rows' entries are removed (here: overwritten with NaN so that a
     read of them cannot go unnoticed).  The correction is not forwarded in
     this call; it is carried as the next call's known root. */
  int64_t keep = len + *n_accepted + 1;
  for (int32_t l = 0; l < cfg->n_layers; ++l)
    for (int32_t g = 0; g < cfg->n_kv; ++g)
      for (int64_t p = keep; p < len + k + 1; ++p)
        for (int32_t e = 0; e < cfg->head_dim; ++e) {
          int64_t off = ((int64_t)g * kv->capacity + p) * cfg->head_dim + e;
          kv->k[l][off] = 0x7FC0;
          kv->v[l][off] = 0x7FC0;
        }
  *new_len = keep;
  *new_root = *correction;
  return 0;
}
