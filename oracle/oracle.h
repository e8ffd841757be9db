/*
 * oracle.h -- plain CPU oracle for AS2D target-side block verification.
 *
 * TEST INFRASTRUCTURE.  Only the tests, the smoke check and the CPU-baseline
 * leg of the benchmark may load this library.  The CUDA library never links,
 * includes or calls it, and it shares no code with the CUDA path.
 *
 * What it computes (paper: Section 3.2 "Target verification"; App. C.2
 * "Verification and state repair"; App. C.4, Eq. 3 and Prop. 1):
 *   - the greedy target transition y_{n+1} = g(kappa_n),
 *     kappa_{n+1} = F(kappa_n, y_{n+1}) of Eq. 3, one token at a time
 *     (oracle_decode_step), for a decoder with RMSNorm, rotary positions,
 *     grouped-query attention and a SwiGLU MLP (the model family of the
 *     workloads; the paper does not describe model internals);
 *   - block verification of a known root followed by k candidates
 *     (oracle_verify_block): the k+1 rows are k+1 sequential decode steps,
 *     the longest prefix of candidates that equal the greedy tokens is
 *     committed, the greedy token after that prefix is the correction (the
 *     bonus token on full acceptance) and the KV entries of rejected rows are
 *     removed (App. C.2; Prop. 1).
 *
 * Arithmetic is in `ORACLE_REAL` (double by default; the float build is a
 * self-check).  Weights, gains and cache entries are bf16 bit patterns
 * (uint16_t).  Interfaces take and return doubles.
 */
#ifndef AS2D_ORACLE_H
#define AS2D_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct oracle_config {
  int32_t n_layers, hidden, n_q, n_kv, head_dim, ffn, vocab;
  double rope_theta, rms_eps;
} oracle_config;

/* Logical (checkpoint-style) layouts, row-major, bf16 bits, host memory:
   embed, lm_head [vocab][hidden]; final_norm, attn_norm[l], mlp_norm[l]
   [hidden]; w_q[l] [n_q*d][hidden]; w_k[l], w_v[l] [n_kv*d][hidden];
   w_o[l] [hidden][n_q*d]; w_gate[l], w_up[l] [ffn][hidden];
   w_down[l] [hidden][ffn].  Head j of q occupies rows [j*d, (j+1)*d). */
typedef struct oracle_weights {
  const uint16_t* embed;
  const uint16_t* final_norm;
  const uint16_t* lm_head;
  const uint16_t* const* attn_norm;
  const uint16_t* const* w_q;
  const uint16_t* const* w_k;
  const uint16_t* const* w_v;
  const uint16_t* const* w_o;
  const uint16_t* const* mlp_norm;
  const uint16_t* const* w_gate;
  const uint16_t* const* w_up;
  const uint16_t* const* w_down;
} oracle_weights;

/* One request's cache: k[l], v[l] each [n_kv][capacity][head_dim] bf16 bits.
   Keys are stored after rotation. */
typedef struct oracle_kv {
  uint16_t* const* k;
  uint16_t* const* v;
  int64_t capacity;
} oracle_kv;

/* bf16 <-> real (round to nearest even). */
double oracle_bf16_to_double(uint16_t b);
uint16_t oracle_double_to_bf16(double x);

/* Sub-steps, exposed so that tests can pin them. */
void oracle_rmsnorm(int32_t n, const double* x, const uint16_t* gain,
                    double eps, double* y);
void oracle_linear(int32_t n_out, int32_t n_in, const uint16_t* w,
                   const double* x, double* y);
void oracle_rope(int32_t d, double* v, int64_t pos, double theta);
void oracle_attend(int32_t d, int64_t n_keys, const double* q,
                   const uint16_t* k_rows, const uint16_t* v_rows,
                   double* out);
double oracle_silu(double x);
int32_t oracle_argmax(int32_t n, const double* x, double* margin);
void oracle_accept(int32_t k, const int32_t* cand, const int32_t* greedy,
                   int32_t* n_accepted, int32_t* correction);

/* One decode step of token `token` at position `pos` (Eq. 3): appends the
   bf16 key/value of every layer at `pos` and writes logits[vocab].
   Returns 0, or -1 on bad arguments (pos outside the cache). */
int32_t oracle_decode_step(const oracle_config* cfg, const oracle_weights* w,
                           const oracle_kv* kv, int64_t pos, int32_t token,
                           double* logits);

/* Block verification (App. C.2): rows [root, cand[0..k-1]] at positions
   L..L+k.  Outputs n_accepted, the correction token, greedy[k+1],
   optionally logits[(k+1)*vocab] and margin[k+1] (top-1 minus top-2 logit).
   Rejected rows' cache entries [L+n+1, L+k+1) are overwritten with bf16 NaN,
   so that any later read of them would show.  new_len = L+n+1 and
   new_root = correction.  Returns 0, or -1 on bad arguments. */
int32_t oracle_verify_block(const oracle_config* cfg, const oracle_weights* w,
                            const oracle_kv* kv, int64_t len, int32_t root,
                            int32_t k, const int32_t* cand,
                            int32_t* n_accepted, int32_t* correction,
                            int32_t* greedy, double* logits, double* margin,
                            int64_t* new_len, int32_t* new_root);

/* Threads of the OpenMP loops (over independent output rows and heads; the
   count changes no sum's order).  n <= 0 leaves the runtime's default.
   Returns the count the next parallel loop will use. */
int32_t oracle_set_threads(int32_t n);

/* sizeof(ORACLE_REAL) this build computes in (8 or 4). */
int32_t oracle_real_bytes(void);

#ifdef __cplusplus
}
#endif
#endif
