// budget.cu -- offline choice of the fixed proposal budget b from a device
// cost profile and development traces (Section 3.3 "Device-profiled
// configuration"; App. D.2 "Fixed configurations and development splits").
//
// Host code.  Each trace is replayed through the library's own candidate
// buffer (cand_buffer.h) with the whole producer text published up front and
// a target that commits the trace's reference text; every call is charged the
// profiled mean time of its width.  Budgets are ranked by pooled committed
// tokens over pooled estimated time.
#include <vector>

#include "cand_buffer.h"

using namespace as2d;

extern "C" as2d_status as2d_budget_select(const double* cost_us, const int32_t* refs,
                                          const int32_t* ref_len, const int32_t* prods,
                                          const int32_t* prod_len, int32_t n_traces,
                                          int32_t n_commit, int32_t window, int32_t b_max,
                                          double* tok_s, int32_t* calls, int32_t* best_b) {
  clear_error();
  if (!cost_us || !refs || !ref_len || !prods || !prod_len || !tok_s || !best_b)
    return report_error(AS2D_ERR_INVALID_ARG, "a required pointer is NULL");
  if (n_traces < 1 || n_commit < 1 || window < 1 || window > 1024 || b_max < 0 ||
      b_max > AS2D_MAX_K)
    return report_error(AS2D_ERR_INVALID_ARG, "bad n_traces, n_commit, window or b_max");
  for (int k = 0; k <= AS2D_MAX_K; ++k)
    if (!(cost_us[k] > 0)) return report_error(AS2D_ERR_INVALID_ARG, "cost_us must be > 0");
  std::vector<size_t> ref_off(n_traces), prod_off(n_traces);
  size_t ro = 0, po = 0;
  for (int t = 0; t < n_traces; ++t) {
    if (ref_len[t] < n_commit + b_max + 1 || prod_len[t] < 0)
      return report_error(AS2D_ERR_INVALID_ARG, "ref_len[t] < n_commit + b_max + 1");
    ref_off[t] = ro;
    prod_off[t] = po;
    ro += ref_len[t];
    po += prod_len[t];
  }
  int best = 0;
  for (int b = 0; b <= b_max; ++b) {
    double time_us = 0;
    long long committed = 0, n_calls = 0;
    int32_t cand[AS2D_MAX_K];
    for (int t = 0; t < n_traces; ++t) {
      const int32_t* ref = refs + ref_off[t];
      const int32_t* prod = prods + prod_off[t];
      CandBuffer buf(window);
      const as2d_source_record rec{t, 0, 0, 0, 0.0, 0.0f, 0};
      for (int i = 0; i < prod_len[t]; i += AS2D_CBUF_BATCH) {
        const int n = std::min(AS2D_CBUF_BATCH, prod_len[t] - i);
        for (int j = 0; j < n; ++j)
          if (prod[i + j] < 0) return report_error(AS2D_ERR_INVALID_ARG, "token id < 0");
        if (buf.publish(prod + i, n, rec) != AS2D_OK) return AS2D_ERR_NO_MEMORY;
      }
      int L = 0;
      while (L < n_commit) {
        const int k = buf.candidates(b, cand);
        int n = 0;
        while (n < k && cand[n] == ref[L + n]) ++n;
        buf.after_call(k, n, ref[L + n]);
        L += n + 1;
        time_us += cost_us[k];
        ++n_calls;
      }
      committed += L;
    }
    tok_s[b] = (double)committed / (time_us * 1e-6);
    if (calls) calls[b] = (int32_t)n_calls;
    if (tok_s[b] > tok_s[best]) best = b;
  }
  *best_b = best;
  return AS2D_OK;
}
