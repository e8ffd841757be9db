// cand_buffer.cu -- the candidate buffer, its read cursor and candidate
// alignment (Section 3.1 "Ordered publication and buffering"; Section 3.2
// "Candidate alignment"; App. C.1 "Source records and incremental
// publication"; App. C.3 "Candidate alignment"; Fig. 4), and the verification
// call that draws its candidates from such buffers.
//
// Host code.  The producer appends immutable batches of at most eight tokens;
// verification copies a snapshot of the published tokens from the cursor.  A
// mutex per buffer makes each entry point atomic, so a producer thread can
// publish while the verifier reads.  The alignment rules R1-R3 are stated in
// include/as2d.h beside the entry points.
#include "cand_buffer.h"

using namespace as2d;

struct as2d_cbuf {
  explicit as2d_cbuf(int window) : b(window) {}
  CandBuffer b;
};

extern "C" as2d_status as2d_cbuf_create(int32_t window, as2d_cbuf** out) {
  clear_error();
  if (!out) return report_error(AS2D_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  if (window < 1 || window > 1024)
    return report_error(AS2D_ERR_INVALID_ARG, "window must be in [1, 1024]");
  *out = new (std::nothrow) as2d_cbuf(window);
  if (!*out) return report_error(AS2D_ERR_NO_MEMORY, "out of host memory");
  return AS2D_OK;
}

extern "C" as2d_status as2d_cbuf_publish(as2d_cbuf* buf, const int32_t* tokens, int32_t n,
                                         const as2d_source_record* rec) {
  clear_error();
  if (!buf || !tokens || !rec)
    return report_error(AS2D_ERR_INVALID_ARG, "buf, tokens and rec are required");
  if (n < 1 || n > AS2D_CBUF_BATCH)
    return report_error(AS2D_ERR_INVALID_ARG, "a batch holds 1..AS2D_CBUF_BATCH tokens");
  for (int i = 0; i < n; ++i)
    if (tokens[i] < 0) return report_error(AS2D_ERR_INVALID_ARG, "token id < 0");
  return buf->b.publish(tokens, n, *rec);
}

extern "C" as2d_status as2d_cbuf_candidates(as2d_cbuf* buf, int32_t b, int32_t* tokens,
                                            int32_t* k) {
  clear_error();
  if (!buf || !k || (b > 0 && !tokens))
    return report_error(AS2D_ERR_INVALID_ARG, "buf, tokens and k are required");
  if (b < 0 || b > AS2D_MAX_K)
    return report_error(AS2D_ERR_INVALID_ARG, "b must be in [0, AS2D_MAX_K]");
  *k = buf->b.candidates(b, tokens);
  return AS2D_OK;
}

extern "C" as2d_status as2d_cbuf_after_call(as2d_cbuf* buf, int32_t k, int32_t n_accepted,
                                            int32_t correction) {
  clear_error();
  if (!buf) return report_error(AS2D_ERR_INVALID_ARG, "buf is NULL");
  return buf->b.after_call(k, n_accepted, correction);
}

extern "C" as2d_status as2d_cbuf_state(as2d_cbuf* buf, int32_t* ready, int32_t* cursor,
                                       int32_t* mode) {
  clear_error();
  if (!buf) return report_error(AS2D_ERR_INVALID_ARG, "buf is NULL");
  buf->b.state(ready, cursor, mode);
  return AS2D_OK;
}

extern "C" as2d_status as2d_cbuf_held(as2d_cbuf* buf, int32_t* tokens, int32_t* records) {
  clear_error();
  if (!buf) return report_error(AS2D_ERR_INVALID_ARG, "buf is NULL");
  buf->b.held(tokens, records);
  return AS2D_OK;
}

extern "C" as2d_status as2d_cbuf_source_of(as2d_cbuf* buf, int32_t position,
                                           as2d_source_record* out) {
  clear_error();
  if (!buf || !out) return report_error(AS2D_ERR_INVALID_ARG, "buf and out are required");
  if (!buf->b.source_of(position, out))
    return report_error(AS2D_ERR_INVALID_ARG, "position is not published or was dropped");
  return AS2D_OK;
}

extern "C" void as2d_cbuf_free(as2d_cbuf* buf) { delete buf; }

extern "C" as2d_status as2d_verify_from_buffers(as2d_kv* kh, as2d_cbuf* const* bufs, int32_t b,
                                                int32_t* k_used, int32_t* committed,
                                                int32_t* n_committed, void* stream) {
  clear_error();
  if (!kh || !bufs) return report_error(AS2D_ERR_INVALID_ARG, "kv and bufs are required");
  if (b < 0 || b > AS2D_MAX_K)
    return report_error(AS2D_ERR_INVALID_ARG, "b must be in [0, AS2D_MAX_K]");
  KvState& s = kh->s;
  const int B = s.batch;
  for (int r = 0; r < B; ++r)
    if (!bufs[r]) return report_error(AS2D_ERR_INVALID_ARG, "bufs[r] is NULL");
  const size_t words = (size_t)B * kMaxK + 2 * (size_t)B;
  if (!s.cb_dev) {
    cudaError_t e = cudaMalloc(&s.cb_dev, words * sizeof(int32_t));
    if (e != cudaSuccess) {
      s.cb_dev = nullptr;
      return report_error(AS2D_ERR_CUDA, std::string("cudaMalloc: ") + cudaGetErrorString(e));
    }
    e = cudaMallocHost(&s.cb_host, words * sizeof(int32_t));
    if (e != cudaSuccess) {
      cudaFree(s.cb_dev);
      s.cb_dev = nullptr;
      s.cb_host = nullptr;
      return report_error(AS2D_ERR_CUDA, std::string("cudaMallocHost: ") + cudaGetErrorString(e));
    }
  }
  const int32_t vocab = s.model->cfg.vocab;
  int32_t k[kMaxBatch];
  int32_t* cand = s.cb_host;  // packed: request r's candidates follow request r-1's
  int total = 0;
  for (int r = 0; r < B; ++r) {
    k[r] = bufs[r]->b.candidates(b, cand + total);
    for (int i = 0; i < k[r]; ++i)
      if (cand[total + i] >= vocab)
        return report_error(AS2D_ERR_INVALID_ARG, "a published candidate is >= vocab");
    total += k[r];
  }
  cudaStream_t st = (cudaStream_t)stream;
  int32_t* d_cand = s.cb_dev;
  int32_t* d_n = s.cb_dev + (size_t)B * kMaxK;
  int32_t* d_corr = d_n + B;
  if (total > 0) {
    cudaError_t e = cudaMemcpyAsync(d_cand, cand, total * sizeof(int32_t),
                                    cudaMemcpyHostToDevice, st);
    if (e != cudaSuccess)
      return report_error(AS2D_ERR_CUDA, std::string("cudaMemcpyAsync: ") + cudaGetErrorString(e));
  }
  as2d_verify_out out{d_n, d_corr, nullptr, nullptr};
  as2d_status rc = as2d_verify_block(kh, total > 0 ? d_cand : nullptr, k, &out, stream);
  if (rc != AS2D_OK) return rc;
  int32_t* h_n = s.cb_host + (size_t)B * kMaxK;
  cudaError_t e = cudaMemcpyAsync(h_n, d_n, 2 * B * sizeof(int32_t), cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess)
    return report_error(AS2D_ERR_CUDA, std::string("read-back: ") + cudaGetErrorString(e));
  const int32_t* h_corr = h_n + B;
  for (int r = 0; r < B; ++r)
    if (h_n[r] < 0 || h_n[r] > k[r] || h_corr[r] < 0 || h_corr[r] >= vocab)
      return report_error(AS2D_ERR_DEVICE, "verification reported an out-of-range result");
  int off = 0;
  for (int r = 0; r < B; ++r) {
    const int n = h_n[r];
    if (committed) {
      int32_t* row = committed + (size_t)r * (b + 1);
      for (int i = 0; i < n; ++i) row[i] = cand[off + i];
      row[n] = h_corr[r];
    }
    if (n_committed) n_committed[r] = n + 1;
    if (k_used) k_used[r] = k[r];
    bufs[r]->b.after_call(k[r], n, h_corr[r]);
    s.len_upper[r] -= k[r] - n;  // the call grew the length by n + 1, not k + 1
    off += k[r];
  }
  return AS2D_OK;
}
