// cand_buffer.h -- the candidate buffer with its read cursor and the
// alignment rules R1-R3 stated in include/as2d.h (Section 3.1; Section 3.2
// "Candidate alignment"; App. C.1; App. C.3; Fig. 4).  Host code shared by
// the C-ABI buffer (cand_buffer.cu) and the offline budget estimate
// (budget.cu).  Not part of the C-ABI.
#pragma once

#include <algorithm>
#include <mutex>
#include <new>
#include <utility>
#include <vector>

#include "as2d_internal.h"

namespace as2d {

class CandBuffer {
 public:
  explicit CandBuffer(int window) : window_(window) {}

  as2d_status publish(const int32_t* t, int n, const as2d_source_record& rec) {
    std::lock_guard<std::mutex> g(mu_);
    try {
      recs_.emplace_back((int)tok_.size(), rec);
      tok_.insert(tok_.end(), t, t + n);
    } catch (const std::bad_alloc&) {
      if (!recs_.empty() && recs_.back().first == (int)tok_.size()) recs_.pop_back();
      return report_error(AS2D_ERR_NO_MEMORY, "out of host memory");
    }
    return AS2D_OK;
  }

  int candidates(int b, int32_t* out) {
    std::lock_guard<std::mutex> g(mu_);
    settle();
    int k = 0;
    if (mode_ != AS2D_CBUF_ALONE && cursor_ < (int)tok_.size())
      k = std::min<int>(b, (int)tok_.size() - cursor_);
    for (int i = 0; i < k; ++i) out[i] = tok_[cursor_ + i];
    last_k_ = k;
    return k;
  }

  as2d_status after_call(int k, int n, int32_t x) {
    std::lock_guard<std::mutex> g(mu_);
    if (k != last_k_)
      return report_error(AS2D_ERR_INVALID_ARG, "k differs from the last as2d_cbuf_candidates");
    if (n < 0 || n > k) return report_error(AS2D_ERR_INVALID_ARG, "n_accepted outside [0, k]");
    if (x < 0) return report_error(AS2D_ERR_INVALID_ARG, "correction < 0");
    last_k_ = -1;
    if (mode_ == AS2D_CBUF_ALONE) {
      // a token decoded alone retires one more position; it is the new anchor
      cursor_ = ++m_;
      x_ = x;
    } else if (mode_ == AS2D_CBUF_NORMAL || n >= 1) {
      // R1 / R2: the call's final token stands at position cursor + n
      m_ = cursor_ + n;
      x_ = x;
      cursor_ = m_;
      mode_ = AS2D_CBUF_REALIGN;
    } else {
      search(x);  // R3: root x_ with the candidates from m_ was rejected at once
    }
    return AS2D_OK;
  }

  void state(int32_t* ready, int32_t* cursor, int32_t* mode) {
    std::lock_guard<std::mutex> g(mu_);
    if (ready) *ready = (int32_t)tok_.size();
    if (cursor) *cursor = cursor_;
    if (mode) *mode = mode_;
  }

  bool source_of(int pos, as2d_source_record* out) {
    std::lock_guard<std::mutex> g(mu_);
    if (pos < 0 || pos >= (int)tok_.size()) return false;
    // the last batch starting at or before pos
    auto it = std::upper_bound(recs_.begin(), recs_.end(), pos,
                               [](int p, const std::pair<int, as2d_source_record>& r) {
                                 return p < r.first;
                               });
    *out = std::prev(it)->second;
    return true;
  }

 private:
  // Checks that wait on publication, run before each call (mu_ held): R1's
  // step over position m once it holds x, and R3's anchor search while the
  // target decodes alone.
  void settle() {
    const int ready = (int)tok_.size();
    if (mode_ == AS2D_CBUF_REALIGN) {
      if (m_ < ready && tok_[m_] == x_) {
        cursor_ = m_ + 1;
        mode_ = AS2D_CBUF_NORMAL;
      }
    } else if (mode_ == AS2D_CBUF_ALONE) {
      const int hi = std::min(m_ + window_, ready);
      for (int j = m_; j < hi; ++j)
        if (tok_[j] == x_) {
          cursor_ = j + 1;
          mode_ = AS2D_CBUF_NORMAL;
          return;
        }
    }
  }

  // R3 (mu_ held): the call with root x_ and the candidates from m_ rejected
  // its first candidate (or had none); t is the target's next token.
  void search(int32_t t) {
    const int last = (int)tok_.size() - 1;
    const int hi = std::min(m_ + window_, last);
    for (int j = m_ + 1; j <= hi; ++j)
      if (tok_[j] == t) {
        cursor_ = j + 1;
        mode_ = AS2D_CBUF_NORMAL;
        return;
      }
    for (int j = m_; j <= hi; ++j)
      if (tok_[j] == x_) {  // x at j: the token after it stands in for t
        cursor_ = j + 2;
        mode_ = AS2D_CBUF_NORMAL;
        return;
      }
    mode_ = AS2D_CBUF_ALONE;
    m_ += 1;
    cursor_ = m_;
    x_ = t;
  }

  std::mutex mu_;
  std::vector<int32_t> tok_;
  std::vector<std::pair<int, as2d_source_record>> recs_;  // (first position, record)
  const int window_;
  int cursor_ = 0;
  int mode_ = AS2D_CBUF_NORMAL;
  int m_ = 0;        // REALIGN: position of x_; ALONE: start of the search window
  int32_t x_ = -1;   // REALIGN: the last call's final token; ALONE: the anchor
  int last_k_ = -1;  // k handed out by the last candidates(), until after_call
};

}  // namespace as2d
