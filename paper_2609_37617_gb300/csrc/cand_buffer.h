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

// Positions are absolute (0 = the first token ever published).  Tokens below
// every position the rules can still read (the cursor and the alignment
// position m) are discarded in steps of kDiscardStep, together with the
// records of batches that lie wholly below them (App. C.1: exhausted records
// are discarded; the rest keep their order and provenance).
class CandBuffer {
 public:
  static constexpr int kDiscardStep = 4096;

  explicit CandBuffer(int window) : window_(window) {}

  as2d_status publish(const int32_t* t, int n, const as2d_source_record& rec) {
    std::lock_guard<std::mutex> g(mu_);
    try {
      recs_.emplace_back(end(), rec);
      tok_.insert(tok_.end(), t, t + n);
    } catch (const std::bad_alloc&) {
      if (!recs_.empty() && recs_.back().first == end()) recs_.pop_back();
      return report_error(AS2D_ERR_NO_MEMORY, "out of host memory");
    }
    return AS2D_OK;
  }

  int candidates(int b, int32_t* out) {
    std::lock_guard<std::mutex> g(mu_);
    settle();
    int k = 0;
    if (mode_ != AS2D_CBUF_ALONE && cursor_ < end()) k = std::min<int>(b, end() - cursor_);
    for (int i = 0; i < k; ++i) out[i] = at(cursor_ + i);
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
    discard();
    return AS2D_OK;
  }

  void state(int32_t* ready, int32_t* cursor, int32_t* mode) {
    std::lock_guard<std::mutex> g(mu_);
    if (ready) *ready = (int32_t)end();
    if (cursor) *cursor = cursor_;
    if (mode) *mode = mode_;
  }

  // tokens and batch records still held
  void held(int32_t* tokens, int32_t* records) {
    std::lock_guard<std::mutex> g(mu_);
    if (tokens) *tokens = (int32_t)tok_.size();
    if (records) *records = (int32_t)recs_.size();
  }

  bool source_of(int pos, as2d_source_record* out) {
    std::lock_guard<std::mutex> g(mu_);
    if (pos < base_ || pos >= end()) return false;
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
  int end() const { return base_ + (int)tok_.size(); }
  int32_t at(int pos) const { return tok_[pos - base_]; }

  // Drops what no rule can read again (mu_ held).
  void discard() {
    int lo = std::min(cursor_, m_);
    if (mode_ == AS2D_CBUF_ALONE) lo = std::min(lo, std::max(f_, m_ - window_));
    if (lo - base_ < kDiscardStep) return;
    const int drop = std::min(lo, end()) - base_;
    tok_.erase(tok_.begin(), tok_.begin() + drop);
    base_ += drop;
    // keep the batch that holds position base_ and every later one
    size_t keep = 0;
    while (keep + 1 < recs_.size() && recs_[keep + 1].first <= base_) ++keep;
    recs_.erase(recs_.begin(), recs_.begin() + keep);
  }

  void settle() {
    const int ready = end();
    if (mode_ == AS2D_CBUF_REALIGN) {
      if (m_ < ready && at(m_) == x_) {
        cursor_ = m_ + 1;
        mode_ = AS2D_CBUF_NORMAL;
      }
    } else if (mode_ == AS2D_CBUF_ALONE) {
      // [s, s + W) upwards, then [max(f, s - W), s) downwards (s = m_, f = f_)
      const int hi = std::min(m_ + window_, ready);
      for (int j = m_; j < hi; ++j)
        if (at(j) == x_) {
          cursor_ = j + 1;
          mode_ = AS2D_CBUF_NORMAL;
          return;
        }
      const int lo = std::max(f_, m_ - window_);
      for (int j = std::min(m_, ready) - 1; j >= lo; --j)
        if (at(j) == x_) {
          cursor_ = j + 1;
          mode_ = AS2D_CBUF_NORMAL;
          return;
        }
    }
  }

  // R3 (mu_ held): the call with root x_ and the candidates from m_ rejected
  // its first candidate (or had none); t is the target's next token.
  void search(int32_t t) {
    const int last = end() - 1;
    const int hi = std::min(m_ + window_, last);
    for (int j = m_ + 1; j <= hi; ++j)
      if (at(j) == t) {
        cursor_ = j + 1;
        mode_ = AS2D_CBUF_NORMAL;
        return;
      }
    for (int j = m_; j <= hi; ++j)
      if (at(j) == x_) {  // x at j: the token after it stands in for t
        cursor_ = j + 2;
        mode_ = AS2D_CBUF_NORMAL;
        return;
      }
    mode_ = AS2D_CBUF_ALONE;
    m_ += 1;
    f_ = m_;
    cursor_ = m_;
    x_ = t;
  }

  std::mutex mu_;
  std::vector<int32_t> tok_;
  std::vector<std::pair<int, as2d_source_record>> recs_;  // (first position, record)
  int base_ = 0;     // absolute position of tok_[0]
  const int window_;
  int cursor_ = 0;
  int mode_ = AS2D_CBUF_NORMAL;
  int m_ = 0;        // REALIGN: position of x_; ALONE: start of the search window
  int f_ = 0;        // ALONE: where the alone search began (nothing below it is searched)
  int32_t x_ = -1;   // REALIGN: the last call's final token; ALONE: the anchor
  int last_k_ = -1;  // k handed out by the last candidates(), until after_call
};

}  // namespace as2d
