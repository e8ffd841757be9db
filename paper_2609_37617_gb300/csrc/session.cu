// session.cu -- a producer and the verifier working on one request through a
// candidate buffer, serially or overlapped, with the service-interval
// accounting of App. D.2 ("Overlap, added work, and performance limits"):
// D = |P|, V = |V|, O = |P n V|, H = |[0, T] \ (P u V)|, T = D + V - O + H.
//
// Host code.  In the overlapped run the producer is a host thread with its own
// CUDA stream: each step is one k = 0 decode step of the drafter state (the
// drafter's compute) followed by taking the step's scripted token; every
// `publish_every` steps the tokens go into the candidate buffer as one batch.
// The verifier (the calling thread) never waits for the producer: with no
// ready candidate it decodes alone (Section 3.1).  The serial comparator runs
// the same producer steps only while the verifier waits.
#include <algorithm>
#include <atomic>
#include <chrono>
#include <string>
#include <thread>
#include <vector>

#include "as2d_internal.h"

using namespace as2d;

namespace {

struct Iv {
  double a, b;
};

// Clip to [0, T], drop empty pieces, sort, and merge overlapping or touching
// intervals.
std::vector<Iv> merged(std::vector<Iv> v, double T) {
  std::vector<Iv> c;
  for (Iv x : v) {
    x.a = std::max(x.a, 0.0);
    x.b = std::min(x.b, T);
    if (x.b > x.a) c.push_back(x);
  }
  std::sort(c.begin(), c.end(), [](const Iv& x, const Iv& y) { return x.a < y.a; });
  std::vector<Iv> out;
  for (const Iv& x : c) {
    if (!out.empty() && x.a <= out.back().b)
      out.back().b = std::max(out.back().b, x.b);
    else
      out.push_back(x);
  }
  return out;
}

double length(const std::vector<Iv>& v) {
  double s = 0;
  for (const Iv& x : v) s += x.b - x.a;
  return s;
}

// |X n Y| of two merged interval lists.
double overlap(const std::vector<Iv>& x, const std::vector<Iv>& y) {
  double s = 0;
  size_t i = 0, j = 0;
  while (i < x.size() && j < y.size()) {
    const double lo = std::max(x[i].a, y[j].a), hi = std::min(x[i].b, y[j].b);
    if (hi > lo) s += hi - lo;
    if (x[i].b < y[j].b)
      ++i;
    else
      ++j;
  }
  return s;
}

void account(const std::vector<Iv>& p, const std::vector<Iv>& v, double T, double* out) {
  const std::vector<Iv> P = merged(p, T), V = merged(v, T);
  std::vector<Iv> both = P;
  both.insert(both.end(), V.begin(), V.end());
  const double U = length(merged(both, T));
  out[0] = length(P);
  out[1] = length(V);
  out[2] = overlap(P, V);
  out[3] = T - U;
  out[4] = T;
}

using Clock = std::chrono::steady_clock;

double since(Clock::time_point t0) {
  return std::chrono::duration<double>(Clock::now() - t0).count();
}

// The producer side: drafter steps and publication.
struct Producer {
  const as2d_session_spec& sp;
  Clock::time_point t0;
  int32_t* d_out = nullptr;  // device [2][AS2D_CBUF_BATCH]: n_accepted, then the token of each step
  int steps = 0;
  int published = 0;
  std::vector<Iv> iv;
  as2d_status err = AS2D_OK;
  std::string err_msg;  // as2d_last_error is per thread: kept for the caller's

  bool fail(as2d_status st) {
    err = st;
    err_msg = as2d_last_error();
    return false;
  }

  bool exhausted() const { return published >= sp.n_script; }

  // One batch: up to publish_every drafter steps, enqueued back to back (the
  // drafter's state lives on the device, so no step waits for the host), one
  // synchronisation, then the publication.  Returns false on error (err set).
  bool batch() {
    const double a = since(t0);
    const int n = std::min(sp.publish_every, sp.n_script - published);
    if (sp.cpu_drafter && !sp.drafter) {
      for (int i = 0; i < n; ++i) {
        const as2d_status st = as2d_cpu_decoder_step(sp.cpu_drafter, nullptr);
        if (st != AS2D_OK) return fail(st);
      }
    }
    if (sp.drafter) {
      for (int i = 0; i < n; ++i) {
        as2d_verify_out o{d_out + i, d_out + AS2D_CBUF_BATCH + i, nullptr, nullptr};
        as2d_status st = as2d_decode_step(sp.drafter, &o, sp.drafter_stream);
        if (st != AS2D_OK) return fail(st);
      }
      if (cudaStreamSynchronize((cudaStream_t)sp.drafter_stream) != cudaSuccess)
        return fail(report_error(AS2D_ERR_CUDA, "drafter stream synchronisation failed"));
    }
    steps += n;
    as2d_source_record rec{0, 0, 0, published, since(t0), 0.0f, 0};
    as2d_status st = as2d_cbuf_publish(sp.buf, sp.script + published, n, &rec);
    if (st != AS2D_OK) return fail(st);
    published += n;
    iv.push_back({a, since(t0)});
    return true;
  }
};

}  // namespace

extern "C" as2d_status as2d_interval_accounting(const double* p, int32_t np, const double* v,
                                                int32_t nv, double T, double* out) {
  clear_error();
  if (np < 0 || nv < 0 || !out || (np > 0 && !p) || (nv > 0 && !v) || !(T >= 0))
    return report_error(AS2D_ERR_INVALID_ARG, "bad interval arrays, counts or T");
  std::vector<Iv> P(np), V(nv);
  for (int i = 0; i < np; ++i) P[i] = {p[2 * i], p[2 * i + 1]};
  for (int i = 0; i < nv; ++i) V[i] = {v[2 * i], v[2 * i + 1]};
  for (const Iv& x : P)
    if (!(x.b >= x.a)) return report_error(AS2D_ERR_INVALID_ARG, "interval with end < start");
  for (const Iv& x : V)
    if (!(x.b >= x.a)) return report_error(AS2D_ERR_INVALID_ARG, "interval with end < start");
  account(P, V, T, out);
  return AS2D_OK;
}

extern "C" as2d_status as2d_session_run(const as2d_session_spec* spec, int32_t* committed,
                                        as2d_session_stats* stats) {
  clear_error();
  if (!spec || !stats) return report_error(AS2D_ERR_INVALID_ARG, "spec and stats are required");
  const as2d_session_spec& sp = *spec;
  if (!sp.target || !sp.buf || sp.n_script < 0 || (sp.n_script > 0 && !sp.script))
    return report_error(AS2D_ERR_INVALID_ARG, "target, buf and script are required");
  if (sp.target->s.batch != 1 || (sp.drafter && sp.drafter->s.batch != 1))
    return report_error(AS2D_ERR_INVALID_ARG, "sessions run batch-1 states");
  if (sp.b < 0 || sp.b > AS2D_MAX_K)
    return report_error(AS2D_ERR_INVALID_ARG, "b must be in [0, AS2D_MAX_K]");
  if (sp.publish_every < 1 || sp.publish_every > AS2D_CBUF_BATCH)
    return report_error(AS2D_ERR_INVALID_ARG, "publish_every must be in [1, AS2D_CBUF_BATCH]");
  if (sp.n_commit < 1) return report_error(AS2D_ERR_INVALID_ARG, "n_commit must be >= 1");
  for (int i = 0; i < sp.n_script; ++i)
    if (sp.script[i] < 0) return report_error(AS2D_ERR_INVALID_ARG, "script token < 0");
  *stats = as2d_session_stats{};

  Producer prod{sp, Clock::now()};
  if (sp.drafter) {
    cudaError_t e = cudaMalloc(&prod.d_out, 2 * AS2D_CBUF_BATCH * sizeof(int32_t));
    if (e != cudaSuccess)
      return report_error(AS2D_ERR_CUDA, std::string("cudaMalloc: ") + cudaGetErrorString(e));
  }
  std::vector<Iv> viv;
  as2d_status rc = AS2D_OK;
  int n_comm = 0;
  as2d_cbuf* bufs[1] = {sp.buf};
  int32_t row[AS2D_MAX_K + 1];

  // One verification round; returns false on error (rc set).
  auto verify_round = [&](const Clock::time_point& t0) {
    const double a = since(t0);
    int32_t k = 0, nc = 0;
    rc = as2d_verify_from_buffers(sp.target, bufs, sp.b, &k, row, &nc, sp.target_stream);
    if (rc != AS2D_OK) return false;
    viv.push_back({a, since(t0)});
    if (committed)
      for (int i = 0; i < nc; ++i) committed[n_comm + i] = row[i];
    n_comm += nc;
    stats->rounds += 1;
    stats->alone_rounds += (k == 0);
    stats->accepted += nc - 1;
    return true;
  };

  const Clock::time_point t0 = prod.t0;
  if (sp.overlapped) {
    std::atomic<bool> stop{false};
    std::thread th;
    try {
      th = std::thread([&] {
        while (!stop.load(std::memory_order_relaxed) && !prod.exhausted())
          if (!prod.batch()) {
            stop.store(true);
            break;
          }
      });
    } catch (const std::exception&) {
      cudaFree(prod.d_out);
      return report_error(AS2D_ERR_NO_MEMORY, "could not start the producer thread");
    }
    while (n_comm < sp.n_commit && !stop.load() && verify_round(t0)) {
    }
    stop.store(true);
    th.join();
    if (rc == AS2D_OK && prod.err != AS2D_OK) rc = report_error(prod.err, prod.err_msg);
  } else {
    while (n_comm < sp.n_commit) {
      int32_t ready = 0, cursor = 0;
      as2d_cbuf_state(sp.buf, &ready, &cursor, nullptr);
      if (!prod.exhausted() && ready - cursor < std::max(sp.b, 1)) {
        if (!prod.batch()) {
          rc = report_error(prod.err, prod.err_msg);
          break;
        }
        continue;
      }
      if (!verify_round(t0)) break;
    }
  }
  const double T = since(t0);
  cudaFree(prod.d_out);
  if (rc != AS2D_OK) return rc;
  double acc[5];
  account(prod.iv, viv, T, acc);
  stats->D = acc[0];
  stats->V = acc[1];
  stats->O = acc[2];
  stats->H = acc[3];
  stats->T = acc[4];
  stats->committed = n_comm;
  stats->producer_steps = prod.steps;
  stats->published = prod.published;
  return AS2D_OK;
}
