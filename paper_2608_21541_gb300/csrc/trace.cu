// trace.cu — optional per-kernel timing with CUDA events (profiling aid).
//
// Off by default.  When enabled, every kernel launch of the library is
// bracketed by two events recorded on the launching stream, so durations are
// measured on the stream the kernel runs on.  Records accumulate until
// certkv_trace_report() synchronises, aggregates them per kernel name and
// clears them.  The event pool is created once, at enable time.
#include <mutex>
#include <stdio.h>
#include <string.h>
#include <vector>

#include "../../include/certkv.h"
#include "internal.cuh"

namespace certkv {

namespace {

constexpr int kPool = 1 << 15;

struct Rec {
  const char* name;
  int begin, end;
};

struct Tracer {
  bool on = false;
  std::vector<cudaEvent_t> ev;
  int used = 0;
  int open = -1;
  const char* open_name = nullptr;
  bool overflow = false;
  std::vector<Rec> recs;
  std::mutex mu;
};

Tracer& tracer() {
  static Tracer t;
  return t;
}

}  // namespace

void trace_begin(const char* name, cudaStream_t st) {
  Tracer& t = tracer();
  if (!t.on) return;
  std::lock_guard<std::mutex> g(t.mu);
  if (t.used + 2 > (int)t.ev.size()) {
    t.overflow = true;
    t.open = -1;
    return;
  }
  cudaEventRecord(t.ev[t.used], st);
  t.open = t.used++;
  t.open_name = name;
}

void trace_end(cudaStream_t st) {
  Tracer& t = tracer();
  if (!t.on) return;
  std::lock_guard<std::mutex> g(t.mu);
  if (t.open < 0) return;
  cudaEventRecord(t.ev[t.used], st);
  t.recs.push_back(Rec{t.open_name, t.open, t.used});
  ++t.used;
  t.open = -1;
}

}  // namespace certkv

extern "C" {

int certkv_trace_enable(int on) {
  using namespace certkv;
  Tracer& t = tracer();
  std::lock_guard<std::mutex> g(t.mu);
  if (on && t.ev.empty()) {
    t.ev.resize(kPool);
    for (auto& e : t.ev)
      if (cudaEventCreate(&e) != cudaSuccess) {
        t.ev.clear();
        return CERTKV_ECUDA;
      }
  }
  t.on = on != 0;
  t.used = 0;
  t.open = -1;
  t.overflow = false;
  t.recs.clear();
  return CERTKV_OK;
}

int certkv_trace_report(char* buf, size_t len) {
  using namespace certkv;
  Tracer& t = tracer();
  std::lock_guard<std::mutex> g(t.mu);
  if (!buf || len == 0) return -1;
  struct Agg {
    const char* name;
    long count;
    double ms;
  };
  std::vector<Agg> agg;
  if (!t.recs.empty() && cudaEventSynchronize(t.ev[t.recs.back().end]) != cudaSuccess) return -1;
  for (const Rec& r : t.recs) {
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, t.ev[r.begin], t.ev[r.end]) != cudaSuccess) return -1;
    size_t i = 0;
    while (i < agg.size() && strcmp(agg[i].name, r.name) != 0) ++i;
    if (i == agg.size()) agg.push_back(Agg{r.name, 0, 0.0});
    agg[i].count += 1;
    agg[i].ms += ms;
  }
  size_t off = 0;
  buf[0] = 0;
  for (const Agg& a : agg) {
    int w = snprintf(buf + off, len - off, "%s %ld %.6f\n", a.name, a.count, a.ms);
    if (w < 0 || (size_t)w >= len - off) return -1;
    off += (size_t)w;
  }
  if (t.overflow) {
    int w = snprintf(buf + off, len - off, "overflow 0 0\n");
    if (w > 0 && (size_t)w < len - off) off += (size_t)w;
  }
  t.used = 0;
  t.open = -1;
  t.overflow = false;
  t.recs.clear();
  return (int)off;
}

}  // extern "C"
