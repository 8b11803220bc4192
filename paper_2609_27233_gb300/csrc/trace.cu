// Optional per-kernel event tracing (profiling aid, off unless started).
#include <mutex>
#include <vector>

#include "common.cuh"

namespace umim {
namespace {

struct Trace {
  std::vector<cudaEvent_t> events;
  std::vector<const char *> labels;   // nullptr marks the end of a call
  int count = 0;
  bool active = false;
};

Trace &trace() {
  static Trace t;
  return t;
}

}  // namespace

void trace_mark(cudaStream_t stream, const char *label) {
  Trace &t = trace();
  if (!t.active || t.count >= (int)t.events.size()) return;
  if (cudaEventRecord(t.events[t.count], stream) != cudaSuccess) return;
  t.labels[t.count] = label;
  ++t.count;
}

}  // namespace umim

using namespace umim;

extern "C" {

umim_status umim_trace_start(int32_t capacity) {
  Trace &t = trace();
  if (capacity < 2) return UMIM_ERR_INVALID_ARG;
  if ((int)t.events.size() < capacity) {
    for (int i = (int)t.events.size(); i < capacity; ++i) {
      cudaEvent_t e;
      if (cudaEventCreate(&e) != cudaSuccess) return UMIM_ERR_CUDA;
      t.events.push_back(e);
    }
  }
  t.labels.assign(t.events.size(), nullptr);
  t.count = 0;
  t.active = true;
  return UMIM_OK;
}

void umim_trace_stop(void) { trace().active = false; }

int32_t umim_trace_read(float *ms, const char **labels, int32_t cap) {
  Trace &t = trace();
  if (t.count == 0) return 0;
  cudaEventSynchronize(t.events[t.count - 1]);
  int n = 0;
  for (int i = 0; i + 1 < t.count && n < cap; ++i) {
    if (t.labels[i] == nullptr) continue;
    float v = 0.f;
    if (cudaEventElapsedTime(&v, t.events[i], t.events[i + 1]) != cudaSuccess) v = -1.f;
    if (ms) ms[n] = v;
    if (labels) labels[n] = t.labels[i];
    ++n;
  }
  return n;
}

}  // extern "C"
