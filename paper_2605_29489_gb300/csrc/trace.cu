// Device-time trace of the library's calls (mp_trace_*) and the host-side NVTX ranges of
// its entry points.  A traced range is two CUDA events recorded on the stream that runs the
// range's work; the events are created when a trace starts, so recording costs one
// cudaEventRecord per end and nothing at all while no trace is held.
#include <nvtx3/nvToolsExt.h>

#include <algorithm>
#include <mutex>
#include <vector>

#include "mp_internal.cuh"

namespace mp {
namespace {

struct TraceRec {
  cudaEvent_t a = nullptr, b = nullptr;
  uint32_t kind = 0, seg = 0, stream = 0;
  bool ended = false;
};

std::mutex g_tr_mu;
std::vector<TraceRec> g_tr;            // one pair of events per range of the capacity
size_t g_tr_used = 0;                  // ranges begun
bool g_tr_on = false;                  // recording
std::vector<mp_trace_range> g_tr_out;  // resolved by mp_trace_stop

void destroy_events() {
  for (TraceRec& r : g_tr) {
    if (r.a) cudaEventDestroy(r.a);
    if (r.b) cudaEventDestroy(r.b);
  }
  g_tr.clear();
  g_tr_used = 0;
}

}  // namespace

int trace_begin(uint32_t kind, uint32_t segment, uint32_t stream_kind, cudaStream_t st) {
  std::lock_guard<std::mutex> lk(g_tr_mu);
  if (!g_tr_on || g_tr_used >= g_tr.size()) return -1;
  TraceRec& r = g_tr[g_tr_used];
  if (cudaEventRecord(r.a, st) != cudaSuccess) {
    cudaGetLastError();
    return -1;
  }
  r.kind = kind;
  r.seg = segment;
  r.stream = stream_kind;
  r.ended = false;
  return (int)g_tr_used++;
}

void trace_end(int ticket, cudaStream_t st) {
  if (ticket < 0) return;
  std::lock_guard<std::mutex> lk(g_tr_mu);
  if ((size_t)ticket >= g_tr_used) return;
  TraceRec& r = g_tr[(size_t)ticket];
  if (cudaEventRecord(r.b, st) != cudaSuccess) {
    cudaGetLastError();
    return;
  }
  r.ended = true;
}

NvtxScope::NvtxScope(const char* name) { nvtxRangePushA(name); }
NvtxScope::~NvtxScope() { nvtxRangePop(); }

}  // namespace mp

using namespace mp;

extern "C" {

mp_status mp_trace_start(uint32_t capacity) {
  if (capacity == 0 || capacity > (1u << 20)) {
    set_static_error("trace capacity must be in [1, 2^20]");
    return MP_ERR_INVALID_ARG;
  }
  std::lock_guard<std::mutex> lk(g_tr_mu);
  g_tr_on = false;
  destroy_events();
  g_tr_out.clear();
  g_tr.resize(capacity);
  for (TraceRec& r : g_tr) {
    cudaError_t e = cudaEventCreate(&r.a);
    if (e == cudaSuccess) e = cudaEventCreate(&r.b);
    if (e != cudaSuccess) {
      destroy_events();
      return cuda_fail(e, "trace events");
    }
  }
  g_tr_on = true;
  return MP_OK;
}

mp_status mp_trace_stop(uint64_t* n_ranges) {
  std::lock_guard<std::mutex> lk(g_tr_mu);
  g_tr_on = false;
  g_tr_out.clear();
  // times relative to the first range's start, shifted so that the earliest start is 0
  std::vector<std::pair<float, float>> t;
  std::vector<size_t> idx;
  if (g_tr_used > 0) {
    const cudaError_t e = cudaEventSynchronize(g_tr[0].a);
    if (e != cudaSuccess) {
      destroy_events();
      return cuda_fail(e, "trace event times");
    }
  }
  for (size_t i = 0; i < g_tr_used; ++i) {
    const TraceRec& r = g_tr[i];
    if (!r.ended) continue;
    cudaError_t e = cudaEventSynchronize(r.b);
    float t0 = 0.0f, t1 = 0.0f;
    if (e == cudaSuccess) e = cudaEventElapsedTime(&t0, g_tr[0].a, r.a);
    if (e == cudaSuccess) e = cudaEventElapsedTime(&t1, g_tr[0].a, r.b);
    if (e != cudaSuccess) {
      destroy_events();
      return cuda_fail(e, "trace event times");
    }
    t.push_back({t0, t1});
    idx.push_back(i);
  }
  float lo = 0.0f;
  for (const auto& x : t) lo = std::min(lo, x.first);
  for (size_t j = 0; j < idx.size(); ++j) {
    const TraceRec& r = g_tr[idx[j]];
    mp_trace_range q;
    q.kind = r.kind;
    q.segment = r.seg;
    q.stream = r.stream;
    q.reserved = 0;
    q.t0_ms = (double)t[j].first - lo;
    q.t1_ms = (double)t[j].second - lo;
    g_tr_out.push_back(q);
  }
  destroy_events();
  if (n_ranges) *n_ranges = g_tr_out.size();
  return MP_OK;
}

mp_status mp_trace_read(mp_trace_range* out, uint64_t n) {
  std::lock_guard<std::mutex> lk(g_tr_mu);
  if (n > g_tr_out.size()) {
    set_static_error("more ranges asked for than the trace holds");
    return MP_ERR_INVALID_ARG;
  }
  if (n && !out) {
    set_static_error("out is NULL");
    return MP_ERR_INVALID_ARG;
  }
  std::copy(g_tr_out.begin(), g_tr_out.begin() + (ptrdiff_t)n, out);
  return MP_OK;
}

}  // extern "C"
