// Host side of the C ABI: argument validation, handle lifetime, block tables and the
// launch sequence of index, plan and merge.  Every device step runs in the kernels of
// index.cu, plan.cu and merge.cu; this file only marshals arguments and memory.
#include <float.h>
#include <limits.h>
#include <math.h>
#include <string.h>

#include <atomic>
#include <mutex>
#include <string>
#include <vector>

#include "mp_internal.cuh"

namespace mp {

namespace {
thread_local std::string g_last_error;
thread_local const char* g_static_error = nullptr;  // set instead of g_last_error by allocation-free paths

// test hooks: failures injected on the host (mp_debug_inject_fault) and device waits made to
// run out (mp_debug_stall_pipeline); nothing faults the GPU.  g_fault_left[kind] counts down
// to the event that fails; 0 = disarmed.
std::atomic<int64_t> g_fault_left[MP_FAULT_GATHER + 1];
thread_local bool g_injected = false;  // the error being reported was injected
std::atomic<uint32_t> g_stall_rounds{0};  // mp_debug_stall_pipeline: wait rounds of stalled launches (0: off)

// true when this event of the given kind is the one armed to fail (it then disarms)
bool inject_fault(int kind) {
  if (g_fault_left[kind].load(std::memory_order_relaxed) <= 0) return false;
  if (g_fault_left[kind].fetch_sub(1) != 1) return false;
  g_injected = true;
  return true;
}

// cudaMallocAsync, or an injected out-of-memory failure
cudaError_t malloc_async(void** p, size_t bytes, cudaStream_t st) {
  if (inject_fault(MP_FAULT_ALLOC)) {
    *p = nullptr;
    return cudaErrorMemoryAllocation;
  }
  return cudaMallocAsync(p, bytes, st);
}
std::atomic<uint64_t> g_next_id{1};
std::atomic<uint64_t> g_launches{0};

// pinned host slots for the small results copied back per handle and the tables a call
// uploads, in three size classes (256 bytes: plan summaries; 32 KiB: manifest counters and
// small tables; 8 MiB: block tables), recycled through free lists.  Kernels read and write
// them through the host mapping, so no copy engine is involved.
std::mutex g_pin_mu;
std::vector<void*> g_pin_free[3];
constexpr size_t kPinSlot[3] = {256, 32768, 8u << 20};
constexpr size_t kPinChunk[3] = {1u << 20, 1u << 20, 8u << 20};

int pin_class(size_t bytes) {
  return bytes <= kPinSlot[0] ? 0 : (bytes <= kPinSlot[1] ? 1 : (bytes <= kPinSlot[2] ? 2 : -1));
}

void* pin_get(size_t bytes) {
  int c = pin_class(bytes);
  if (c < 0) return nullptr;
  std::lock_guard<std::mutex> lk(g_pin_mu);
  if (g_pin_free[c].empty()) {
    void* chunk = nullptr;
    // a new chunk may be needed while a stream of this thread is being captured into a
    // graph: the allocation is host-side only, so it is made in relaxed capture mode
    cudaStreamCaptureMode mode = cudaStreamCaptureModeRelaxed;
    cudaThreadExchangeStreamCaptureMode(&mode);
    const cudaError_t e = cudaHostAlloc(&chunk, kPinChunk[c], cudaHostAllocDefault);
    cudaThreadExchangeStreamCaptureMode(&mode);
    if (e != cudaSuccess) {
      cudaGetLastError();
      return nullptr;
    }
    for (size_t k = 0; k < kPinChunk[c] / kPinSlot[c]; ++k)
      g_pin_free[c].push_back(static_cast<char*>(chunk) + kPinSlot[c] * k);
  }
  void* p = g_pin_free[c].back();
  g_pin_free[c].pop_back();
  return p;
}

void pin_put(void* p, size_t bytes) {
  int c = pin_class(bytes);
  if (!p || c < 0) return;
  std::lock_guard<std::mutex> lk(g_pin_mu);
  g_pin_free[c].push_back(p);
}

size_t align_up(size_t v) { return (v + 255) & ~(size_t)255; }

// Host data into the index's device memory by kernel: staged in a pinned slot that the handle
// keeps until mp_free, read by launch_copy over the host mapping.  Data larger than the
// largest slot goes by cudaMemcpyAsync.
cudaError_t upload(mp_index_s* ix, void* dst, const void* src, size_t bytes, cudaStream_t cs) {
  if (bytes == 0) return cudaSuccess;
  void* h = pin_get(bytes);
  if (!h) return cudaMemcpyAsync(dst, src, bytes, cudaMemcpyHostToDevice, cs);
  memcpy(h, src, bytes);
  ix->pinned.push_back({h, bytes});
  return launch_copy(dst, h, bytes, cs);
}

void release_pinned(mp_index_s* ix) {
  for (auto& q : ix->pinned) pin_put(q.first, q.second);
  ix->pinned.clear();
}

mp_status fail(mp_status st, const std::string& msg) {
  g_static_error = nullptr;
  g_last_error = msg;
  return st;
}

mp_status dev_alloc(Alloc& a, size_t bytes, cudaStream_t st) {
  a.bytes = bytes;
  a.stream = st;
  cudaError_t e = malloc_async(&a.ptr, bytes ? bytes : 256, st);
  if (e != cudaSuccess) {
    a.ptr = nullptr;
    return cuda_fail(e, "cudaMallocAsync");
  }
  return MP_OK;
}

void dev_free(Alloc& a) {
  if (a.ptr) cudaFree(a.ptr);  // synchronising free: no pending work can still use it
  a.ptr = nullptr;
}

bool is_device_ptr(const void* p) {
  cudaPointerAttributes at;
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

const void* pinned_device_view(const void* p) {
  cudaPointerAttributes at;
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  if (at.type != cudaMemoryTypeHost) return nullptr;
  return at.devicePointer;
}

mp_status build_geometry(const mp_family* f, Geometry& g) {
  if (!f) return fail(MP_ERR_INVALID_ARG, "family is NULL");
  if (f->dtype != MP_BF16 && f->dtype != MP_F32) return fail(MP_ERR_INVALID_ARG, "dtype must be MP_BF16 or MP_F32");
  if (f->K < 1 || f->K > (uint32_t)kMaxK) return fail(MP_ERR_INVALID_ARG, "K must be in 1..32");
  if (f->n_tensors < 1 || !f->tensors) return fail(MP_ERR_INVALID_ARG, "family has no tensors");
  if (f->block_elems < 256 || f->block_elems > (1u << 24) || f->block_elems % 8 != 0)
    return fail(MP_ERR_INVALID_ARG, "block_elems must be a multiple of 8 in [256, 2^24]");
  if (!f->base || !f->experts) return fail(MP_ERR_INVALID_ARG, "base or experts is NULL");
  if (f->experts_location > 1) return fail(MP_ERR_INVALID_ARG, "experts_location must be 0 or 1");
  g.dtype = f->dtype;
  g.elem_size = f->dtype == MP_BF16 ? 2u : 4u;
  g.K = f->K;
  g.block_elems = f->block_elems;
  g.n_tensors = f->n_tensors;
  g.t_off.resize(f->n_tensors);
  g.t_numel.resize(f->n_tensors);
  g.t_first_block.resize(f->n_tensors);
  uint64_t nb = 0, np = 0, end = 0;
  uint32_t maxlen = 0;
  for (uint32_t t = 0; t < f->n_tensors; ++t) {
    const mp_tensor& ts = f->tensors[t];
    if (ts.numel == 0) return fail(MP_ERR_INVALID_ARG, "tensor " + std::to_string(t) + " has numel 0");
    if ((ts.offset_elems * g.elem_size) % 16 != 0)
      return fail(MP_ERR_INVALID_ARG, "tensor " + std::to_string(t) + " does not start on a 16-byte boundary");
    if (ts.offset_elems < end)
      return fail(MP_ERR_INVALID_ARG, "tensors must be in ascending, non-overlapping offset order");
    g.t_off[t] = ts.offset_elems;
    g.t_numel[t] = ts.numel;
    g.t_first_block[t] = nb;
    uint64_t tb = (ts.numel + f->block_elems - 1) / f->block_elems;
    nb += tb;
    np += ts.numel;
    end = ts.offset_elems + ts.numel;
    uint32_t l = (uint32_t)(ts.numel < f->block_elems ? ts.numel : f->block_elems);
    if (l > maxlen) maxlen = l;
  }
  if (nb * (uint64_t)f->K > 0xFFFFFFFFull) return fail(MP_ERR_INVALID_ARG, "too many units (K * blocks >= 2^32)");
  g.n_blocks = nb;
  g.n_params = np;
  g.span_elems = end;
  g.max_blk_len = maxlen;
  if (reinterpret_cast<uintptr_t>(f->base) % 16 != 0) return fail(MP_ERR_INVALID_ARG, "base is not 16-byte aligned");
  for (uint32_t i = 0; i < f->K; ++i) {
    if (!f->experts[i]) return fail(MP_ERR_INVALID_ARG, "expert " + std::to_string(i) + " is NULL");
    if (reinterpret_cast<uintptr_t>(f->experts[i]) % 16 != 0)
      return fail(MP_ERR_INVALID_ARG, "expert " + std::to_string(i) + " is not 16-byte aligned");
  }
  return MP_OK;
}

mp_status resolve_pointers(const mp_family* f, const void*& base, ExpertPtrs& ex) {
  if (!is_device_ptr(f->base)) return fail(MP_ERR_INVALID_ARG, "base must be device memory");
  base = f->base;
  memset(&ex, 0, sizeof(ex));
  for (uint32_t i = 0; i < f->K; ++i) {
    if (f->experts_location == 0) {
      if (!is_device_ptr(f->experts[i]))
        return fail(MP_ERR_INVALID_ARG, "expert " + std::to_string(i) + " must be device memory");
      ex.p[i] = f->experts[i];
    } else {
      const void* d = pinned_device_view(f->experts[i]);
      if (!d) return fail(MP_ERR_INVALID_ARG, "expert " + std::to_string(i) + " must be pinned host memory");
      ex.p[i] = d;
    }
  }
  return MP_OK;
}

mp_status check_op(const mp_op* op, uint32_t K) {
  if (!op) return fail(MP_ERR_INVALID_ARG, "op is NULL");
  if (op->kind < MP_OP_AVG || op->kind > MP_OP_TIES_MASKED) return fail(MP_ERR_INVALID_ARG, "unknown operator kind");
  if (op->kind == MP_OP_TIES || op->kind == MP_OP_DARE_TIES || op->kind == MP_OP_TIES_MASKED) {
    if (!isfinite(op->lambda)) return fail(MP_ERR_INVALID_ARG, "lambda must be finite");
  } else {
    if (!op->alpha) return fail(MP_ERR_INVALID_ARG, "alpha is required for AVG, TA, DARE and AVG_RENORM");
    for (uint32_t i = 0; i < K; ++i)
      if (!isfinite(op->alpha[i])) return fail(MP_ERR_INVALID_ARG, "alpha must be finite");
    if (op->kind == MP_OP_AVG_RENORM)
      for (uint32_t i = 0; i < K; ++i)
        if (!(op->alpha[i] > 0.0f)) return fail(MP_ERR_INVALID_ARG, "AVG_RENORM needs every alpha > 0");
  }
  if (op->kind == MP_OP_TIES || op->kind == MP_OP_TIES_MASKED) {
    if (!(op->density >= 0.0f && op->density <= 1.0f)) return fail(MP_ERR_INVALID_ARG, "density must be in [0, 1]");
    if (op->trim_scope > 1) return fail(MP_ERR_INVALID_ARG, "trim_scope must be 0 or 1");
  }
  if ((op->kind == MP_OP_DARE || op->kind == MP_OP_DARE_TIES) && !(op->drop_p >= 0.0 && op->drop_p <= 1.0))
    return fail(MP_ERR_INVALID_ARG, "drop_p must be in [0, 1]");
  if (op->score_mode > 1) return fail(MP_ERR_INVALID_ARG, "score_mode must be 0 or 1");
  return MP_OK;
}

mp_status check_handle(const void* h, uint32_t magic, const char* what) {
  if (!h || *static_cast<const uint32_t*>(h) != magic) return fail(MP_ERR_INVALID_ARG, std::string(what) + " handle is invalid");
  return MP_OK;
}

void put_u32(std::vector<uint8_t>& v, uint32_t x) {
  for (int k = 0; k < 4; ++k) v.push_back((uint8_t)(x >> (8 * k)));
}
void put_u64(std::vector<uint8_t>& v, uint64_t x) {
  for (int k = 0; k < 8; ++k) v.push_back((uint8_t)(x >> (8 * k)));
}
uint32_t fbits(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  return u;
}

}  // namespace

void set_error(const std::string& msg) {
  g_static_error = nullptr;
  g_last_error = msg;
}

void set_static_error(const char* msg) { g_static_error = msg; }

void count_launches(uint64_t n) { g_launches.fetch_add(n, std::memory_order_relaxed); }

bool capturing(cudaStream_t st) {
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(st, &cs) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return cs == cudaStreamCaptureStatusActive;
}

// the caller's stream waits for another handle's work: inside one capture state as usual; a
// call under capture waits for an eager handle through an external event-wait node; an
// eager call on a handle built under capture relies on the caller to have run the graph
cudaError_t stream_wait(cudaStream_t cs, cudaEvent_t ev, bool ev_captured, bool now_captured) {
  if (!ev) return cudaSuccess;
  if (ev_captured == now_captured) return cudaStreamWaitEvent(cs, ev, 0);
  if (now_captured) return cudaStreamWaitEvent(cs, ev, cudaEventWaitExternal);
  return cudaSuccess;
}

cudaError_t wait_handle(cudaEvent_t done, bool captured) {
  if (captured) return cudaDeviceSynchronize();
  return done ? cudaEventSynchronize(done) : cudaSuccess;
}

mp_status cuda_fail(cudaError_t e, const char* what) {
  cudaGetLastError();
  g_static_error = nullptr;
  if (g_injected) {
    g_injected = false;
    g_last_error = std::string(what) + ": injected fault (test hook)";
    return e == cudaErrorMemoryAllocation ? MP_ERR_OOM : MP_ERR_CUDA;
  }
  g_last_error = std::string(what) + ": " + cudaGetErrorString(e);
  return e == cudaErrorMemoryAllocation ? MP_ERR_OOM : MP_ERR_CUDA;
}

mp_status new_index(const Geometry& g, const mp_op* op, bool host_pool, size_t work_bytes, cudaStream_t cs,
                    mp_index_s** out, char** work);
cudaError_t finish_index(mp_index_s* ix, cudaStream_t cs);
void discard_index(mp_index_s* ix, cudaStream_t cs);
mp_status alloc_hashes(mp_index_s* ix, cudaStream_t cs);

// ---- experts in pinned host memory: segment pipeline -------------------------------------
//
// The family is walked in segments of consecutive blocks (about kSegmentElems elements
// each).  Two HBM staging buffers alternate: while the kernels of the caller's stream
// work on segment s, segment s+1 is brought in on a side stream by a gather kernel that
// reads the host experts over the host mapping — every expert block for the index pass,
// only the planned (block, expert) pairs for the merge.  The planned blocks are scattered
// (one copy call per run of consecutive blocks would mean ~10^5 calls per merge), and the
// kernel reads them at the host link's rate.

namespace {

constexpr uint64_t kSegmentElems = 32ull << 20;
constexpr int kSide = 1;  // side streams of the host-pool gathers (one gather kernel saturates the link)

struct Segment {
  uint64_t b0, b1, e0, e1;  // blocks [b0, b1), elements [e0, e1)
};

std::vector<Segment> make_segments(const std::vector<uint64_t>& off, const std::vector<uint32_t>& len,
                                   uint64_t& max_span) {
  std::vector<Segment> segs;
  max_span = 0;
  const uint64_t nb = off.size();
  uint64_t b0 = 0;
  while (b0 < nb) {
    uint64_t b1 = b0, acc = 0;
    while (b1 < nb && (b1 == b0 || acc + len[b1] <= kSegmentElems)) acc += len[b1++];
    const uint64_t e0 = off[b0], e1 = off[b1 - 1] + len[b1 - 1];
    segs.push_back({b0, b1, e0, e1});
    if (e1 - e0 > max_span) max_span = e1 - e0;
    b0 = b1;
  }
  return segs;
}

struct HostPipe {
  cudaStream_t main = nullptr;
  cudaStream_t side[kSide] = {};
  cudaEvent_t ready[2][kSide] = {};
  cudaEvent_t freed[2] = {};
  void* staging = nullptr;
  size_t per_expert = 0;
  uint32_t K = 0;

  cudaError_t init(cudaStream_t m, uint32_t k, uint64_t span_elems, uint32_t es) {
    main = m;
    K = k;
    per_expert = align_up(span_elems * es);
    cudaError_t e;
    for (int q = 0; q < kSide; ++q)
      if ((e = cudaStreamCreateWithFlags(&side[q], cudaStreamNonBlocking)) != cudaSuccess) return e;
    for (int b = 0; b < 2; ++b) {
      for (int q = 0; q < kSide; ++q)
        if ((e = cudaEventCreateWithFlags(&ready[b][q], cudaEventDisableTiming)) != cudaSuccess) return e;
      if ((e = cudaEventCreateWithFlags(&freed[b], cudaEventDisableTiming)) != cudaSuccess) return e;
    }
    if ((e = malloc_async(&staging, 2 * (size_t)K * per_expert, main)) != cudaSuccess) {
      staging = nullptr;
      return e;
    }
    for (int b = 0; b < 2; ++b)
      if ((e = cudaEventRecord(freed[b], main)) != cudaSuccess) return e;
    return cudaSuccess;
  }

  void* buf(int b, uint32_t i) const { return static_cast<char*>(staging) + ((size_t)b * K + i) * per_expert; }

  // side streams may fill buffer b once the caller's stream has finished with it
  cudaError_t side_acquire(int b) {
    cudaError_t e;
    for (int q = 0; q < kSide; ++q)
      if ((e = cudaStreamWaitEvent(side[q], freed[b], 0)) != cudaSuccess) return e;
    return cudaSuccess;
  }

  // the caller's stream may use buffer b once the side streams have filled it
  cudaError_t main_acquire(int b) {
    cudaError_t e;
    for (int q = 0; q < kSide; ++q) {
      if ((e = cudaEventRecord(ready[b][q], side[q])) != cudaSuccess) return e;
      if ((e = cudaStreamWaitEvent(main, ready[b][q], 0)) != cudaSuccess) return e;
    }
    return cudaSuccess;
  }

  cudaError_t main_release(int b) { return cudaEventRecord(freed[b], main); }

  // the caller's stream waits for everything the side streams were given (on the normal
  // path it already has; after an error a gather may be the last work enqueued), so the
  // staging memory can be returned in the caller's stream order
  void finish() {
    for (int q = 0; q < kSide && staging; ++q) {
      if (!side[q] || !ready[0][q]) continue;
      if (cudaEventRecord(ready[0][q], side[q]) != cudaSuccess || cudaStreamWaitEvent(main, ready[0][q], 0) != cudaSuccess) {
        cudaGetLastError();
        cudaStreamSynchronize(side[q]);
      }
    }
    if (staging) cudaFreeAsync(staging, main);
    staging = nullptr;
    for (int b = 0; b < 2; ++b) {
      for (int q = 0; q < kSide; ++q)
        if (ready[b][q]) cudaEventDestroy(ready[b][q]);
      if (freed[b]) cudaEventDestroy(freed[b]);
    }
    for (int q = 0; q < kSide; ++q)
      if (side[q]) cudaStreamDestroy(side[q]);
  }
};

}  // namespace

// One walk over the segments: every expert block of a segment is brought into HBM staging by
// the gather kernel (on a side stream, one segment ahead), then `stage` enqueues the
// segment's catalog kernels on the caller's stream.  gate: when set, the gathers copy
// nothing unless *gate != 0 (the fallback walk of the windowed TIES catalog).
template <typename Stage>
cudaError_t walk_segments(const IndexLaunch& p, const mp_index_s* ix, cudaStream_t cs, const uint32_t* gate,
                          Stage stage) {
  uint64_t span = 0;
  const std::vector<Segment> segs = make_segments(ix->h_blk_off, ix->h_blk_len, span);
  HostPipe hp;
  cudaError_t e = hp.init(cs, p.K, span, ix->g.elem_size);
  for (size_t s = 0; s < segs.size() && e == cudaSuccess; ++s) {
    const int b = (int)(s & 1);
    const Segment& g = segs[s];
    if ((e = hp.side_acquire(b)) != cudaSuccess) break;
    // every expert block of the segment, read over the host mapping by a copy kernel.  It
    // moves bytes at the host link's rate, as large contiguous cudaMemcpyAsync copies do,
    // and it gathers any selection of blocks in one launch per segment, where copies would
    // take one call per run of consecutive selected blocks (the merge below gathers only
    // the planned blocks)
    GatherLaunch gl;
    memset(&gl, 0, sizeof(gl));
    gl.K = p.K;
    gl.elem_size = ix->g.elem_size;
    gl.b_begin = g.b0;
    gl.b_end = g.b1;
    gl.origin = g.e0;
    gl.blk_off = p.blk_off;
    gl.blk_len = p.blk_len;
    gl.mask = nullptr;
    gl.src = p.experts;
    gl.gate = gate;
    gl.ext = Extents{p.ext.span, span};
    gl.err = p.err;
    for (uint32_t i = 0; i < p.K; ++i) gl.dst.p[i] = hp.buf(b, i);
    if (inject_fault(MP_FAULT_GATHER)) {
      e = cudaErrorLaunchFailure;  // reported as an injected failure; nothing was launched
      break;
    }
    const int tg = trace_begin(MP_TRACE_GATHER, (uint32_t)s, 1, hp.side[0]);
    e = launch_gather(gl, hp.side[0]);
    trace_end(tg, hp.side[0]);
    if (e != cudaSuccess) break;
    if ((e = hp.main_acquire(b)) != cudaSuccess) break;
    IndexLaunch ps = p;
    ps.b_begin = g.b0;
    ps.b_end = g.b1;
    ps.expert_origin = g.e0;
    ps.ext.x_span = span;
    ps.defer_ties_select = 1;
    for (uint32_t i = 0; i < p.K; ++i) ps.experts.p[i] = hp.buf(b, i);
    const int tk = trace_begin(MP_TRACE_SEGMENT, (uint32_t)s, 0, cs);
    e = stage(ps);
    trace_end(tk, cs);
    if (e != cudaSuccess) break;
    e = hp.main_release(b);
  }
  hp.finish();
  return e;
}

cudaError_t index_host_pool(IndexLaunch p, const mp_index_s* ix, cudaStream_t cs) {
  cudaError_t e;
  if (p.wlo) {
    // the windowed TIES catalog: the sample reads the host experts in place (32 vectors per
    // block), one walk counts every pair's window, the finish marks the pairs whose threshold
    // left it; a second walk, whose gathers and kernels do nothing unless some pair was
    // marked, bins the marked groups coarsely for the two-level select
    if ((e = launch_ties_window_begin(p, cs)) != cudaSuccess) return e;
    if ((e = walk_segments(p, ix, cs, nullptr, [&](const IndexLaunch& ps) { return launch_index_pass(ps, true, cs); })) !=
        cudaSuccess)
      return e;
    if ((e = launch_ties_window_end(p, cs)) != cudaSuccess) return e;
    if ((e = walk_segments(p, ix, cs, p.miss, [&](const IndexLaunch& ps) { return launch_index_pass(ps, false, cs); })) !=
        cudaSuccess)
      return e;
  } else {
    if ((e = walk_segments(p, ix, cs, nullptr, [&](const IndexLaunch& ps) { return launch_index(ps, cs); })) !=
        cudaSuccess)
      return e;
  }
  if (p.coarse) {
    // the second level of the TIES select reads the host experts directly (fewer blocks; in
    // the windowed catalog only for the marked pairs)
    p.b_begin = 0;
    p.b_end = p.n_blocks;
    p.expert_origin = 0;
    e = launch_ties_finish(p, cs);
  }
  return e;
}

cudaError_t merge_host_pool(MergeLaunch p, const mp_index_s* ix, cudaStream_t cs) {
  uint64_t span = 0;
  const std::vector<Segment> segs = make_segments(ix->h_blk_off, ix->h_blk_len, span);
  const uint32_t es = ix->g.elem_size;
  HostPipe hp;
  cudaError_t e = hp.init(cs, p.K, span, es);
  for (size_t s = 0; s < segs.size() && e == cudaSuccess; ++s) {
    const int b = (int)(s & 1);
    const Segment& g = segs[s];
    if ((e = hp.side_acquire(b)) != cudaSuccess) break;
    GatherLaunch gl;
    memset(&gl, 0, sizeof(gl));
    gl.K = p.K;
    gl.elem_size = es;
    gl.b_begin = g.b0;
    gl.b_end = g.b1;
    gl.origin = g.e0;
    gl.blk_off = p.blk_off;
    gl.blk_len = p.blk_len;
    gl.mask = p.mask;
    gl.src = p.experts;
    gl.ext = Extents{p.ext.span, span};
    gl.err = p.err;
    for (uint32_t i = 0; i < p.K; ++i) gl.dst.p[i] = hp.buf(b, i);
    if (inject_fault(MP_FAULT_GATHER)) {
      e = cudaErrorLaunchFailure;  // reported as an injected failure; nothing was launched
      break;
    }
    const int tg = trace_begin(MP_TRACE_GATHER, (uint32_t)s, 1, hp.side[0]);
    e = launch_gather(gl, hp.side[0]);
    trace_end(tg, hp.side[0]);
    if (e != cudaSuccess) break;
    if ((e = hp.main_acquire(b)) != cudaSuccess) break;
    MergeLaunch ps = p;
    ps.b_begin = g.b0;
    ps.b_end = g.b1;
    ps.expert_origin = g.e0;
    ps.ext.x_span = span;
    ps.experts = gl.dst;
    const int tk = trace_begin(MP_TRACE_SEGMENT, (uint32_t)s, 0, cs);
    e = launch_merge(ps, cs);
    trace_end(tk, cs);
    if (e != cudaSuccess) break;
    e = hp.main_release(b);
  }
  hp.finish();
  return e;
}

// A new index handle for geometry g: one device allocation holding the block table
// (offset, length, TIES trim group and tensor of each block, first block of each tensor),
// the statistics, the error word and work_bytes of scratch for the caller (*work).  The
// table is uploaded and the error word and tau cleared on cs.
mp_status new_index(const Geometry& g, const mp_op* op, bool host_pool, size_t work_bytes, cudaStream_t cs,
                    mp_index_s** out, char** work) {
  const bool ties = op && (op->kind == MP_OP_TIES || op->kind == MP_OP_TIES_MASKED);
  const bool masked = op && op->kind == MP_OP_TIES_MASKED;
  const uint32_t scope = ties ? op->trim_scope : 0u;
  const uint32_t n_groups = scope == 0 ? g.n_tensors : 1u;
  const uint64_t nb = g.n_blocks, U = nb * g.K, KG = (uint64_t)g.K * n_groups;
  std::vector<uint64_t> h_off(nb);
  std::vector<uint32_t> h_len(nb), h_grp(nb), h_tens(nb), h_tb0(g.n_tensors + 1);
  for (uint32_t t = 0; t < g.n_tensors; ++t) {
    const uint64_t b0 = g.t_first_block[t], tb = (g.t_numel[t] + g.block_elems - 1) / g.block_elems;
    h_tb0[t] = (uint32_t)b0;
    for (uint64_t k = 0; k < tb; ++k) {
      h_off[b0 + k] = g.t_off[t] + k * g.block_elems;
      const uint64_t rem = g.t_numel[t] - k * g.block_elems;
      h_len[b0 + k] = (uint32_t)(rem < g.block_elems ? rem : g.block_elems);
      h_grp[b0 + k] = scope == 0 ? t : 0u;
      h_tens[b0 + k] = t;
    }
  }
  h_tb0[g.n_tensors] = (uint32_t)nb;

  size_t o = 0;
  auto slot = [&](size_t bytes) { size_t r = o; o += align_up(bytes); return r; };
  const size_t o_off = slot(nb * 8), o_len = slot(nb * 4), o_grp = slot(nb * 4), o_tens = slot(nb * 4);
  const size_t o_tb0 = slot(((size_t)g.n_tensors + 1) * 4);
  const size_t o_norm = slot(U * 4), o_max = slot(U * 4), o_nnz = slot(U * 4), o_tau = slot(KG * 4);
  const size_t o_err = slot(16);
  const size_t o_uh = slot(masked ? U * 256 * 4 : 0);
  const size_t o_work = slot(work_bytes);
  mp_index_s* ix = new (std::nothrow) mp_index_s();
  if (!ix) return fail(MP_ERR_OOM, "host allocation failed");
  ix->magic = kMagicIndex;
  ix->id = g_next_id++;
  cudaGetDevice(&ix->device);
  ix->g = g;
  ix->op_kind = op ? (int)op->kind : -1;
  ix->density = ties ? op->density : 0.0f;
  ix->trim_scope = scope;
  ix->n_groups = n_groups;
  ix->has_missing = false;
  ix->done = nullptr;
  ix->captured = capturing(cs);
  ix->order_captured = false;
  ix->order_ready = nullptr;
  ix->order_mu = new (std::nothrow) std::mutex();
  if (!ix->order_mu) {
    delete ix;
    return fail(MP_ERR_OOM, "host allocation failed");
  }
  mp_status st;
  if ((st = dev_alloc(ix->mem, o, cs)) != MP_OK) {
    delete ix->order_mu;
    delete ix;
    return st;
  }
  char* m = static_cast<char*>(ix->mem.ptr);
  ix->d_blk_off = (uint64_t*)(m + o_off);
  ix->d_blk_len = (uint32_t*)(m + o_len);
  ix->d_blk_group = (uint32_t*)(m + o_grp);
  ix->d_blk_tensor = (uint32_t*)(m + o_tens);
  ix->d_t_blk0 = (uint32_t*)(m + o_tb0);
  ix->d_norm = (float*)(m + o_norm);
  ix->d_maxabs = (float*)(m + o_max);
  ix->d_nnz = (uint32_t*)(m + o_nnz);
  ix->d_tau = (uint32_t*)(m + o_tau);
  ix->d_err = (uint32_t*)(m + o_err);
  ix->d_unit_hist = masked ? (uint32_t*)(m + o_uh) : nullptr;
  cudaError_t e = cudaSuccess;
  const char* what = "block table copy";
  {
    // the five table arrays are consecutive in the allocation: one staged upload
    const size_t t_end = o_tb0 + ((size_t)g.n_tensors + 1) * 4;
    std::vector<char> tab(t_end, 0);
    memcpy(tab.data() + o_off, h_off.data(), nb * 8);
    memcpy(tab.data() + o_len, h_len.data(), nb * 4);
    memcpy(tab.data() + o_grp, h_grp.data(), nb * 4);
    memcpy(tab.data() + o_tens, h_tens.data(), nb * 4);
    memcpy(tab.data() + o_tb0, h_tb0.data(), ((size_t)g.n_tensors + 1) * 4);
    e = upload(ix, m, tab.data(), t_end, cs);
  }
  if (e == cudaSuccess) what = "fill", e = launch_fill(ix->d_err, 0, 16, cs);
  if (e == cudaSuccess) e = launch_fill(ix->d_tau, 0, KG * 4, cs);
  if (e != cudaSuccess) {
    mp_status r = cuda_fail(e, what);
    discard_index(ix, cs);
    return r;
  }
  if (host_pool) {
    ix->h_blk_off = std::move(h_off);
    ix->h_blk_len = std::move(h_len);
  }
  *out = ix;
  *work = m + o_work;
  return MP_OK;
}

// the handle is complete once the stream reaches this point
cudaError_t finish_index(mp_index_s* ix, cudaStream_t cs) {
  cudaError_t e;
  if ((e = cudaEventCreateWithFlags(&ix->done, cudaEventDisableTiming)) != cudaSuccess) return e;
  return cudaEventRecord(ix->done, cs);
}

// the catalog's hash arrays (base, then K experts), allocated once per index
mp_status alloc_hashes(mp_index_s* ix, cudaStream_t cs) {
  if (ix->hash_mem.ptr) return MP_OK;
  const uint64_t nb = ix->g.n_blocks;
  mp_status st = dev_alloc(ix->hash_mem, (size_t)(ix->g.K + 1) * nb * 8, cs);
  if (st != MP_OK) return st;
  ix->d_base_hash = static_cast<unsigned long long*>(ix->hash_mem.ptr);
  ix->d_expert_hash = ix->d_base_hash + nb;
  return MP_OK;
}

// frees a handle whose construction failed (after the stream's work on it is done)
void discard_index(mp_index_s* ix, cudaStream_t cs) {
  cudaStreamSynchronize(cs);
  cudaGetLastError();
  release_pinned(ix);
  dev_free(ix->hash_mem);
  dev_free(ix->order_mem);
  dev_free(ix->mem);
  if (ix->done) cudaEventDestroy(ix->done);
  if (ix->order_ready) cudaEventDestroy(ix->order_ready);
  delete ix->order_mu;
  delete ix;
}

}  // namespace mp

using namespace mp;

extern "C" {

const char* mp_last_error(void) { return g_static_error ? g_static_error : g_last_error.c_str(); }

const char* mp_version(void) {
  return kChecked ? "mergepipe-gb300 0.1 (sm_103a, checked)" : "mergepipe-gb300 0.1 (sm_103a)";
}

uint64_t mp_kernel_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

mp_status mp_debug_inject_fault(int32_t kind, uint64_t n) {
  if (kind != MP_FAULT_ALLOC && kind != MP_FAULT_GATHER) return fail(MP_ERR_INVALID_ARG, "unknown fault kind");
  g_fault_left[kind].store(n > (uint64_t)INT64_MAX ? INT64_MAX : (int64_t)n, std::memory_order_relaxed);
  return MP_OK;
}

void mp_debug_stall_pipeline(uint32_t rounds) { g_stall_rounds.store(rounds, std::memory_order_relaxed); }

uint64_t mp_budget_from_fraction(const mp_family* family, double f) {
  Geometry g;
  if (build_geometry(family, g) != MP_OK) return 0;
  if (!(f > 0.0)) return 0;
  if (f > 1.0) f = 1.0;
  const uint64_t full = (uint64_t)g.K * g.n_params * g.elem_size;
  return (uint64_t)floor(f * (double)full);
}

mp_status mp_index_blocks(const mp_family* family, const mp_op* op, mp_stream stream, mp_index** out) {
  NvtxScope nv("mp_index_blocks");
  if (!out) return fail(MP_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  Geometry g;
  mp_status st = build_geometry(family, g);
  if (st != MP_OK) return st;
  const bool ties = op && (op->kind == MP_OP_TIES || op->kind == MP_OP_TIES_MASKED);
  if (op && (st = check_op(op, g.K)) != MP_OK) return st;
  const void* base;
  ExpertPtrs ex;
  if ((st = resolve_pointers(family, base, ex)) != MP_OK) return st;
  cudaStream_t cs = reinterpret_cast<cudaStream_t>(stream);
  TraceScope tr(MP_TRACE_INDEX, cs);

  const uint32_t scope = ties ? op->trim_scope : 0u;
  const uint32_t n_groups = scope == 0 ? g.n_tensors : 1u;
  const uint64_t KG = (uint64_t)g.K * n_groups;
  std::vector<unsigned long long> h_kth(n_groups, 0);
  if (ties) {
    std::vector<uint64_t> gnumel(n_groups, 0);
    for (uint32_t t = 0; t < g.n_tensors; ++t) gnumel[scope == 0 ? t : 0] += g.t_numel[t];
    for (uint32_t q = 0; q < n_groups; ++q)
      h_kth[q] = (unsigned long long)floor((double)op->density * (double)gnumel[q]);
  }
  // the index kernels' work space after the handle's own arrays
  size_t o = 0;
  auto slot = [&](size_t bytes) { size_t r = o; o += align_up(bytes); return r; };
  const size_t o_work = slot(16);  // the index kernel's work counter
  size_t o_coarse = 0, o_fine = 0, o_kth = 0, o_est = 0, o_rank = 0;
  size_t o_wfine = 0, o_wabove = 0, o_wlo = 0, o_gmiss = 0, o_miss = 0, o_wend = 0;
  // device-resident TIES (not after masking) takes its thresholds from predicted windows
  const bool windowed = ties && op->kind == MP_OP_TIES;
  if (ties) {
    o_coarse = slot(KG * 256 * 8);
    o_fine = slot(KG * 128 * 8);
    o_kth = slot(n_groups * 8);
    o_est = slot(KG * 4);
    o_rank = slot(KG * 8);
  }
  // the sampling CTAs' spans: up to 64 blocks of one trim group each
  std::vector<uint32_t> h_spans;
  size_t o_shist = 0, o_scnt = 0, o_spans = 0;
  if (windowed) {
    for (uint32_t q = 0; q < n_groups; ++q) {
      const uint64_t b0 = scope == 0 ? g.t_first_block[q] : 0;
      const uint64_t b1 = scope == 0 ? (q + 1 < g.n_tensors ? g.t_first_block[q + 1] : g.n_blocks) : g.n_blocks;
      for (uint64_t b = b0; b < b1; b += 64) {
        h_spans.push_back(q);
        h_spans.push_back((uint32_t)b);
      }
    }
    // zeroed together: window counts, keys above, marks, the flag, sampled bins and counts
    o_wfine = slot(KG * 384 * 8);
    o_wabove = slot(KG * 8);
    o_gmiss = slot(KG * 4);
    o_miss = slot(16);
    o_shist = slot(KG * 256 * 8);
    o_scnt = slot(n_groups * 8);
    o_wend = o;
    o_wlo = slot(KG * 4);
    o_spans = slot(h_spans.size() * 4);
  }
  mp_index_s* ix = nullptr;
  char* m = nullptr;
  if ((st = new_index(g, op, family->experts_location != 0, o, cs, &ix, &m)) != MP_OK) return st;

  cudaError_t e;
  auto bail = [&](cudaError_t err, const char* what) {
    mp_status r = cuda_fail(err, what);
    discard_index(ix, cs);
    return r;
  };
  IndexLaunch p;
  memset(&p, 0, sizeof(p));
  p.dtype = g.dtype;
  p.K = g.K;
  p.n_blocks = g.n_blocks;
  p.n_groups = n_groups;
  p.base = base;
  p.experts = ex;
  p.blk_off = ix->d_blk_off;
  p.blk_len = ix->d_blk_len;
  p.blk_group = ix->d_blk_group;
  p.norm = ix->d_norm;
  p.maxabs = ix->d_maxabs;
  p.nnz = ix->d_nnz;
  p.err = ix->d_err;
  p.work = (unsigned long long*)(m + o_work);
  p.wait_limit = g_stall_rounds.load(std::memory_order_relaxed);
  p.stall = p.wait_limit ? 1u : 0u;
  if (ties) {
    p.coarse = (unsigned long long*)(m + o_coarse);
    p.fine = (unsigned long long*)(m + o_fine);
    p.kth = (const unsigned long long*)(m + o_kth);
    p.estar = (uint32_t*)(m + o_est);
    p.rank = (unsigned long long*)(m + o_rank);
    p.tau = ix->d_tau;
    p.unit_hist = ix->d_unit_hist;
    if ((e = launch_fill(p.coarse, 0, KG * 256 * 8, cs)) != cudaSuccess) return bail(e, "fill");
    if ((e = launch_fill(p.fine, 0, KG * 128 * 8, cs)) != cudaSuccess) return bail(e, "fill");
    if ((e = upload(ix, (void*)p.kth, h_kth.data(), n_groups * 8, cs)) != cudaSuccess) return bail(e, "k copy");
  }
  if (windowed) {
    p.density = op->density;
    p.grp_blk0 = ix->d_t_blk0;
    p.wfine = (unsigned long long*)(m + o_wfine);
    p.wabove = (unsigned long long*)(m + o_wabove);
    p.gmiss = (uint32_t*)(m + o_gmiss);
    p.miss = (uint32_t*)(m + o_miss);
    p.wlo = (uint32_t*)(m + o_wlo);
    p.shist = (unsigned long long*)(m + o_shist);
    p.scnt = (unsigned long long*)(m + o_scnt);
    p.samp_span = (const uint2*)(m + o_spans);
    p.n_samp_spans = (uint32_t)(h_spans.size() / 2);
    if ((e = launch_fill(m + o_wfine, 0, o_wend - o_wfine, cs)) != cudaSuccess) return bail(e, "fill");
    if ((e = upload(ix, m + o_spans, h_spans.data(), h_spans.size() * 4, cs)) != cudaSuccess)
      return bail(e, "span copy");
  }
  p.b_begin = 0;
  p.b_end = g.n_blocks;
  p.expert_origin = 0;
  p.ext = Extents{g.span_elems, g.span_elems};
  if (family->experts_location == 0) {
    if ((e = launch_index(p, cs)) != cudaSuccess) return bail(e, "index kernels");
  } else {
    if ((e = index_host_pool(p, ix, cs)) != cudaSuccess) return bail(e, "index (host pool)");
  }
  if ((e = finish_index(ix, cs)) != cudaSuccess) return bail(e, "event");
  *out = ix;
  return MP_OK;
}

mp_status mp_index_import(const mp_family* family, const mp_op* op, const float* norm, const float* maxabs,
                          const uint32_t* nnz, const uint32_t* tau, const uint64_t* base_hash,
                          const uint64_t* expert_hash, mp_stream stream, mp_index** out) {
  if (!out) return fail(MP_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  Geometry g;
  mp_status st = build_geometry(family, g);
  if (st != MP_OK) return st;
  const bool ties = op && op->kind == MP_OP_TIES;
  if (op && (st = check_op(op, g.K)) != MP_OK) return st;
  if (op && op->kind == MP_OP_TIES_MASKED)
    return fail(MP_ERR_UNSUPPORTED, "a TIES_MASKED catalog holds per-block key histograms, which are not imported");
  if (!norm || !maxabs || !nnz) return fail(MP_ERR_INVALID_ARG, "norm, maxabs and nnz are required");
  if (ties && !tau) return fail(MP_ERR_INVALID_ARG, "a TIES catalog needs tau");
  if ((base_hash == nullptr) != (expert_hash == nullptr))
    return fail(MP_ERR_INVALID_ARG, "block hashes come as base_hash and expert_hash together");
  const uint32_t n_groups = (ties && op->trim_scope == 1) ? 1u : g.n_tensors;
  const uint64_t nb = g.n_blocks, U = nb * g.K, KG = (uint64_t)g.K * n_groups;
  // every entry is either statistics of its block or marked missing
  bool missing = false;
  for (uint32_t t = 0; t < g.n_tensors; ++t) {
    const uint64_t b0 = g.t_first_block[t], tb = (g.t_numel[t] + g.block_elems - 1) / g.block_elems;
    for (uint64_t k = 0; k < tb; ++k) {
      const uint64_t rem = g.t_numel[t] - k * g.block_elems;
      const uint32_t len = (uint32_t)(rem < g.block_elems ? rem : g.block_elems);
      for (uint32_t i = 0; i < g.K; ++i) {
        const uint64_t q = (uint64_t)i * nb + b0 + k;
        if (nnz[q] == MP_NNZ_MISSING) {
          missing = true;
          continue;
        }
        if (nnz[q] > len || !(norm[q] >= 0.0f && norm[q] <= FLT_MAX) || !(maxabs[q] >= 0.0f && maxabs[q] <= FLT_MAX))
          return fail(MP_ERR_INVALID_ARG, "catalog entry " + std::to_string(q) +
                                              " is not a block statistic (nnz above the block length, or a "
                                              "negative or non-finite norm or maxabs)");
      }
    }
  }
  if (ties)
    for (uint64_t q = 0; q < KG; ++q)
      if (tau[q] > 0x8000u) return fail(MP_ERR_INVALID_ARG, "tau entries must be in [0, 0x8000]");
  cudaStream_t cs = reinterpret_cast<cudaStream_t>(stream);
  mp_index_s* ix = nullptr;
  char* m = nullptr;
  if ((st = new_index(g, op, family->experts_location != 0, 0, cs, &ix, &m)) != MP_OK) return st;
  ix->has_missing = missing;
  cudaError_t e;
  auto bail = [&](cudaError_t err, const char* what) {
    mp_status r = cuda_fail(err, what);
    discard_index(ix, cs);
    return r;
  };
  if ((e = cudaMemcpyAsync(ix->d_norm, norm, U * 4, cudaMemcpyHostToDevice, cs)) != cudaSuccess)
    return bail(e, "catalog copy");
  if ((e = cudaMemcpyAsync(ix->d_maxabs, maxabs, U * 4, cudaMemcpyHostToDevice, cs)) != cudaSuccess)
    return bail(e, "catalog copy");
  if ((e = cudaMemcpyAsync(ix->d_nnz, nnz, U * 4, cudaMemcpyHostToDevice, cs)) != cudaSuccess)
    return bail(e, "catalog copy");
  if (ties && (e = cudaMemcpyAsync(ix->d_tau, tau, KG * 4, cudaMemcpyHostToDevice, cs)) != cudaSuccess)
    return bail(e, "catalog copy");
  if (base_hash) {
    if ((st = alloc_hashes(ix, cs)) != MP_OK) {
      discard_index(ix, cs);
      return st;
    }
    if ((e = cudaMemcpyAsync(ix->d_base_hash, base_hash, nb * 8, cudaMemcpyHostToDevice, cs)) != cudaSuccess)
      return bail(e, "hash copy");
    if ((e = cudaMemcpyAsync(ix->d_expert_hash, expert_hash, U * 8, cudaMemcpyHostToDevice, cs)) != cudaSuccess)
      return bail(e, "hash copy");
  }
  if ((e = finish_index(ix, cs)) != cudaSuccess) return bail(e, "event");
  *out = ix;
  return MP_OK;
}

mp_status mp_plan(const mp_index* index, const mp_op* op, uint64_t budget_bytes, mp_stream stream, mp_plan_t** out) {
  NvtxScope nv("mp_plan");
  if (!out) return fail(MP_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  mp_status st;
  if ((st = check_handle(index, kMagicIndex, "index")) != MP_OK) return st;
  const Geometry& g = index->g;
  if ((st = check_op(op, g.K)) != MP_OK) return st;
  if ((op->kind == MP_OP_TIES || op->kind == MP_OP_TIES_MASKED) &&
      (index->op_kind != op->kind || index->density != op->density || index->trim_scope != op->trim_scope))
    return fail(MP_ERR_MISMATCH, "a TIES plan needs an index built for the same TIES kind, density and trim scope");
  cudaStream_t cs = reinterpret_cast<cudaStream_t>(stream);
  TraceScope tr(MP_TRACE_PLAN, cs);
  const uint64_t nb = g.n_blocks, U = nb * g.K;

  mp_plan_s* pl = new (std::nothrow) mp_plan_s();
  if (!pl) return fail(MP_ERR_OOM, "host allocation failed");
  pl->magic = kMagicPlan;
  pl->id = g_next_id++;
  pl->index_id = index->id;
  pl->device = index->device;
  pl->g = g;
  pl->op_kind = op->kind;
  for (uint32_t i = 0; i < kMaxK; ++i) pl->alpha[i] = (op->alpha && i < g.K) ? op->alpha[i] : 0.0f;
  pl->lambda = op->lambda;
  pl->density = op->density;
  pl->trim_scope = op->trim_scope;
  pl->drop_p = op->drop_p;
  pl->seed = op->seed;
  pl->budget = budget_bytes;
  pl->n_groups = index->n_groups;
  pl->done = nullptr;
  pl->captured = capturing(cs);
  pl->h_summary = static_cast<uint64_t*>(pin_get(64));
  if (!pl->h_summary) {
    delete pl;
    return fail(MP_ERR_OOM, "pinned host allocation failed");
  }
  size_t o = 0;
  auto slot = [&](size_t bytes) { size_t r = o; o += align_up(bytes); return r; };
  const size_t o_mask = slot(nb * 4), o_order = slot(U * 4), o_sum = slot(8 * 8);
  if ((st = dev_alloc(pl->mem, o, cs)) != MP_OK) {
    pin_put(pl->h_summary, 64);
    delete pl;
    return st;
  }
  char* m = static_cast<char*>(pl->mem.ptr);
  pl->d_mask = (uint32_t*)(m + o_mask);
  pl->d_order = (uint32_t*)(m + o_order);
  pl->d_summary = (uint64_t*)(m + o_sum);

  Alloc scratch;
  auto bail = [&](cudaError_t err, const char* what) {
    mp_status r = cuda_fail(err, what);
    cudaStreamSynchronize(cs);
    if (scratch.ptr) cudaFree(scratch.ptr);
    dev_free(pl->mem);
    pin_put(pl->h_summary, 64);
    if (pl->done) cudaEventDestroy(pl->done);
    delete pl;
    return r;
  };
  cudaError_t e;
  if ((e = stream_wait(cs, index->done, index->captured, pl->captured)) != cudaSuccess) return bail(e, "stream wait");
  const uint64_t n_pairs = index->has_missing ? (uint64_t)g.K * g.n_tensors : 0ull;
  if ((e = malloc_async(&scratch.ptr, plan_scratch_bytes(U, n_pairs), cs)) != cudaSuccess) {
    scratch.ptr = nullptr;
    return bail(e, "plan scratch");
  }

  PlanLaunch p;
  memset(&p, 0, sizeof(p));
  p.K = g.K;
  p.n_blocks = nb;
  p.n_groups = index->n_groups;
  p.elem_size = g.elem_size;
  p.op_kind = op->kind;
  p.score_mode = op->score_mode;
  const bool by_lambda = op->kind == MP_OP_TIES || op->kind == MP_OP_DARE_TIES || op->kind == MP_OP_TIES_MASKED;
  for (uint32_t i = 0; i < g.K; ++i) p.coef[i] = fabsf(by_lambda ? op->lambda : op->alpha[i]);
  p.blk_len = index->d_blk_len;
  p.blk_group = index->d_blk_group;
  p.norm = index->d_norm;
  p.maxabs = index->d_maxabs;
  p.nnz = index->d_nnz;
  p.tau = index->d_tau;
  p.index_err = index->d_err;
  p.fallback = index->has_missing ? 1u : 0u;
  p.n_tensors = g.n_tensors;
  p.blk_tensor = index->d_blk_tensor;
  p.t_blk0 = index->d_t_blk0;
  p.budget = budget_bytes;
  p.mask = pl->d_mask;
  p.order = pl->d_order;
  p.summary = pl->d_summary;
  std::vector<uint8_t> hdr;
  put_u32(hdr, (uint32_t)op->kind);
  put_u32(hdr, g.K);
  for (uint32_t i = 0; i < g.K; ++i) put_u32(hdr, op->alpha ? fbits(op->alpha[i]) : 0u);
  put_u32(hdr, fbits(op->lambda));
  put_u32(hdr, fbits(op->density));
  put_u32(hdr, op->trim_scope);
  uint64_t pb;
  memcpy(&pb, &op->drop_p, 8);
  put_u64(hdr, pb);
  put_u64(hdr, op->seed);
  put_u32(hdr, op->score_mode);
  const std::vector<uint8_t> order_key = hdr;  // everything the traversal order depends on
  put_u64(hdr, budget_bytes);
  memcpy(p.hdr_prefix, hdr.data(), hdr.size());
  p.hdr_prefix_len = (uint32_t)hdr.size();

  // the first operator planned on this index leaves its traversal order behind; later
  // plans with the same operator start from it (the order is written once, by a launch
  // that runs and records order_ready under the lock, and is only read afterwards)
  mp_index_s* ixw = const_cast<mp_index_s*>(index);
  {
    std::lock_guard<std::mutex> lk(*ixw->order_mu);
    bool fill = false;
    if (!index->has_missing) {
      // a cached order is reused only in the capture state it was written in (an event
      // recorded in a graph cannot be waited for outside it, nor an eager one inside it)
      if (ixw->order_mem.ptr && ixw->order_ready && ixw->order_key == order_key && ixw->order_captured == pl->captured) {
        if ((e = cudaStreamWaitEvent(cs, ixw->order_ready, 0)) != cudaSuccess) return bail(e, "stream wait");
        p.cache_order_in = ixw->d_order_cache;
        p.cache_q_in = ixw->d_order_q;
      } else if (!ixw->order_mem.ptr && dev_alloc(ixw->order_mem, align_up(U * 4) + 16, cs) == MP_OK) {
        ixw->d_order_cache = static_cast<uint32_t*>(ixw->order_mem.ptr);
        ixw->d_order_q = reinterpret_cast<unsigned long long*>(static_cast<char*>(ixw->order_mem.ptr) + align_up(U * 4));
        p.cache_order_out = ixw->d_order_cache;
        p.cache_q_out = ixw->d_order_q;
        // an invalid count until the filling plan completes its sort
        if ((e = launch_fill(ixw->d_order_q, 0xFF, 8, cs)) != cudaSuccess) return bail(e, "fill");
        fill = true;
      }
    }
    if ((e = launch_plan(p, scratch.ptr, cs)) != cudaSuccess) return bail(e, "plan kernels");
    if (fill) {
      if ((e = cudaEventCreateWithFlags(&ixw->order_ready, cudaEventDisableTiming)) != cudaSuccess)
        return bail(e, "event");
      if ((e = cudaEventRecord(ixw->order_ready, cs)) != cudaSuccess) return bail(e, "event record");
      ixw->order_key = order_key;
      ixw->order_captured = pl->captured;
    }
  }
  if ((e = cudaFreeAsync(scratch.ptr, cs)) != cudaSuccess) return bail(e, "free scratch");
  scratch.ptr = nullptr;
  if ((e = launch_copy(pl->h_summary, pl->d_summary, 64, cs)) != cudaSuccess)
    return bail(e, "summary copy");
  if ((e = cudaEventCreateWithFlags(&pl->done, cudaEventDisableTiming)) != cudaSuccess) return bail(e, "event");
  if ((e = cudaEventRecord(pl->done, cs)) != cudaSuccess) return bail(e, "event record");
  *out = pl;
  return MP_OK;
}

}  // extern "C"

namespace {

// mp_merge and mp_merge_touched: touched_only leaves every block whose mask is empty
// unwritten (and then out may be the base itself)
mp_status merge_common(const mp_family* family, const mp_index* index, const mp_plan_t* plan, void* out_buf,
                       mp_stream stream, mp_manifest** man_out, bool touched_only) {
  NvtxScope nv(touched_only ? "mp_merge_touched" : "mp_merge");
  if (!man_out) return fail(MP_ERR_INVALID_ARG, "manifest out is NULL");
  *man_out = nullptr;
  mp_status st;
  if ((st = check_handle(index, kMagicIndex, "index")) != MP_OK) return st;
  if ((st = check_handle(plan, kMagicPlan, "plan")) != MP_OK) return st;
  if (plan->index_id != index->id) return fail(MP_ERR_MISMATCH, "plan was built from a different index");
  Geometry g;
  if ((st = build_geometry(family, g)) != MP_OK) return st;
  if (!g.same_as(index->g)) return fail(MP_ERR_MISMATCH, "family geometry differs from the index's");
  if (!out_buf || reinterpret_cast<uintptr_t>(out_buf) % 16 != 0)
    return fail(MP_ERR_INVALID_ARG, "out must be a 16-byte aligned device buffer");
  if (!is_device_ptr(out_buf)) return fail(MP_ERR_INVALID_ARG, "out must be device memory");
  const void* base;
  ExpertPtrs ex;
  if ((st = resolve_pointers(family, base, ex)) != MP_OK) return st;
  {
    const char* o0 = static_cast<const char*>(out_buf);
    const char* o1 = o0 + g.span_elems * g.elem_size;
    auto overlaps = [&](const void* q) {
      const char* a = static_cast<const char*>(q);
      return a < o1 && o0 < a + g.span_elems * g.elem_size;
    };
    if (overlaps(base) && !(touched_only && static_cast<const void*>(out_buf) == base))
      return fail(MP_ERR_INVALID_ARG, touched_only ? "out overlaps the base without being the base"
                                                   : "out overlaps the base");
    for (uint32_t i = 0; i < g.K; ++i)
      if (family->experts_location == 0 && overlaps(ex.p[i]))
        return fail(MP_ERR_INVALID_ARG, "out overlaps an expert");
  }
  cudaStream_t cs = reinterpret_cast<cudaStream_t>(stream);
  TraceScope tr(MP_TRACE_MERGE, cs);
  const bool masked = plan->op_kind == MP_OP_TIES_MASKED;
  if (masked && !index->d_unit_hist)
    return fail(MP_ERR_MISMATCH, "a TIES_MASKED merge needs an index built for TIES_MASKED");

  mp_manifest_s* mf = new (std::nothrow) mp_manifest_s();
  if (!mf) return fail(MP_ERR_OOM, "host allocation failed");
  mf->magic = kMagicManifest;
  mf->plan_id = plan->id;
  mf->device = plan->device;
  mf->K = g.K;
  mf->n_blocks = g.n_blocks;
  mf->done = nullptr;
  mf->captured = capturing(cs);
  mf->valid_done = nullptr;
  for (uint32_t i = 0; i <= kMaxK; ++i) mf->lineage[i] = (family->lineage_ids && i <= g.K) ? family->lineage_ids[i] : 0u;
  const size_t counters_bytes = (size_t)kCounterSlots * g.K * 8;
  // the counters (64 slots x K), the plan summary, the error word and the TIES_MASKED
  // threshold reads come back in one copy
  const size_t back_bytes = counters_bytes + 64 + 16 + 16;
  mf->h_realized = static_cast<unsigned long long*>(pin_get(back_bytes));
  if (!mf->h_realized) {
    delete mf;
    return fail(MP_ERR_OOM, "pinned host allocation failed");
  }
  auto release_pinned = [&]() { pin_put(mf->h_realized, back_bytes); };
  // device side: what comes back, then the merge kernel's work counter, then (TIES_MASKED)
  // the scratch of the masked threshold
  const uint64_t KG = (uint64_t)g.K * plan->n_groups;
  size_t mo = 0;
  auto mslot = [&](size_t bytes) { size_t r = mo; mo += align_up(bytes); return r; };
  const size_t m_coarse = mslot(KG * 256 * 8), m_fine = mslot(KG * 128 * 8), m_kth = mslot(plan->n_groups * 8);
  const size_t m_est = mslot(KG * 4), m_rank = mslot(KG * 8), m_tau = mslot(KG * 4);
  const size_t scratch_off = align_up(back_bytes + 16);
  if ((st = dev_alloc(mf->mem, scratch_off + (masked ? mo : 0), cs)) != MP_OK) {
    release_pinned();
    delete mf;
    return st;
  }
  mf->d_realized = static_cast<unsigned long long*>(mf->mem.ptr);
  uint64_t* d_sum_copy = reinterpret_cast<uint64_t*>(static_cast<char*>(mf->mem.ptr) + counters_bytes);
  mf->d_err = reinterpret_cast<uint32_t*>(static_cast<char*>(mf->mem.ptr) + counters_bytes + 64);
  auto bail = [&](cudaError_t err, const char* what) {
    mp_status r = cuda_fail(err, what);
    cudaStreamSynchronize(cs);
    dev_free(mf->mem);
    release_pinned();
    if (mf->done) cudaEventDestroy(mf->done);
    delete mf;
    return r;
  };
  cudaError_t e;
  if ((e = stream_wait(cs, index->done, index->captured, mf->captured)) != cudaSuccess) return bail(e, "stream wait");
  if ((e = stream_wait(cs, plan->done, plan->captured, mf->captured)) != cudaSuccess) return bail(e, "stream wait");
  if ((e = launch_fill(mf->mem.ptr, 0, back_bytes, cs)) != cudaSuccess) return bail(e, "fill");
  uint32_t* masked_tau = nullptr;
  if (masked) {
    // TIES after masking: the threshold of the zero-completed masked deltas of this plan
    char* sm = static_cast<char*>(mf->mem.ptr) + scratch_off;
    std::vector<unsigned long long> kth(plan->n_groups, 0);
    {
      std::vector<uint64_t> gnumel(plan->n_groups, 0);
      for (uint32_t t = 0; t < g.n_tensors; ++t) gnumel[plan->trim_scope == 0 ? t : 0] += g.t_numel[t];
      for (uint32_t q = 0; q < plan->n_groups; ++q)
        kth[q] = (unsigned long long)floor((double)plan->density * (double)gnumel[q]);
    }
    if ((e = cudaMemsetAsync(sm, 0, m_kth, cs)) != cudaSuccess) return bail(e, "memset");  // coarse + fine
    if ((e = cudaMemcpyAsync(sm + m_kth, kth.data(), plan->n_groups * 8, cudaMemcpyHostToDevice, cs)) != cudaSuccess)
      return bail(e, "k copy");
    IndexLaunch q;
    memset(&q, 0, sizeof(q));
    q.dtype = g.dtype;
    q.K = g.K;
    q.n_blocks = g.n_blocks;
    q.n_groups = plan->n_groups;
    q.base = base;
    q.experts = ex;
    q.blk_off = index->d_blk_off;
    q.blk_len = index->d_blk_len;
    q.blk_group = index->d_blk_group;
    q.norm = index->d_norm;
    q.maxabs = index->d_maxabs;
    q.nnz = index->d_nnz;
    q.err = mf->d_err;
    q.coarse = (unsigned long long*)(sm + m_coarse);
    q.fine = (unsigned long long*)(sm + m_fine);
    q.kth = (const unsigned long long*)(sm + m_kth);
    q.estar = (uint32_t*)(sm + m_est);
    q.rank = (unsigned long long*)(sm + m_rank);
    q.tau = masked_tau = (uint32_t*)(sm + m_tau);
    q.unit_hist = index->d_unit_hist;
    q.mask = plan->d_mask;
    q.thr_reads = reinterpret_cast<unsigned long long*>(static_cast<char*>(mf->mem.ptr) + counters_bytes + 80);
    q.b_begin = 0;
    q.b_end = g.n_blocks;
    q.expert_origin = 0;
    q.ext = Extents{g.span_elems, g.span_elems};
    q.wait_limit = g_stall_rounds.load(std::memory_order_relaxed);
    q.stall = q.wait_limit ? 1u : 0u;
    if ((e = launch_ties_masked(q, cs)) != cudaSuccess) return bail(e, "masked TIES threshold");
  }

  MergeLaunch p;
  memset(&p, 0, sizeof(p));
  p.dtype = g.dtype;
  p.op_kind = masked ? MP_OP_TIES : plan->op_kind;  // TIES with the plan's threshold
  p.K = g.K;
  p.n_blocks = g.n_blocks;
  p.block_elems = g.block_elems;
  p.n_groups = plan->n_groups;
  p.base = base;
  p.experts = ex;
  p.out = out_buf;
  p.blk_off = index->d_blk_off;
  p.blk_len = index->d_blk_len;
  p.blk_group = index->d_blk_group;
  p.mask = plan->d_mask;
  p.tau = masked ? masked_tau : index->d_tau;
  p.nnz = index->d_nnz;
  for (uint32_t i = 0; i < kMaxK; ++i) p.alpha[i] = plan->alpha[i];
  p.lambda = plan->lambda;
  p.sigma = plan->drop_p < 1.0 ? (float)(1.0 / (1.0 - plan->drop_p)) : 0.0f;
  {
    double t = floor(plan->drop_p * 65536.0);
    p.dare_T = !(t > 0.0) ? 0u : (t > 65536.0 ? 65536u : (uint32_t)t);
    p.dare_T16 = (p.dare_T > 65535u ? 65535u : p.dare_T) << 16;
  }
  p.seed = plan->seed;
  for (int r = 0; r < 10; ++r) {
    p.dare_rk[r][0] = (uint32_t)plan->seed + (uint32_t)r * 0x9E3779B9u;
    p.dare_rk[r][1] = (uint32_t)(plan->seed >> 32) + (uint32_t)r * 0xBB67AE85u;
  }
  p.realized = mf->d_realized;
  p.work = reinterpret_cast<unsigned long long*>(static_cast<char*>(mf->mem.ptr) + back_bytes);
  p.err = mf->d_err;
  p.b_begin = 0;
  p.b_end = g.n_blocks;
  p.expert_origin = 0;
  p.ext = Extents{g.span_elems, g.span_elems};
  p.touched_only = touched_only ? 1u : 0u;
  p.wait_limit = g_stall_rounds.load(std::memory_order_relaxed);
  p.stall = p.wait_limit ? 1u : 0u;
  if (family->experts_location == 0) {
    if ((e = launch_merge(p, cs)) != cudaSuccess) return bail(e, "merge kernels");
  } else {
    if (index->h_blk_off.size() != g.n_blocks)
      return bail(cudaErrorInvalidValue, "an index of a host-resident pool is needed for a host-pool merge");
    if ((e = merge_host_pool(p, index, cs)) != cudaSuccess) return bail(e, "merge (host pool)");
  }
  if ((e = launch_copy(d_sum_copy, plan->d_summary, 64, cs)) != cudaSuccess)
    return bail(e, "summary copy");
  if ((e = launch_copy(mf->h_realized, mf->mem.ptr, back_bytes, cs)) != cudaSuccess)
    return bail(e, "manifest copy");
  if ((e = cudaEventCreateWithFlags(&mf->done, cudaEventDisableTiming)) != cudaSuccess) return bail(e, "event");
  if ((e = cudaEventRecord(mf->done, cs)) != cudaSuccess) return bail(e, "event record");
  *man_out = mf;
  return MP_OK;
}

}  // namespace

extern "C" {

mp_status mp_merge(const mp_family* family, const mp_index* index, const mp_plan_t* plan, void* out_buf,
                   mp_stream stream, mp_manifest** man_out) {
  return merge_common(family, index, plan, out_buf, stream, man_out, false);
}

mp_status mp_merge_touched(const mp_family* family, const mp_index* index, const mp_plan_t* plan, void* out_buf,
                           mp_stream stream, mp_manifest** man_out) {
  return merge_common(family, index, plan, out_buf, stream, man_out, true);
}

void mp_free(void* handle) {
  if (!handle) return;
  uint32_t magic = *static_cast<uint32_t*>(handle);
  if (magic == kMagicIndex) {
    mp_index_s* ix = static_cast<mp_index_s*>(handle);
    wait_handle(ix->done, ix->captured);
    if (ix->done) cudaEventDestroy(ix->done);
    if (ix->order_ready) {
      wait_handle(ix->order_ready, ix->order_captured);
      cudaEventDestroy(ix->order_ready);
    }
    dev_free(ix->hash_mem);
    dev_free(ix->order_mem);
    dev_free(ix->mem);
    release_pinned(ix);
    delete ix->order_mu;
    ix->magic = 0;
    delete ix;
  } else if (magic == kMagicPlan) {
    mp_plan_s* pl = static_cast<mp_plan_s*>(handle);
    wait_handle(pl->done, pl->captured);
    if (pl->done) cudaEventDestroy(pl->done);
    dev_free(pl->mem);
    pin_put(pl->h_summary, 64);
    pl->magic = 0;
    delete pl;
  } else if (magic == kMagicManifest) {
    mp_manifest_s* mf = static_cast<mp_manifest_s*>(handle);
    wait_handle(mf->done, mf->captured);
    if (mf->done) cudaEventDestroy(mf->done);
    if (mf->valid_done) cudaEventSynchronize(mf->valid_done), cudaEventDestroy(mf->valid_done);
    dev_free(mf->valid_mem);
    dev_free(mf->mem);
    pin_put(mf->h_realized, (size_t)kCounterSlots * mf->K * 8 + 64 + 16 + 16);
    mf->magic = 0;
    delete mf;
  }
}

mp_status mp_index_shape(const mp_index* index, uint64_t* n_blocks, uint64_t* n_units, uint32_t* n_groups) {
  mp_status st;
  if ((st = check_handle(index, kMagicIndex, "index")) != MP_OK) return st;
  if (n_blocks) *n_blocks = index->g.n_blocks;
  if (n_units) *n_units = index->g.n_blocks * index->g.K;
  if (n_groups) *n_groups = index->n_groups;
  return MP_OK;
}

mp_status mp_index_stats(const mp_index* index, float* norm, float* maxabs, uint32_t* nnz, uint32_t* tau) {
  mp_status st;
  if ((st = check_handle(index, kMagicIndex, "index")) != MP_OK) return st;
  cudaError_t e;
  if ((e = wait_handle(index->done, index->captured)) != cudaSuccess) return cuda_fail(e, "index work");
  const uint64_t U = index->g.n_blocks * index->g.K;
  if (norm && (e = cudaMemcpy(norm, index->d_norm, U * 4, cudaMemcpyDeviceToHost)) != cudaSuccess)
    return cuda_fail(e, "copy");
  if (maxabs && (e = cudaMemcpy(maxabs, index->d_maxabs, U * 4, cudaMemcpyDeviceToHost)) != cudaSuccess)
    return cuda_fail(e, "copy");
  if (nnz && (e = cudaMemcpy(nnz, index->d_nnz, U * 4, cudaMemcpyDeviceToHost)) != cudaSuccess)
    return cuda_fail(e, "copy");
  if (tau && (e = cudaMemcpy(tau, index->d_tau, (size_t)index->g.K * index->n_groups * 4,
                             cudaMemcpyDeviceToHost)) != cudaSuccess)
    return cuda_fail(e, "copy");
  uint32_t err = 0;
  if ((e = cudaMemcpy(&err, index->d_err, 4, cudaMemcpyDeviceToHost)) != cudaSuccess) return cuda_fail(e, "copy");
  if (err & kErrNonfinite) return fail(MP_ERR_NONFINITE, "a delta in the family is NaN or infinite");
  if (err & kErrTimeout) return fail(MP_ERR_TIMEOUT, "a bounded device wait in the index gave up");
  if (err & kErrBounds) return fail(MP_ERR_CUDA, "a bounds check of the checked build failed in the index kernels");
  if (err) return fail(MP_ERR_CUDA, "an internal check of the index kernels failed");
  return MP_OK;
}

mp_status mp_plan_info(const mp_plan_t* plan, uint64_t* planned_bytes, uint64_t* n_selected, uint64_t* n_candidates,
                       uint64_t* digest, uint32_t* mask, uint32_t* order) {
  mp_status st;
  if ((st = check_handle(plan, kMagicPlan, "plan")) != MP_OK) return st;
  cudaError_t e;
  if ((e = wait_handle(plan->done, plan->captured)) != cudaSuccess) return cuda_fail(e, "plan work");
  const uint64_t* s = plan->h_summary;
  if (planned_bytes) *planned_bytes = s[0];
  if (n_selected) *n_selected = s[1];
  if (n_candidates) *n_candidates = s[2];
  if (digest) *digest = s[4];
  if (mask && (e = cudaMemcpy(mask, plan->d_mask, plan->g.n_blocks * 4, cudaMemcpyDeviceToHost)) != cudaSuccess)
    return cuda_fail(e, "copy");
  if (order && s[2] && (e = cudaMemcpy(order, plan->d_order, s[2] * 4, cudaMemcpyDeviceToHost)) != cudaSuccess)
    return cuda_fail(e, "copy");
  if (s[6] & kErrNonfinite) return fail(MP_ERR_NONFINITE, "the index saw a NaN or infinite delta");
  if (s[6] & kErrMissing) return fail(MP_ERR_UNSUPPORTED, "a catalog entry without statistics and no tensor map");
  if (s[6] & kErrTimeout) return fail(MP_ERR_TIMEOUT, "a bounded device wait in the index gave up");
  if (s[6] & kErrBounds) return fail(MP_ERR_CUDA, "a bounds check of the checked build failed in the index kernels");
  if (s[6]) return fail(MP_ERR_CUDA, "an internal check of the index or plan kernels failed");
  if (s[0] > plan->budget) return fail(MP_ERR_BUDGET, "planned bytes exceed the budget");
  return MP_OK;
}

mp_status mp_manifest_info(const mp_manifest* man, uint64_t* realized_per_expert, uint64_t* realized_total,
                           uint64_t* touched_blocks, uint64_t* digest) {
  mp_status st;
  if ((st = check_handle(man, kMagicManifest, "manifest")) != MP_OK) return st;
  cudaError_t e;
  if ((e = wait_handle(man->done, man->captured)) != cudaSuccess) return cuda_fail(e, "merge work");
  const unsigned long long* c = man->h_realized;
  const uint64_t* s = reinterpret_cast<const uint64_t*>(c + (size_t)kCounterSlots * man->K);
  const uint32_t err = *reinterpret_cast<const uint32_t*>(s + 8);
  uint64_t tot = 0;
  for (uint32_t i = 0; i < man->K; ++i) {
    uint64_t r = 0;
    for (int k = 0; k < kCounterSlots; ++k) r += c[(size_t)k * man->K + i];
    if (realized_per_expert) realized_per_expert[i] = r;
    tot += r;
  }
  if (realized_total) *realized_total = tot;
  if (touched_blocks) *touched_blocks = s[5];
  if (digest) *digest = s[4];
  if (err & kErrTimeout) return fail(MP_ERR_TIMEOUT, "a bounded device wait in the merge gave up");
  if (err & kErrBounds) return fail(MP_ERR_CUDA, "a bounds check of the checked build failed in the merge kernels");
  if (err) return fail(MP_ERR_CUDA, "merge kernels reported an error");
  if (tot > s[0]) return fail(MP_ERR_BUDGET, "realized expert reads exceed the planned bytes");
  return MP_OK;
}

mp_status mp_index_hashes(const mp_family* family, mp_index* index, mp_stream stream) {
  mp_status st;
  if ((st = check_handle(index, kMagicIndex, "index")) != MP_OK) return st;
  Geometry g;
  if ((st = build_geometry(family, g)) != MP_OK) return st;
  if (!g.same_as(index->g)) return fail(MP_ERR_MISMATCH, "family geometry differs from the index's");
  const void* base;
  ExpertPtrs ex;
  if ((st = resolve_pointers(family, base, ex)) != MP_OK) return st;
  cudaStream_t cs = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e;
  // after whatever built the index; the index's event then covers the hashes too
  if (index->done && (e = cudaStreamWaitEvent(cs, index->done, 0)) != cudaSuccess) return cuda_fail(e, "stream wait");
  if ((st = alloc_hashes(index, cs)) != MP_OK) return st;
  HashLaunch p;
  memset(&p, 0, sizeof(p));
  p.K = g.K;
  p.elem_size = g.elem_size;
  p.n_blocks = g.n_blocks;
  p.blk_off = index->d_blk_off;
  p.blk_len = index->d_blk_len;
  p.base = base;
  p.experts = ex;
  p.base_hash = index->d_base_hash;
  p.expert_hash = index->d_expert_hash;
  p.ext = Extents{g.span_elems, g.span_elems};
  p.err = index->d_err;
  if ((e = launch_hash(p, cs)) != cudaSuccess) return cuda_fail(e, "hash kernel");
  if ((e = cudaEventRecord(index->done, cs)) != cudaSuccess) return cuda_fail(e, "event record");
  return MP_OK;
}

mp_status mp_index_hash_values(const mp_index* index, uint64_t* base_hash, uint64_t* expert_hash) {
  mp_status st;
  if ((st = check_handle(index, kMagicIndex, "index")) != MP_OK) return st;
  if (!index->hash_mem.ptr) return fail(MP_ERR_INVALID_ARG, "the index holds no block hashes (mp_index_hashes)");
  cudaError_t e;
  if ((e = wait_handle(index->done, index->captured)) != cudaSuccess) return cuda_fail(e, "index work");
  const uint64_t nb = index->g.n_blocks;
  if (base_hash && (e = cudaMemcpy(base_hash, index->d_base_hash, nb * 8, cudaMemcpyDeviceToHost)) != cudaSuccess)
    return cuda_fail(e, "copy");
  if (expert_hash && (e = cudaMemcpy(expert_hash, index->d_expert_hash, nb * index->g.K * 8,
                                     cudaMemcpyDeviceToHost)) != cudaSuccess)
    return cuda_fail(e, "copy");
  return MP_OK;
}

mp_status mp_manifest_validate(const mp_family* family, const mp_index* index, const mp_plan_t* plan, const void* out,
                               mp_stream stream, mp_manifest* man) {
  mp_status st;
  if ((st = check_handle(index, kMagicIndex, "index")) != MP_OK) return st;
  if ((st = check_handle(plan, kMagicPlan, "plan")) != MP_OK) return st;
  if ((st = check_handle(man, kMagicManifest, "manifest")) != MP_OK) return st;
  if (plan->index_id != index->id || man->plan_id != plan->id)
    return fail(MP_ERR_MISMATCH, "index, plan and manifest do not belong together");
  if (!index->hash_mem.ptr)
    return fail(MP_ERR_UNSUPPORTED, "the index holds no block hashes to validate against (mp_index_hashes)");
  Geometry g;
  if ((st = build_geometry(family, g)) != MP_OK) return st;
  if (!g.same_as(index->g)) return fail(MP_ERR_MISMATCH, "family geometry differs from the index's");
  if (!out || reinterpret_cast<uintptr_t>(out) % 16 != 0 || !is_device_ptr(out))
    return fail(MP_ERR_INVALID_ARG, "out must be the 16-byte aligned device buffer the merge wrote");
  const void* base;
  ExpertPtrs ex;
  if ((st = resolve_pointers(family, base, ex)) != MP_OK) return st;
  cudaStream_t cs = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e;
  if (!man->valid_mem.ptr) {
    if ((st = dev_alloc(man->valid_mem, 32 + (size_t)g.n_blocks * 8, cs)) != MP_OK) return st;
    man->d_vresult = static_cast<unsigned long long*>(man->valid_mem.ptr);
    man->d_out_hash = man->d_vresult + 4;
  }
  // after the merge (its output) and the index's own work (the hashes, perhaps added later)
  if ((e = cudaStreamWaitEvent(cs, man->done, 0)) != cudaSuccess) return cuda_fail(e, "stream wait");
  if ((e = cudaStreamWaitEvent(cs, index->done, 0)) != cudaSuccess) return cuda_fail(e, "stream wait");
  if ((e = cudaMemsetAsync(man->d_vresult, 0, 16, cs)) != cudaSuccess) return cuda_fail(e, "memset");
  if ((e = cudaMemsetAsync(man->d_vresult + 2, 0xFF, 8, cs)) != cudaSuccess) return cuda_fail(e, "memset");
  HashLaunch p;
  memset(&p, 0, sizeof(p));
  p.K = g.K;
  p.elem_size = g.elem_size;
  p.n_blocks = g.n_blocks;
  p.blk_off = index->d_blk_off;
  p.blk_len = index->d_blk_len;
  p.base = base;
  p.experts = ex;
  p.out = out;
  p.mask = plan->d_mask;
  p.validate = 1;
  p.base_hash = index->d_base_hash;
  p.expert_hash = index->d_expert_hash;
  p.out_hash = man->d_out_hash;
  p.result = man->d_vresult;
  p.ext = Extents{g.span_elems, g.span_elems};
  p.err = man->d_err;
  if ((e = launch_hash(p, cs)) != cudaSuccess) return cuda_fail(e, "hash kernel");
  if (!man->valid_done && (e = cudaEventCreateWithFlags(&man->valid_done, cudaEventDisableTiming)) != cudaSuccess)
    return cuda_fail(e, "event");
  if ((e = cudaEventRecord(man->valid_done, cs)) != cudaSuccess) return cuda_fail(e, "event record");
  return MP_OK;
}

mp_status mp_manifest_validation(const mp_manifest* man, uint64_t* checked, uint64_t* mismatched, uint64_t* out_hash) {
  mp_status st;
  if ((st = check_handle(man, kMagicManifest, "manifest")) != MP_OK) return st;
  if (!man->valid_done) return fail(MP_ERR_INVALID_ARG, "the manifest was not validated (mp_manifest_validate)");
  cudaError_t e;
  if ((e = cudaEventSynchronize(man->valid_done)) != cudaSuccess) return cuda_fail(e, "validation work");
  unsigned long long r[3];
  if ((e = cudaMemcpy(r, man->d_vresult, sizeof(r), cudaMemcpyDeviceToHost)) != cudaSuccess) return cuda_fail(e, "copy");
  uint32_t err = 0;
  if ((e = cudaMemcpy(&err, man->d_err, 4, cudaMemcpyDeviceToHost)) != cudaSuccess) return cuda_fail(e, "copy");
  if (err & kErrBounds) return fail(MP_ERR_CUDA, "a bounds check of the checked build failed");
  if (out_hash && (e = cudaMemcpy(out_hash, man->d_out_hash, man->n_blocks * 8, cudaMemcpyDeviceToHost)) != cudaSuccess)
    return cuda_fail(e, "copy");
  if (checked) *checked = r[0];
  if (mismatched) *mismatched = r[1];
  if (r[1]) {
    const uint64_t k = r[2] / man->n_blocks, b = r[2] % man->n_blocks;
    return fail(MP_ERR_MISMATCH, std::to_string(r[1]) + " block(s) read by the merge differ from the catalog; first: " +
                                     (k == 0 ? std::string("base") : "expert " + std::to_string(k - 1)) + " block " +
                                     std::to_string(b));
  }
  return MP_OK;
}

mp_status mp_manifest_threshold_reads(const mp_manifest* man, uint64_t* bytes) {
  mp_status st;
  if ((st = check_handle(man, kMagicManifest, "manifest")) != MP_OK) return st;
  if (!bytes) return fail(MP_ERR_INVALID_ARG, "bytes is NULL");
  cudaError_t e;
  if ((e = wait_handle(man->done, man->captured)) != cudaSuccess) return cuda_fail(e, "merge work");
  *bytes = man->h_realized[(size_t)kCounterSlots * man->K + 10];
  return MP_OK;
}

mp_status mp_manifest_lineage(const mp_manifest* man, uint64_t* ids) {
  mp_status st;
  if ((st = check_handle(man, kMagicManifest, "manifest")) != MP_OK) return st;
  if (!ids) return fail(MP_ERR_INVALID_ARG, "ids is NULL");
  for (uint32_t i = 0; i <= man->K; ++i) ids[i] = man->lineage[i];
  return MP_OK;
}

}  // extern "C"
