// Host-resident expert pool: the gather stage of Alg. 2 (DeltaIterator materialising only
// the selected deltas, Sec. 3 "Executor").  For a range of blocks it copies exactly the
// planned (block, expert) pairs (or, with no mask, every expert block: the index pass) — read from the experts' pinned host memory through the
// host mapping, i.e. over NVLink-C2C on GB300 — into HBM staging buffers laid out like the
// flat checkpoint from element `origin` on.  The mask is read on the device, so the gather
// needs no host synchronisation; unselected expert blocks are never touched (the realized
// reads stay within the plan, Prop. 1).  One CTA per block; four 16-byte loads in flight
// per thread.
//
// The small copies and fills of the calls (block tables in, summaries and manifests out,
// zeroed counters) are kernels here too: a copy engine serves its direction in order, so a
// small cudaMemcpyAsync queued behind a caller's multi-gigabyte transfer on another stream
// would wait for all of it.  A host buffer these kernels read or write is pinned memory,
// which the device reaches through its host mapping.
#include "mp_internal.cuh"

namespace mp {
namespace {

constexpr int kThreads = 256;
constexpr int kUnroll = 4;

__global__ void __launch_bounds__(kThreads) gather_kernel(const GatherLaunch g) {
  const uint64_t b = g.b_begin + blockIdx.x;
  if (b >= g.b_end) return;
  if (g.gate && *g.gate == 0u) return;  // a gated launch with nothing to bring in
  const uint32_t all = g.K >= 32 ? 0xFFFFFFFFu : ((1u << g.K) - 1u);
  const uint32_t m = g.mask ? g.mask[b] : all;
  if (m == 0u) return;
  const uint64_t off = g.blk_off[b];
  if (kChecked && !chunk_in_bounds(b, g.b_begin, g.b_end, off, g.blk_len[b], off, g.blk_len[b], m, g.K, g.elem_size,
                                   g.origin, g.ext)) {  // uniform over the CTA
    if (threadIdx.x == 0 && g.err) atomicOr(g.err, kErrBounds);
    return;
  }
  const uint64_t bytes = (uint64_t)g.blk_len[b] * g.elem_size;
  const uint64_t nvec = bytes / 16u;
  const uint32_t tail = (uint32_t)(bytes % 16u);
  unsigned long long copied = 0;
  for (uint32_t mm = m; mm; mm &= mm - 1u) {
    const uint32_t i = __ffs(mm) - 1u;
    const char* src = static_cast<const char*>(g.src.p[i]) + off * g.elem_size;
    char* dst = static_cast<char*>(const_cast<void*>(g.dst.p[i])) + (off - g.origin) * g.elem_size;
    const uint4* s4 = reinterpret_cast<const uint4*>(src);
    uint4* d4 = reinterpret_cast<uint4*>(dst);
    for (uint64_t v = threadIdx.x; v < nvec; v += (uint64_t)kUnroll * kThreads) {
      uint4 r[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u)
        if (v + (uint64_t)u * kThreads < nvec) r[u] = s4[v + (uint64_t)u * kThreads];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u)
        if (v + (uint64_t)u * kThreads < nvec) d4[v + (uint64_t)u * kThreads] = r[u];
    }
    if (threadIdx.x < tail) dst[nvec * 16u + threadIdx.x] = src[nvec * 16u + threadIdx.x];
    copied += bytes;
  }
  if (threadIdx.x == 0 && g.gathered) atomicAdd(g.gathered, copied);
}

// small copies and fills on the caller's stream, by kernel: 16-byte vectors where both
// addresses allow, bytes at the ends
__global__ void __launch_bounds__(kThreads) copy_kernel(char* dst, const char* src, size_t bytes) {
  const size_t tid = (size_t)blockIdx.x * kThreads + threadIdx.x, nt = (size_t)gridDim.x * kThreads;
  if (((reinterpret_cast<uintptr_t>(dst) | reinterpret_cast<uintptr_t>(src)) & 15u) == 0) {
    const size_t nv = bytes / 16u;
    for (size_t v = tid; v < nv; v += nt) reinterpret_cast<uint4*>(dst)[v] = reinterpret_cast<const uint4*>(src)[v];
    for (size_t i = nv * 16u + tid; i < bytes; i += nt) dst[i] = src[i];
  } else {
    for (size_t i = tid; i < bytes; i += nt) dst[i] = src[i];
  }
}

__global__ void __launch_bounds__(kThreads) fill_kernel(char* dst, uint32_t v, size_t bytes) {
  const size_t tid = (size_t)blockIdx.x * kThreads + threadIdx.x, nt = (size_t)gridDim.x * kThreads;
  const uint32_t w = (v & 0xFFu) * 0x01010101u;
  if ((reinterpret_cast<uintptr_t>(dst) & 15u) == 0) {
    const size_t nv = bytes / 16u;
    for (size_t k = tid; k < nv; k += nt) reinterpret_cast<uint4*>(dst)[k] = make_uint4(w, w, w, w);
    for (size_t i = nv * 16u + tid; i < bytes; i += nt) dst[i] = (char)v;
  } else {
    for (size_t i = tid; i < bytes; i += nt) dst[i] = (char)v;
  }
}

unsigned small_grid(size_t bytes) {
  const size_t per = (size_t)kThreads * 16u * 4u;  // four vectors per thread
  const size_t g = (bytes + per - 1) / per;
  return (unsigned)(g < 1 ? 1 : (g > 1024 ? 1024 : g));
}

}  // namespace

cudaError_t launch_copy(void* dst, const void* src, size_t bytes, cudaStream_t st) {
  if (bytes == 0) return cudaSuccess;
  copy_kernel<<<small_grid(bytes), kThreads, 0, st>>>(static_cast<char*>(dst), static_cast<const char*>(src), bytes);
  count_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_fill(void* dst, uint32_t byte_value, size_t bytes, cudaStream_t st) {
  if (bytes == 0) return cudaSuccess;
  fill_kernel<<<small_grid(bytes), kThreads, 0, st>>>(static_cast<char*>(dst), byte_value, bytes);
  count_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_gather(const GatherLaunch& g, cudaStream_t st) {
  const uint64_t nb = g.b_end - g.b_begin;
  if (nb == 0) return cudaSuccess;
  if (nb > 0x7FFFFFFFull) return cudaErrorInvalidValue;
  gather_kernel<<<(unsigned)nb, kThreads, 0, st>>>(g);
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace mp
