// Alg. 2 ExecuteMerge on the device: M_A[t,b] = M_0[t,b] + Psi_op(A_{.,t,b}, Delta_{.,t,b})
// (Eq. 4) for every block, reading only the experts the access mask selects.
//
// Pipeline (one persistent CTA pair per SM, 256 consumer threads + 1 producer warp):
//  * work unit = one chunk of 8 KiB of a block (4096 bf16 / 2048 fp32 elements); chunks
//    are handed out dynamically through a global counter, GRAB at a time;
//  * the producer thread walks each chunk's fills — the base chunk, then every selected
//    expert's chunk in ascending expert order — and streams each fill into the next slot
//    of a ring of NS shared-memory slots with one cp.async.bulk (TMA 1-D bulk copy),
//    completing on the slot's "full" mbarrier; it writes the slot's metadata (chunk,
//    which checkpoint, offset, length, mask) before arming the barrier;
//  * consumers take the slots in the same order: the base fill loads M_0 into registers,
//    each expert fill folds Delta_i into fp32 accumulators, the last fill of a chunk
//    writes the output with 16-byte streaming stores; each warp releases a slot on its
//    "empty" mbarrier as soon as it has read it;
//  * the bytes in flight are the ring (NS x 8 KiB per CTA), independent of registers and
//    of how many experts a block selects.
// Per element, in the fixed ascending expert order:
//   AVG/TA: acc = fma(alpha_i, delta_i, acc)                          out = M_0 + acc
//   DARE:   delta_i kept by a Philox word >= T, scaled by sigma; then as AVG
//   TIES:   trimmed by tau_i; S, P, N, counts;  m = P/c+ | N/c- | 0;   out = fma(lambda, m, M_0)
// An omitted expert contributes exactly zero to every accumulator, so skipping it equals
// reading a zero-completed tuple (App. A.1) and it is never dereferenced.
// Every mbarrier wait is bounded: on expiry the CTA records kErrTimeout, stops, waits
// (bounded) for its own copies in flight and returns.
#include <cuda_bf16.h>

#include "mp_internal.cuh"
#include "philox.cuh"
#include "tma.cuh"

namespace mp {
namespace {

constexpr int kConsumers = 256;
constexpr int kThreads = kConsumers + 32;  // + one producer warp
constexpr uint32_t kRingBytes = 98304;     // slot ring per CTA (96 KiB; two CTAs per SM)
constexpr uint32_t kGrab = 4;              // chunks taken per counter increment
constexpr uint32_t kEnd = 0xFFFFFFFFu;

enum { OP_ADD = 0, OP_TIES = 1, OP_DARE = 2 };

// slot geometry per operator: TIES keeps five fp32 values per element in flight, so its
// chunks are half as long (one 16-byte vector per consumer thread, no register spills)
template <int OPC>
struct Geo {
  static constexpr uint32_t kSlotBytes = OPC == OP_TIES ? 4096u : 8192u;  // one chunk of one checkpoint
  static constexpr int kSlots = (int)(kRingBytes / kSlotBytes);
};

struct SlotMeta {
  uint64_t off;   // element offset of the chunk in the flat buffers
  uint32_t q;     // chunk id, or kEnd
  uint32_t which; // 0 = base, 1 + i = expert i
  uint32_t n;     // elements in the chunk
  uint32_t m;     // the block's access mask
  uint32_t grp;   // the block's trim group
  uint32_t tau;   // TIES threshold of this (expert, trim group)
};

template <int NS, uint32_t SB>
struct __align__(128) Smem {
  uint8_t slot[NS][SB];
  SlotMeta meta[NS];
  uint64_t full[NS];
  uint64_t empty[NS];
  unsigned long long realized[kMaxK];
  int abort;
};

template <bool BF16>
__device__ __forceinline__ void unpack(const uint4 r, float* x) {
  if constexpr (BF16) {
    x[0] = __uint_as_float(r.x << 16);
    x[1] = __uint_as_float(r.x & 0xFFFF0000u);
    x[2] = __uint_as_float(r.y << 16);
    x[3] = __uint_as_float(r.y & 0xFFFF0000u);
    x[4] = __uint_as_float(r.z << 16);
    x[5] = __uint_as_float(r.z & 0xFFFF0000u);
    x[6] = __uint_as_float(r.w << 16);
    x[7] = __uint_as_float(r.w & 0xFFFF0000u);
  } else {
    x[0] = __uint_as_float(r.x);
    x[1] = __uint_as_float(r.y);
    x[2] = __uint_as_float(r.z);
    x[3] = __uint_as_float(r.w);
  }
}

// vector v of a fill: from the slot when inside the bulk-copied bytes, else (the ragged
// tail of a tensor, < 16 bytes) straight from global memory; zeros past the chunk
template <bool BF16>
__device__ __forceinline__ void read_vec(const uint8_t* slot, const void* gsrc, uint64_t off, uint32_t k0,
                                         uint32_t n, uint32_t n_tma, float* x) {
  constexpr uint32_t V = BF16 ? 8u : 4u;
  if (k0 + V <= n_tma) {
    unpack<BF16>(*reinterpret_cast<const uint4*>(slot + k0 * (BF16 ? 2u : 4u)), x);
    return;
  }
#pragma unroll
  for (uint32_t e = 0; e < V; ++e) {
    float v = 0.0f;
    if (k0 + e < n) {
      if constexpr (BF16) v = __uint_as_float((uint32_t)(static_cast<const uint16_t*>(gsrc)[off + k0 + e]) << 16);
      else v = static_cast<const float*>(gsrc)[off + k0 + e];
    }
    x[e] = v;
  }
}

template <bool BF16>
__device__ __forceinline__ void store_vec(void* ptr, uint64_t elem, uint32_t navail, const float* y) {
  constexpr uint32_t V = BF16 ? 8u : 4u;
  if constexpr (BF16) {
    uint32_t h[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) h[e] = __bfloat16_as_ushort(__float2bfloat16_rn(y[e]));
    if (navail >= V) {
      uint4 w = make_uint4(h[0] | (h[1] << 16), h[2] | (h[3] << 16), h[4] | (h[5] << 16), h[6] | (h[7] << 16));
      __stcs(reinterpret_cast<uint4*>(static_cast<char*>(ptr) + elem * 2u), w);
    } else {
      for (uint32_t e = 0; e < navail; ++e) static_cast<uint16_t*>(ptr)[elem + e] = (uint16_t)h[e];
    }
  } else {
    if (navail >= V) {
      __stcs(reinterpret_cast<float4*>(static_cast<char*>(ptr) + elem * 4u), make_float4(y[0], y[1], y[2], y[3]));
    } else {
      for (uint32_t e = 0; e < navail; ++e) static_cast<float*>(ptr)[elem + e] = y[e];
    }
  }
}

template <bool BF16, int OPC>
__global__ void __launch_bounds__(kThreads, 2)
    merge_tma_kernel(const MergeLaunch p, uint32_t cpb, uint64_t n_chunks, unsigned long long* work) {
  constexpr uint32_t ES = BF16 ? 2u : 4u;
  constexpr uint32_t SB = Geo<OPC>::kSlotBytes;
  constexpr int kSlots = Geo<OPC>::kSlots;
  constexpr uint32_t CH = SB / ES;  // elements per chunk
  constexpr int V = BF16 ? 8 : 4;
  constexpr int VPT = (int)(CH / (kConsumers * V));  // vectors per consumer thread per chunk
  static_assert(CH == (uint32_t)(kConsumers * VPT * V), "chunk geometry");
  extern __shared__ __align__(128) uint8_t smem_raw[];
  Smem<kSlots, SB>& S = *reinterpret_cast<Smem<kSlots, SB>*>(smem_raw);
  const uint32_t tid = threadIdx.x, warp = tid >> 5, lane = tid & 31u;
  volatile int* abort_flag = &S.abort;

  if (tid == 0) {
    for (int s = 0; s < kSlots; ++s) {
      mbar_init(&S.full[s], 1);
      mbar_init(&S.empty[s], kConsumers / 32);
    }
    S.abort = 0;
    mbar_fence_init();
  }
  if (tid < (uint32_t)kMaxK) S.realized[tid] = 0;
  __syncthreads();

  if (warp == kConsumers / 32) {
    // ---------------- producer ----------------
    if (lane == 0) {
      uint32_t fill = 0;
      bool ok = true;
      auto produce = [&](uint32_t q, uint32_t which, uint64_t off, uint32_t n, uint32_t m, uint32_t grp,
                         const char* src_row, uint32_t bytes) -> bool {
        const uint32_t s = fill % kSlots, r = fill / kSlots;
        if (r > 0 && !mbar_wait(&S.empty[s], (r - 1) & 1u, abort_flag)) return false;
        S.meta[s].off = off;
        S.meta[s].q = q;
        S.meta[s].which = which;
        S.meta[s].n = n;
        S.meta[s].m = m;
        S.meta[s].grp = grp;
        S.meta[s].tau = (OPC == OP_TIES && which > 0) ? p.tau[(uint64_t)(which - 1) * p.n_groups + grp] : 0u;
        mbar_arrive_expect_tx(&S.full[s], bytes);
        if (bytes) tma_load_1d(S.slot[s], src_row, bytes, &S.full[s]);
        ++fill;
        return true;
      };
      while (ok) {
        const unsigned long long q0 = atomicAdd(work, (unsigned long long)kGrab);
        if (q0 >= n_chunks) break;
        const unsigned long long q1 = min(q0 + kGrab, (unsigned long long)n_chunks);
        for (unsigned long long q = q0; q < q1 && ok; ++q) {
          const uint64_t b = p.b_begin + q / cpb;
          const uint32_t start = (uint32_t)(q % cpb) * CH;
          const uint32_t len = p.blk_len[b];
          if (start >= len) continue;
          const uint32_t n = min(CH, len - start);
          const uint64_t off = p.blk_off[b] + start;
          const uint32_t m = p.mask[b];
          const uint32_t grp = OPC == OP_TIES ? p.blk_group[b] : 0u;
          const uint32_t bytes = (n * ES) & ~15u;
          ok = produce((uint32_t)q, 0, off, n, m, grp, static_cast<const char*>(p.base) + off * ES, bytes);
          for (uint32_t mm = m; ok && mm; mm &= mm - 1) {
            const uint32_t i = __ffs(mm) - 1;
            ok = produce((uint32_t)q, 1 + i, off, n, m, grp,
                         static_cast<const char*>(p.experts.p[i]) + (off - p.expert_origin) * ES, bytes);
            S.realized[i] += (unsigned long long)n * ES;
          }
        }
      }
      if (ok) ok = produce(kEnd, 0, 0, 0, 0, 0, nullptr, 0);
      if (!ok) {
        atomicOr(p.err, kErrTimeout);
        S.abort = 1;
      }
      // drain: the last fill of every slot must have landed before the CTA may exit
      for (uint32_t s = 0; s < (uint32_t)kSlots && s < fill; ++s) {
        const uint32_t last = fill - 1 - ((fill - 1 + kSlots - s) % kSlots);
        mbar_wait_drain(&S.full[s], (last / kSlots) & 1u);
      }
      for (uint32_t i = 0; i < p.K; ++i)
        if (S.realized[i])
          atomicAdd(p.realized + (uint64_t)(blockIdx.x % kCounterSlots) * p.K + i, S.realized[i]);
    }
    return;
  }

  // ---------------- consumers ----------------
  float x0[VPT][V], acc[VPT][V], Sg[VPT][V], Pp[VPT][V], Nn[VPT][V];
  uint32_t cnt[VPT][V];  // TIES: positive count | negative count << 16
  uint64_t off = 0;
  uint32_t n = 0, n_tma = 0, remaining = 0;
  for (uint32_t fill = 0;; ++fill) {
    const uint32_t s = fill % kSlots, r = fill / kSlots;
    if (!warp_wait(&S.full[s], r & 1u, abort_flag)) {
      atomicOr(p.err, kErrTimeout);
      S.abort = 1;
      break;
    }
    const SlotMeta mt = S.meta[s];
    if (mt.q == kEnd) break;
    const uint8_t* slot = S.slot[s];
    if (mt.which == 0) {
      off = mt.off;
      n = mt.n;
      n_tma = ((n * ES) & ~15u) / ES;
      remaining = __popc(mt.m);
#pragma unroll
      for (int u = 0; u < VPT; ++u) {
        const uint32_t k0 = (tid + (uint32_t)u * kConsumers) * V;
        read_vec<BF16>(slot, p.base, off, k0, n, n_tma, x0[u]);
#pragma unroll
        for (int e = 0; e < V; ++e) {
          acc[u][e] = 0.0f;
          Sg[u][e] = 0.0f;
          Pp[u][e] = 0.0f;
          Nn[u][e] = 0.0f;
          cnt[u][e] = 0u;
        }
      }
    } else {
      const uint32_t i = mt.which - 1;
      const void* src = p.experts.p[i];
      if constexpr (OPC == OP_TIES) {
        const uint32_t tau = mt.tau;
#pragma unroll
        for (int u = 0; u < VPT; ++u) {
          const uint32_t k0 = (tid + (uint32_t)u * kConsumers) * V;
          float xe[V];
          read_vec<BF16>(slot, src, off - p.expert_origin, k0, n, n_tma, xe);
#pragma unroll
          for (int e = 0; e < V; ++e) {
            const float d = __fsub_rn(xe[e], x0[u][e]);
            const uint32_t key = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(fabsf(d))) & 0x7FFFu;
            const float dh = key >= tau ? d : 0.0f;
            // branch-free tally: S, P and N are never -0, so adding +0 leaves them unchanged
            const bool pos = dh > 0.0f, neg = dh < 0.0f;
            Sg[u][e] = __fadd_rn(Sg[u][e], dh);
            Pp[u][e] = __fadd_rn(Pp[u][e], pos ? dh : 0.0f);
            Nn[u][e] = __fadd_rn(Nn[u][e], neg ? dh : 0.0f);
            cnt[u][e] += (pos ? 1u : 0u) + (neg ? 0x10000u : 0u);
          }
        }
      } else {
        const float a = p.alpha[i];
#pragma unroll
        for (int u = 0; u < VPT; ++u) {
          const uint32_t k0 = (tid + (uint32_t)u * kConsumers) * V;
          float xe[V];
          read_vec<BF16>(slot, src, off - p.expert_origin, k0, n, n_tma, xe);
          uint32_t keep = 0xFFu;
          if constexpr (OPC == OP_DARE) {
            const uint64_t j0 = off + k0;
            keep = dare_keep8(p.seed, i, j0 >> 3, p.dare_T) >> (uint32_t)(j0 & 7u);
          }
#pragma unroll
          for (int e = 0; e < V; ++e) {
            float d = __fsub_rn(xe[e], x0[u][e]);
            if constexpr (OPC == OP_DARE) d = ((keep >> e) & 1u) ? __fmul_rn(d, p.sigma) : 0.0f;
            acc[u][e] = __fmaf_rn(a, d, acc[u][e]);
          }
        }
      }
      --remaining;
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&S.empty[s]);
    if (remaining == 0) {
#pragma unroll
      for (int u = 0; u < VPT; ++u) {
        const uint32_t k0 = (tid + (uint32_t)u * kConsumers) * V;
        if (k0 >= n) continue;
        float y[V];
#pragma unroll
        for (int e = 0; e < V; ++e) {
          if constexpr (OPC == OP_TIES) {
            // one division per element: the mean of the entries whose sign was elected
            const bool pos = Sg[u][e] > 0.0f;
            const float num = pos ? Pp[u][e] : Nn[u][e];
            const uint32_t c = pos ? (cnt[u][e] & 0xFFFFu) : (cnt[u][e] >> 16);
            const float mm = Sg[u][e] != 0.0f ? __fdiv_rn(num, __uint2float_rn(c)) : 0.0f;
            y[e] = __fmaf_rn(p.lambda, mm, x0[u][e]);
          } else {
            y[e] = __fadd_rn(x0[u][e], acc[u][e]);
          }
        }
        store_vec<BF16>(p.out, off + k0, n - k0, y);
      }
    }
  }
}

template <bool BF16, int OPC>
cudaError_t launch_op(const MergeLaunch& p, cudaStream_t st) {
  const uint32_t chunk = Geo<OPC>::kSlotBytes / (BF16 ? 2u : 4u);
  const uint32_t cpb = (p.block_elems + chunk - 1) / chunk;
  const uint64_t n_chunks = (p.b_end - p.b_begin) * cpb;
  if (n_chunks == 0) return cudaSuccess;
  if (n_chunks >= 0xFFFFFFFFull) return cudaErrorInvalidValue;
  int dev = 0, sms = 0;
  cudaError_t e;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
  const size_t smem = sizeof(Smem<Geo<OPC>::kSlots, Geo<OPC>::kSlotBytes>);
  if ((e = cudaFuncSetAttribute(merge_tma_kernel<BF16, OPC>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)) !=
      cudaSuccess)
    return e;
  uint64_t grid = (uint64_t)sms * 2;
  if (grid > n_chunks) grid = n_chunks;
  if ((e = cudaMemsetAsync(p.work, 0, sizeof(unsigned long long), st)) != cudaSuccess) return e;
  merge_tma_kernel<BF16, OPC><<<(unsigned)grid, kThreads, smem, st>>>(p, cpb, n_chunks, p.work);
  count_launches(1);
  return cudaGetLastError();
}

template <bool BF16>
cudaError_t launch_dtype(const MergeLaunch& p, cudaStream_t st) {
  switch (p.op_kind) {
    case MP_OP_AVG:
    case MP_OP_TA: return launch_op<BF16, OP_ADD>(p, st);
    case MP_OP_TIES: return launch_op<BF16, OP_TIES>(p, st);
    case MP_OP_DARE: return launch_op<BF16, OP_DARE>(p, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

cudaError_t launch_merge(const MergeLaunch& p, cudaStream_t st) {
  return p.dtype == MP_BF16 ? launch_dtype<true>(p, st) : launch_dtype<false>(p, st);
}

}  // namespace mp
