// Alg. 2 ExecuteMerge on the device: M_A[t,b] = M_0[t,b] + Psi_op(A_{.,t,b}, Delta_{.,t,b})
// (Eq. 4) for every block, reading only the experts the access mask selects.
//
// Work item = (block, 16 KiB chunk of it); one CTA of 256 threads per item, each thread
// one 16-byte vector of the base and of every selected expert per step.  Experts are
// visited in ascending index in groups of 8 (their loads issued together), and each
// element folds them into fp32 accumulators in that fixed order:
//   AVG/TA: acc = fma(alpha_i, delta_i, acc)                          out = M_0 + acc
//   DARE:   delta_i kept by a Philox word >= T, scaled by sigma; then as AVG
//   TIES:   trimmed by tau_i; S, P, N, counts;  m = P/c+ | N/c- | 0;   out = fma(lambda, m, M_0)
// An omitted expert contributes exactly zero to every accumulator, so skipping it is the
// same as reading a zero-completed tuple (App. A.1) and it is never dereferenced.
#include <cuda_bf16.h>

#include "mp_internal.cuh"
#include "philox.cuh"

namespace mp {
namespace {

constexpr int kThreads = 256;
constexpr uint32_t kChunkBytes = 16384;
constexpr int kGroup = 8;

template <bool BF16>
__device__ __forceinline__ void load_vec(const void* ptr, uint64_t elem, uint32_t navail, float (&x)[BF16 ? 8 : 4]) {
  constexpr uint32_t V = BF16 ? 8u : 4u;
  if (navail >= V) {
    const uint4 r = __ldcs(reinterpret_cast<const uint4*>(static_cast<const char*>(ptr) + elem * (BF16 ? 2u : 4u)));
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
    return;
  }
#pragma unroll
  for (uint32_t e = 0; e < V; ++e) {
    float v = 0.0f;
    if (e < navail) {
      if constexpr (BF16) v = __uint_as_float((uint32_t)(static_cast<const uint16_t*>(ptr)[elem + e]) << 16);
      else v = static_cast<const float*>(ptr)[elem + e];
    }
    x[e] = v;
  }
}

template <bool BF16>
__device__ __forceinline__ void store_vec(void* ptr, uint64_t elem, uint32_t navail, const float (&y)[BF16 ? 8 : 4]) {
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

enum { OP_ADD = 0, OP_TIES = 1, OP_DARE = 2 };

template <bool BF16, int OPC, int KMAX>
__global__ void __launch_bounds__(kThreads) merge_kernel(const MergeLaunch p, uint32_t cpb, uint32_t chunk_elems) {
  constexpr int V = BF16 ? 8 : 4;
  __shared__ uint32_t s_tau[KMAX];
  const uint64_t item = blockIdx.x;
  const uint64_t b = item / cpb;
  const uint32_t start = (uint32_t)(item % cpb) * chunk_elems;
  const uint32_t len = p.blk_len[b];
  if (start >= len) return;
  const uint32_t n = min(chunk_elems, len - start);
  const uint64_t off = p.blk_off[b] + start;
  const uint32_t m = p.mask[b];
  const uint32_t K = p.K;
  if constexpr (OPC == OP_TIES) {
    const uint32_t grp = p.blk_group[b];
    for (uint32_t i = threadIdx.x; i < K; i += kThreads) s_tau[i] = p.tau[(uint64_t)i * p.n_groups + grp];
    __syncthreads();
  }
  const uint32_t nvec = (n + V - 1) / V;
  for (uint32_t v = threadIdx.x; v < nvec; v += kThreads) {
    const uint32_t k0 = v * V;
    const uint32_t navail = n - k0;
    const uint64_t j0 = off + k0;
    float x0[V];
    load_vec<BF16>(p.base, j0, navail, x0);
    float acc[V], S[V], P[V], N[V];
    uint32_t cp[V], cn[V];
#pragma unroll
    for (int e = 0; e < V; ++e) {
      acc[e] = 0.0f;
      S[e] = 0.0f;
      P[e] = 0.0f;
      N[e] = 0.0f;
      cp[e] = 0u;
      cn[e] = 0u;
    }
#pragma unroll
    for (int g0 = 0; g0 < KMAX; g0 += kGroup) {
      if ((uint32_t)g0 >= K) break;
      float xe[kGroup][V];
#pragma unroll
      for (int k = 0; k < kGroup; ++k) {
        const uint32_t i = g0 + k;
        if (i < K && ((m >> i) & 1u)) load_vec<BF16>(p.experts.p[i], j0, navail, xe[k]);
      }
#pragma unroll
      for (int k = 0; k < kGroup; ++k) {
        const uint32_t i = g0 + k;
        if (!(i < K && ((m >> i) & 1u))) continue;
        if constexpr (OPC == OP_TIES) {
          const uint32_t tau = s_tau[i];
#pragma unroll
          for (int e = 0; e < V; ++e) {
            const float d = __fsub_rn(xe[k][e], x0[e]);
            const uint32_t key = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(fabsf(d))) & 0x7FFFu;
            const float dh = key >= tau ? d : 0.0f;
            S[e] = __fadd_rn(S[e], dh);
            if (dh > 0.0f) {
              P[e] = __fadd_rn(P[e], dh);
              ++cp[e];
            } else if (dh < 0.0f) {
              N[e] = __fadd_rn(N[e], dh);
              ++cn[e];
            }
          }
        } else {
          uint32_t keep = 0xFFu;
          if constexpr (OPC == OP_DARE) {
            keep = dare_keep8(p.seed, i, j0 >> 3, p.dare_T) >> (uint32_t)(j0 & 7u);
          }
          const float a = p.alpha[i];
#pragma unroll
          for (int e = 0; e < V; ++e) {
            float d = __fsub_rn(xe[k][e], x0[e]);
            if constexpr (OPC == OP_DARE) d = ((keep >> e) & 1u) ? __fmul_rn(d, p.sigma) : 0.0f;
            acc[e] = __fmaf_rn(a, d, acc[e]);
          }
        }
      }
    }
    float y[V];
#pragma unroll
    for (int e = 0; e < V; ++e) {
      if constexpr (OPC == OP_TIES) {
        float mm = 0.0f;
        if (S[e] > 0.0f) mm = __fdiv_rn(P[e], __uint2float_rn(cp[e]));
        else if (S[e] < 0.0f) mm = __fdiv_rn(N[e], __uint2float_rn(cn[e]));
        y[e] = __fmaf_rn(p.lambda, mm, x0[e]);
      } else {
        y[e] = __fadd_rn(x0[e], acc[e]);
      }
    }
    store_vec<BF16>(p.out, j0, navail, y);
  }
  if (threadIdx.x == 0 && m) {
    const unsigned long long bytes = (unsigned long long)n * (BF16 ? 2u : 4u);
    unsigned long long* slot = p.realized + (uint64_t)(blockIdx.x % kCounterSlots) * K;
    for (uint32_t i = 0; i < K; ++i)
      if ((m >> i) & 1u) atomicAdd(slot + i, bytes);
  }
}

template <bool BF16, int OPC>
cudaError_t launch_op(const MergeLaunch& p, cudaStream_t st) {
  const uint32_t chunk = kChunkBytes / (BF16 ? 2u : 4u);
  const uint32_t cpb = (p.block_elems + chunk - 1) / chunk;
  const uint64_t grid = p.n_blocks * cpb;
  if (grid == 0) return cudaSuccess;
  if (grid > 0x7FFFFFFFull) return cudaErrorInvalidValue;
  if (p.K <= 8) merge_kernel<BF16, OPC, 8><<<(unsigned)grid, kThreads, 0, st>>>(p, cpb, chunk);
  else if (p.K <= 16) merge_kernel<BF16, OPC, 16><<<(unsigned)grid, kThreads, 0, st>>>(p, cpb, chunk);
  else merge_kernel<BF16, OPC, 32><<<(unsigned)grid, kThreads, 0, st>>>(p, cpb, chunk);
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
