// Catalog pass (Sec. 3 "Catalog"; the Analyze reads of Sec. 2): per-(expert, block)
// statistics of Delta = M_i - M_0 and, for TIES, the per-(expert, trim group) threshold.
//
// Mapping: one CTA of 256 threads per (block, group of up to 8 experts).  Thread l is
// lane l of the fixed summation order: it streams 16-byte vectors l, l+256, ... of the
// block (base once, each expert of the group), keeps a sequential fma chain of delta^2
// per expert, then the lanes are combined by a xor butterfly inside each warp and over
// the 8 warp sums.  That order is part of the definition of the norm (it decides the
// plan), so it must not change with tuning.
//
// TIES threshold (k-th largest 15-bit key bits(bf16(|delta|)) & 0x7FFF per trim group)
// is a two-level radix select: the index pass histograms the upper 8 key bits in shared
// memory; a select kernel finds the bin holding the k-th key; a second pass over only the
// blocks that can hold keys in that bin histograms the lower 7 bits; a last select kernel
// finishes the threshold.
#include <cuda_bf16.h>

#include "mp_internal.cuh"

namespace mp {
namespace {

constexpr uint32_t kNoBin = 0xFFFFFFFFu;

__device__ __forceinline__ uint4 load_vec_raw(const void* base_ptr, bool bf16, uint64_t elem0, uint32_t v,
                                              uint32_t len) {
  // vector v of a block starting at element elem0 with len elements; zero fill past len
  const uint32_t V = bf16 ? 8u : 4u;
  uint32_t k0 = v * V;
  if (k0 + V <= len) {
    const uint4* q = reinterpret_cast<const uint4*>(static_cast<const char*>(base_ptr) +
                                                    (elem0 + k0) * (bf16 ? 2u : 4u));
    return __ldcs(q);
  }
  uint32_t w[4] = {0u, 0u, 0u, 0u};
  if (k0 < len) {
    if (bf16) {
      const uint16_t* s = static_cast<const uint16_t*>(base_ptr) + elem0 + k0;
      for (uint32_t e = 0; e < V && k0 + e < len; ++e) w[e >> 1] |= (uint32_t)s[e] << (16u * (e & 1u));
    } else {
      const uint32_t* s = static_cast<const uint32_t*>(base_ptr) + elem0 + k0;
      for (uint32_t e = 0; e < V && k0 + e < len; ++e) w[e] = s[e];
    }
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}

template <bool BF16>
__device__ __forceinline__ void unpack(const uint4 r, float (&x)[BF16 ? 8 : 4]) {
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

__device__ __forceinline__ uint32_t ties_key(float d) {
  return (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(fabsf(d))) & 0x7FFFu;
}

template <bool BF16, int KG, bool TIES>
__global__ void __launch_bounds__(256) index_kernel(const IndexLaunch p) {
  constexpr int V = BF16 ? 8 : 4;
  __shared__ uint32_t s_hist[TIES ? KG : 1][TIES ? 256 : 1];
  __shared__ float s_ss[KG][8];
  __shared__ float s_mx[KG][8];
  __shared__ uint32_t s_nz[KG][8];

  const uint32_t G = (p.K + KG - 1) / KG;
  const uint64_t b = blockIdx.x / G;
  const uint32_t i0 = (blockIdx.x % G) * KG;
  const uint32_t kc = min((uint32_t)KG, p.K - i0);
  const uint64_t off = p.blk_off[b];
  const uint32_t len = p.blk_len[b];
  const uint32_t nvec = (len + V - 1) / V;
  const uint32_t tid = threadIdx.x, lane = tid & 31u, warp = tid >> 5;

  if constexpr (TIES) {
    for (uint32_t x = tid; x < (uint32_t)KG * 256u; x += 256u) (&s_hist[0][0])[x] = 0u;
    __syncthreads();
  }

  float ss[KG], mx[KG];
  uint32_t nz[KG];
#pragma unroll
  for (int k = 0; k < KG; ++k) {
    ss[k] = 0.0f;
    mx[k] = 0.0f;
    nz[k] = 0u;
  }
  uint32_t bad = 0u;

  for (uint32_t v0 = tid; v0 < nvec; v0 += 2u * kLanes) {
    uint4 rb[2], re[2][KG];
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      uint32_t v = v0 + (uint32_t)u * kLanes;
      if (v < nvec) {
        rb[u] = load_vec_raw(p.base, BF16, off, v, len);
#pragma unroll
        for (int k = 0; k < KG; ++k)
          if ((uint32_t)k < kc) re[u][k] = load_vec_raw(p.experts.p[i0 + k], BF16, off, v, len);
      }
    }
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      uint32_t v = v0 + (uint32_t)u * kLanes;
      if (v >= nvec) break;
      float xb[V];
      unpack<BF16>(rb[u], xb);
#pragma unroll
      for (int k = 0; k < KG; ++k) {
        if ((uint32_t)k >= kc) continue;
        float xe[V];
        unpack<BF16>(re[u][k], xe);
#pragma unroll
        for (int e = 0; e < V; ++e) {
          float d = __fsub_rn(xe[e], xb[e]);
          ss[k] = __fmaf_rn(d, d, ss[k]);
          mx[k] = fmaxf(mx[k], fabsf(d));
          nz[k] += d != 0.0f ? 1u : 0u;
          bad |= ((__float_as_uint(d) & 0x7F800000u) == 0x7F800000u) ? 1u : 0u;
          if constexpr (TIES) {
            if (d != 0.0f) atomicAdd(&s_hist[k][ties_key(d) >> 7], 1u);
          }
        }
      }
    }
  }

  // canonical combine: xor butterfly within each warp, then over the 8 warp sums
#pragma unroll
  for (int k = 0; k < KG; ++k) {
#pragma unroll
    for (int s = 16; s >= 1; s >>= 1) {
      ss[k] = __fadd_rn(ss[k], __shfl_xor_sync(0xFFFFFFFFu, ss[k], s));
      mx[k] = fmaxf(mx[k], __shfl_xor_sync(0xFFFFFFFFu, mx[k], s));
      nz[k] += __shfl_xor_sync(0xFFFFFFFFu, nz[k], s);
    }
    if (lane == 0) {
      s_ss[k][warp] = ss[k];
      s_mx[k][warp] = mx[k];
      s_nz[k][warp] = nz[k];
    }
  }
  if (__syncthreads_or(bad) && tid == 0) atomicOr(p.err, kErrNonfinite);
  if (warp == 0) {
#pragma unroll
    for (int k = 0; k < KG; ++k) {
      float a = lane < 8 ? s_ss[k][lane] : 0.0f;
      float m = lane < 8 ? s_mx[k][lane] : 0.0f;
      uint32_t c = lane < 8 ? s_nz[k][lane] : 0u;
#pragma unroll
      for (int s = 4; s >= 1; s >>= 1) {
        a = __fadd_rn(a, __shfl_xor_sync(0xFFFFFFFFu, a, s));
        m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, s));
        c += __shfl_xor_sync(0xFFFFFFFFu, c, s);
      }
      if (lane == 0 && (uint32_t)k < kc) {
        uint64_t u = (uint64_t)(i0 + k) * p.n_blocks + b;
        p.norm[u] = __fsqrt_rn(a);
        p.maxabs[u] = m;
        p.nnz[u] = c;
        s_nz[k][0] = c;
      }
    }
  }
  if constexpr (TIES) {
    __syncthreads();
    const uint32_t grp = p.blk_group[b];
    for (uint32_t x = tid; x < kc * 256u; x += 256u) {
      uint32_t k = x >> 8, e = x & 255u;
      unsigned long long c = s_hist[k][e];
      if (e == 0) c += len - s_nz[k][0];  // zero deltas have key 0
      if (c) atomicAdd(&p.coarse[((uint64_t)(i0 + k) * p.n_groups + grp) * 256u + e], c);
    }
  }
}

// coarse select: bin e* of the upper 8 key bits holding the k-th largest key, and the
// rank of that key inside the bin
__global__ void ties_coarse_select(const IndexLaunch p) {
  uint64_t x = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (x >= (uint64_t)p.K * p.n_groups) return;
  uint32_t grp = (uint32_t)(x % p.n_groups);
  unsigned long long k = p.kth[grp];
  if (k == 0) {
    p.estar[x] = kNoBin;
    p.rank[x] = 0;
    return;
  }
  const unsigned long long* h = p.coarse + x * 256u;
  unsigned long long cum = 0;
  for (int e = 255; e >= 0; --e) {
    if (cum + h[e] >= k) {
      p.estar[x] = (uint32_t)e;
      p.rank[x] = k - cum;
      return;
    }
    cum += h[e];
  }
  p.estar[x] = 0u;  // unreachable for k <= numel
  p.rank[x] = k - cum;
}

template <bool BF16, int KG>
__global__ void __launch_bounds__(256) ties_fine_kernel(const IndexLaunch p) {
  constexpr int V = BF16 ? 8 : 4;
  __shared__ uint32_t s_fine[KG][128];
  const uint32_t G = (p.K + KG - 1) / KG;
  const uint64_t b = blockIdx.x / G;
  const uint32_t i0 = (blockIdx.x % G) * KG;
  const uint32_t kc = min((uint32_t)KG, p.K - i0);
  const uint32_t grp = p.blk_group[b];
  const uint32_t tid = threadIdx.x;

  uint32_t estar[KG];
  uint32_t want = 0u;  // bit k: expert i0+k may hold keys in its bin e*
#pragma unroll
  for (int k = 0; k < KG; ++k) {
    estar[k] = kNoBin;
    if ((uint32_t)k < kc) {
      uint32_t i = i0 + k;
      uint32_t es = p.estar[(uint64_t)i * p.n_groups + grp];
      uint64_t u = (uint64_t)i * p.n_blocks + b;
      if (es != kNoBin && p.nnz[u] != 0u && (ties_key(p.maxabs[u]) >> 7) >= es) {
        estar[k] = es;
        want |= 1u << k;
      }
    }
  }
  if (want == 0u) return;  // uniform over the CTA
  for (uint32_t x = tid; x < (uint32_t)KG * 128u; x += 256u) (&s_fine[0][0])[x] = 0u;
  __syncthreads();

  const uint64_t off = p.blk_off[b];
  const uint32_t len = p.blk_len[b];
  const uint32_t nvec = (len + V - 1) / V;
  for (uint32_t v = tid; v < nvec; v += kLanes) {
    float xb[V];
    unpack<BF16>(load_vec_raw(p.base, BF16, off, v, len), xb);
#pragma unroll
    for (int k = 0; k < KG; ++k) {
      if (!((want >> k) & 1u)) continue;
      float xe[V];
      unpack<BF16>(load_vec_raw(p.experts.p[i0 + k], BF16, off, v, len), xe);
#pragma unroll
      for (int e = 0; e < V; ++e) {
        float d = __fsub_rn(xe[e], xb[e]);
        uint32_t key = ties_key(d);
        if (d != 0.0f && (key >> 7) == estar[k]) atomicAdd(&s_fine[k][key & 127u], 1u);
      }
    }
  }
  __syncthreads();
  for (uint32_t x = tid; x < (uint32_t)KG * 128u; x += 256u) {
    uint32_t k = x >> 7, m = x & 127u;
    if (!((want >> k) & 1u)) continue;
    uint32_t c = s_fine[k][m];
    if (c) atomicAdd(&p.fine[((uint64_t)(i0 + k) * p.n_groups + grp) * 128u + m], (unsigned long long)c);
  }
}

__global__ void ties_fine_select(const IndexLaunch p) {
  uint64_t x = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (x >= (uint64_t)p.K * p.n_groups) return;
  uint32_t es = p.estar[x];
  if (es == kNoBin) {
    p.tau[x] = kTauNone;
    return;
  }
  const unsigned long long* f = p.fine + x * 128u;
  unsigned long long r = p.rank[x], cum = 0;
  for (int m = 127; m >= 0; --m) {
    cum += f[m];
    if (cum >= r) {
      p.tau[x] = (es << 7) | (uint32_t)m;
      return;
    }
  }
  // only bin 0 can fall short: its uncounted members are exact zeros, key 0
  p.tau[x] = es << 7;
}

template <bool BF16, int KG>
cudaError_t launch_t(const IndexLaunch& p, cudaStream_t st) {
  const uint32_t G = (p.K + KG - 1) / KG;
  const uint64_t grid = p.n_blocks * G;
  if (grid == 0) return cudaSuccess;
  if (grid > 0x7FFFFFFFull) return cudaErrorInvalidValue;
  const bool ties = p.coarse != nullptr;
  if (ties) index_kernel<BF16, KG, true><<<(unsigned)grid, 256, 0, st>>>(p);
  else index_kernel<BF16, KG, false><<<(unsigned)grid, 256, 0, st>>>(p);
  count_launches(1);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess || !ties) return e;
  const uint64_t nsel = (uint64_t)p.K * p.n_groups;
  const unsigned sgrid = (unsigned)((nsel + 127) / 128);
  ties_coarse_select<<<sgrid, 128, 0, st>>>(p);
  ties_fine_kernel<BF16, KG><<<(unsigned)grid, 256, 0, st>>>(p);
  ties_fine_select<<<sgrid, 128, 0, st>>>(p);
  count_launches(3);
  return cudaGetLastError();
}

template <bool BF16>
cudaError_t launch_dtype(const IndexLaunch& p, cudaStream_t st) {
  if (p.K <= 1) return launch_t<BF16, 1>(p, st);
  if (p.K <= 2) return launch_t<BF16, 2>(p, st);
  if (p.K <= 4) return launch_t<BF16, 4>(p, st);
  return launch_t<BF16, 8>(p, st);
}

}  // namespace

cudaError_t launch_index(const IndexLaunch& p, cudaStream_t st) {
  return p.dtype == MP_BF16 ? launch_dtype<true>(p, st) : launch_dtype<false>(p, st);
}

}  // namespace mp
