// Block content hashes (Sec. 3 "Catalog": the catalog stores hashes of every block;
// Alg. 2 validates hashes before it builds the manifest).
//
//   hash(block) = SplitMix64(H xor L),  H = sum_q lo_q * (k_q | 1) + hi_q * (rotl(k_q, 32) | 1)
//
// mod 2^64, over the block's 16-byte vectors q (zero-padded), lo_q / hi_q its two
// little-endian 64-bit words, k_q = SplitMix64(q) with q counted from the block's start,
// L = the block's bytes.  The sum is exact in any order, so 256 threads each take vectors
// t, t + 256, ... and the partial sums are added in a tree.
//
// One pass streams each block once with 16-byte loads (eight in flight per thread); it is
// bound by HBM (or by the host link for a pinned host pool).  Items are (checkpoint, block)
// pairs, one CTA per item, taken in grid-stride order by a grid of resident CTAs.
#include "mp_internal.cuh"

namespace mp {
namespace {

constexpr int kHT = 256;
constexpr int kUnroll = 8;

__device__ __forceinline__ uint64_t splitmix64(uint64_t z) {
  z += 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

__device__ __forceinline__ uint64_t vec_term(const uint4 v, uint64_t q) {
  const uint64_t k = splitmix64(q);
  const uint64_t a = k | 1ull, b = ((k << 32) | (k >> 32)) | 1ull;
  const uint64_t lo = ((uint64_t)v.y << 32) | v.x, hi = ((uint64_t)v.w << 32) | v.z;
  return lo * a + hi * b;
}

// vector q of a block of `bytes` bytes at p (16-byte aligned): whole vectors by one load,
// the ragged last vector by 16-bit loads (a block holds whole 2- or 4-byte elements),
// zero past the end
__device__ __forceinline__ uint4 load_vec(const uint8_t* p, uint64_t q, uint64_t bytes) {
  const uint64_t o = q * 16u;
  if (o + 16u <= bytes) return __ldcs(reinterpret_cast<const uint4*>(p + o));
  uint32_t w[4] = {0u, 0u, 0u, 0u};
  for (uint32_t h = 0; h < 8u && o + 2u * h < bytes; ++h)
    w[h >> 1] |= (uint32_t)(reinterpret_cast<const uint16_t*>(p + o)[h]) << (16u * (h & 1u));
  return make_uint4(w[0], w[1], w[2], w[3]);
}

// H of one block, reduced over the CTA (valid in thread 0)
__device__ __forceinline__ uint64_t block_sum(const uint8_t* p, uint64_t bytes) {
  __shared__ uint64_t s_w[kHT / 32];
  const uint64_t nq = (bytes + 15u) / 16u;
  uint64_t h = 0;
  for (uint64_t q0 = threadIdx.x; q0 < nq; q0 += (uint64_t)kHT * kUnroll) {
    uint4 v[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const uint64_t q = q0 + (uint64_t)u * kHT;
      v[u] = q < nq ? load_vec(p, q, bytes) : make_uint4(0u, 0u, 0u, 0u);
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const uint64_t q = q0 + (uint64_t)u * kHT;
      if (q < nq) h += vec_term(v[u], q);
    }
  }
#pragma unroll
  for (int s = 16; s >= 1; s >>= 1) h += __shfl_xor_sync(0xFFFFFFFFu, h, s);
  if ((threadIdx.x & 31u) == 0) s_w[threadIdx.x >> 5] = h;
  __syncthreads();
  uint64_t t = 0;
  if (threadIdx.x == 0)
    for (int w = 0; w < kHT / 32; ++w) t += s_w[w];
  __syncthreads();
  return t;
}

// items: k * n_blocks + b for checkpoint k = 0 (base), 1..K (experts), K + 1 (output,
// validation only).  Catalog mode writes the hashes; validation compares the base and the
// selected expert blocks with the catalog and writes the output's hashes.
__global__ void __launch_bounds__(kHT) hash_kernel(const HashLaunch p) {
  const uint64_t nb = p.n_blocks;
  const uint32_t n_ck = p.K + 1u + (p.validate ? 1u : 0u);
  const uint64_t n_items = (uint64_t)n_ck * nb;
  for (uint64_t it = blockIdx.x; it < n_items; it += gridDim.x) {
    const uint32_t k = (uint32_t)(it / nb);
    const uint64_t b = it % nb;
    if (p.validate && k >= 1u && k <= p.K && !((p.mask[b] >> (k - 1u)) & 1u)) continue;  // not read
    const uint64_t off = p.blk_off[b], bytes = (uint64_t)p.blk_len[b] * p.elem_size;
    if (kChecked && !chunk_in_bounds(b, 0, nb, off, p.blk_len[b], off, p.blk_len[b],
                                     k >= 1u && k <= p.K ? 1ull << (k - 1u) : 0ull, p.K, p.elem_size, 0, p.ext)) {
      if (threadIdx.x == 0 && p.err) atomicOr(p.err, kErrBounds);  // uniform over the CTA
      continue;
    }
    const uint8_t* src;
    if (k == 0u) src = static_cast<const uint8_t*>(p.base) + off * p.elem_size;
    else if (k <= p.K) src = static_cast<const uint8_t*>(p.experts.p[k - 1u]) + off * p.elem_size;
    else src = static_cast<const uint8_t*>(p.out) + off * p.elem_size;
    const uint64_t H = block_sum(src, bytes);
    if (threadIdx.x != 0) continue;
    const uint64_t hash = splitmix64(H ^ bytes);
    if (!p.validate) {
      if (k == 0u) p.base_hash[b] = hash;
      else p.expert_hash[(uint64_t)(k - 1u) * nb + b] = hash;
    } else if (k > p.K) {
      p.out_hash[b] = hash;
    } else {
      const uint64_t want = k == 0u ? p.base_hash[b] : p.expert_hash[(uint64_t)(k - 1u) * nb + b];
      atomicAdd(&p.result[0], 1ull);  // blocks checked
      if (hash != want) {
        atomicAdd(&p.result[1], 1ull);  // mismatches
        atomicMin(&p.result[2], (unsigned long long)it);  // the first mismatching item
      }
    }
  }
}

}  // namespace

cudaError_t launch_hash(const HashLaunch& p, cudaStream_t st) {
  if (p.n_blocks == 0) return cudaSuccess;
  int dev = 0, sms = 0;
  cudaError_t e;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
  int per_sm = 0;
  if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, hash_kernel, kHT, 0)) != cudaSuccess) return e;
  if (per_sm < 1) per_sm = 1;
  const uint64_t n_items = (uint64_t)(p.K + 1u + (p.validate ? 1u : 0u)) * p.n_blocks;
  uint64_t grid = (uint64_t)sms * (uint64_t)per_sm;  // every CTA resident
  if (grid > n_items) grid = n_items;
  hash_kernel<<<(unsigned)grid, kHT, 0, st>>>(p);
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace mp
