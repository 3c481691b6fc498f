// Alg. 1 PlanGen on the device.
//
//  1. score: unit u = b*K + i is a candidate iff nnz > 0 (TIES: and key(maxabs) >= tau);
//     score = |coef_i| * norm (fp32), sort key = ~bits(score) so ascending key order is
//     decreasing score;
//  2. stable compaction of the candidates in unit order (so equal scores stay in
//     ascending unit order);
//  3. stable LSD radix sort of (key, unit) pairs, four 8-bit digits; stability plus the
//     unit-ordered input gives the total order (score desc, unit asc);
//  4. inclusive prefix sum of the costs in that order; every position before the first
//     prefix > B is selected (the greedy takes them all);
//  5. after that first overflow only candidates with cost <= the remaining budget R0 can
//     ever be taken (R only shrinks): they are compacted and one warp runs the greedy
//     with skip over them in order;
//  6. the mask, the set hash and the count are scattered from the selected positions,
//     then the last CTA computes the touched-block count and the digest.
#include "mp_internal.cuh"

namespace mp {
namespace {

constexpr int kThreads = 256;
constexpr int kItems = 8;
constexpr uint32_t kTile = kThreads * kItems;  // 2048
constexpr uint32_t kNone = 0xFFFFFFFFu;

// summary words (plan handle) and scratch scalars
enum { S_CHAT = 0, S_NSEL = 1, S_NCAND = 2, S_SETHASH = 3, S_DIGEST = 4, S_TOUCHED = 5, S_ERR = 6 };
enum { X_Q = 0, X_P = 1, X_L = 2, X_R0 = 3, X_PREFIX_BEFORE_P = 4, X_TAILSUM = 5, X_DONE = 6, X_COUNT = 8 };

struct Scratch {
  uint8_t* flag;        // [U] candidate flag in unit order
  uint32_t* key;        // [U] sort key in unit order
  uint32_t* keys_a;     // [U]
  uint32_t* keys_b;     // [U]
  uint32_t* vals_b;     // [U]
  uint32_t* tile_a;     // [n_tiles]
  uint32_t* thist;      // [256 * n_tiles]
  unsigned long long* prefix;   // [U]
  unsigned long long* tile64;   // [n_tiles]
  uint32_t* tail;       // [U]
  uint8_t* tailsel;     // [U]
  unsigned long long* x;        // [X_COUNT]
};

inline size_t align_up(size_t v) { return (v + 255) & ~(size_t)255; }

Scratch carve(void* base, uint64_t U) {
  const uint64_t nt = (U + kTile - 1) / kTile;
  char* p = static_cast<char*>(base);
  Scratch s;
  size_t o = 0;
  auto take = [&](size_t bytes) { char* r = p + o; o += align_up(bytes); return r; };
  s.flag = (uint8_t*)take(U);
  s.key = (uint32_t*)take(U * 4);
  s.keys_a = (uint32_t*)take(U * 4);
  s.keys_b = (uint32_t*)take(U * 4);
  s.vals_b = (uint32_t*)take(U * 4);
  s.tile_a = (uint32_t*)take(nt * 4);
  s.thist = (uint32_t*)take(nt * 256 * 4);
  s.prefix = (unsigned long long*)take(U * 8);
  s.tile64 = (unsigned long long*)take(nt * 8);
  s.tail = (uint32_t*)take(U * 4);
  s.tailsel = (uint8_t*)take(U);
  s.x = (unsigned long long*)take(X_COUNT * 8);
  return s;
}

size_t carve_bytes(uint64_t U) {
  const uint64_t nt = (U + kTile - 1) / kTile;
  return align_up(U) + 4 * align_up(U * 4) + align_up(nt * 4) + align_up(nt * 256 * 4) + align_up(U * 8) +
         align_up(nt * 8) + align_up(U * 4) + align_up(U) + align_up(X_COUNT * 8);
}

__device__ __forceinline__ uint32_t ties_key(float d) {
  // bits(bf16_rne(|d|)) & 0x7FFF, written with integer rounding so it does not depend on
  // a conversion intrinsic: |d| is finite and non-negative here
  uint32_t u = __float_as_uint(fabsf(d));
  uint32_t r = (u + 0x7FFFu + ((u >> 16) & 1u)) >> 16;
  return r & 0x7FFFu;
}

__device__ __forceinline__ uint64_t splitmix64(uint64_t state) {
  uint64_t z = state + 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// block-wide exclusive scan of one value per thread (256 threads); returns the exclusive
// prefix and the block total
template <typename T>
__device__ __forceinline__ T block_exclusive_scan(T v, T& total) {
  __shared__ T s_warp[kThreads / 32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  T x = v;
#pragma unroll
  for (int s = 1; s < 32; s <<= 1) {
    T y = __shfl_up_sync(0xFFFFFFFFu, x, s);
    if (lane >= s) x += y;
  }
  if (lane == 31) s_warp[warp] = x;
  __syncthreads();
  if (warp == 0) {
    T t = lane < kThreads / 32 ? s_warp[lane] : T(0);
#pragma unroll
    for (int s = 1; s < kThreads / 32; s <<= 1) {
      T y = __shfl_up_sync(0xFFFFFFFFu, t, s);
      if (lane >= s) t += y;
    }
    if (lane < kThreads / 32) s_warp[lane] = t;
  }
  __syncthreads();
  T before = warp > 0 ? s_warp[warp - 1] : T(0);
  total = s_warp[kThreads / 32 - 1];
  __syncthreads();  // s_warp reusable by the next call
  return before + x - v;
}

template <typename T>
__device__ __forceinline__ T block_sum(T v) {
  T total;
  block_exclusive_scan<T>(v, total);
  return total;
}

// ---- 1. score + per-tile candidate counts ---------------------------------------------
__global__ void __launch_bounds__(kThreads) k_score(const PlanLaunch p, Scratch s, uint64_t U) {
  const uint64_t t0 = (uint64_t)blockIdx.x * kTile + (uint64_t)threadIdx.x * kItems;
  uint32_t cnt = 0;
#pragma unroll
  for (int k = 0; k < kItems; ++k) {
    uint64_t u = t0 + k;
    if (u >= U) break;
    uint64_t b = u / p.K;
    uint32_t i = (uint32_t)(u % p.K);
    uint64_t st = (uint64_t)i * p.n_blocks + b;
    bool cand = p.nnz[st] != 0u;
    if (cand && p.op_kind == MP_OP_TIES)
      cand = ties_key(p.maxabs[st]) >= p.tau[(uint64_t)i * p.n_groups + p.blk_group[b]];
    float score = __fmul_rn(p.coef[i], p.norm[st]);
    s.flag[u] = cand ? 1 : 0;
    s.key[u] = ~__float_as_uint(score);
    cnt += cand ? 1u : 0u;
  }
  uint32_t tot = block_sum<uint32_t>(cnt);
  if (threadIdx.x == 0) s.tile_a[blockIdx.x] = tot;
}

// single-CTA exclusive scan of n values in place; total to *total_out
template <typename T>
__global__ void __launch_bounds__(1024) k_scan_single(T* data, uint64_t n, unsigned long long* total_out) {
  __shared__ T s_part[1024];
  __shared__ T s_w[32];
  const uint32_t tid = threadIdx.x;
  const uint64_t per = (n + 1023) / 1024;
  const uint64_t a = (uint64_t)tid * per, e = min(n, a + per);
  T sum = 0;
  for (uint64_t j = a; j < e; ++j) sum += data[j];
  // block scan over 1024 thread sums
  const int lane = tid & 31, warp = tid >> 5;
  T x = sum;
  for (int s = 1; s < 32; s <<= 1) {
    T y = __shfl_up_sync(0xFFFFFFFFu, x, s);
    if (lane >= s) x += y;
  }
  if (lane == 31) s_w[warp] = x;
  __syncthreads();
  if (warp == 0) {
    T t = s_w[lane];
    for (int s = 1; s < 32; s <<= 1) {
      T y = __shfl_up_sync(0xFFFFFFFFu, t, s);
      if (lane >= s) t += y;
    }
    s_w[lane] = t;
  }
  __syncthreads();
  T run = (warp > 0 ? s_w[warp - 1] : T(0)) + x - sum;
  for (uint64_t j = a; j < e; ++j) {
    T v = data[j];
    data[j] = run;
    run += v;
  }
  if (tid == 1023 && total_out) *total_out = (unsigned long long)(s_w[31]);
  (void)s_part;
}

// ---- 2. stable compaction of candidates -----------------------------------------------
__global__ void __launch_bounds__(kThreads) k_compact(Scratch s, uint32_t* vals_a, uint64_t U) {
  const uint64_t t0 = (uint64_t)blockIdx.x * kTile + (uint64_t)threadIdx.x * kItems;
  uint32_t cnt = 0;
#pragma unroll
  for (int k = 0; k < kItems; ++k)
    if (t0 + k < U) cnt += s.flag[t0 + k];
  uint32_t tot;
  uint32_t pos = s.tile_a[blockIdx.x] + block_exclusive_scan<uint32_t>(cnt, tot);
#pragma unroll
  for (int k = 0; k < kItems; ++k) {
    uint64_t u = t0 + k;
    if (u < U && s.flag[u]) {
      s.keys_a[pos] = s.key[u];
      vals_a[pos] = (uint32_t)u;
      ++pos;
    }
  }
}

// ---- 3. stable LSD radix sort, one 8-bit digit per pass --------------------------------
__global__ void __launch_bounds__(kThreads) k_sort_hist(const uint32_t* keys, const unsigned long long* x,
                                                        uint32_t* thist, uint32_t shift, uint32_t n_tiles) {
  __shared__ uint32_t h[256];
  h[threadIdx.x] = 0;
  __syncthreads();
  const uint64_t Q = x[X_Q];
  const uint64_t t0 = (uint64_t)blockIdx.x * kTile;
  for (int r = 0; r < kItems; ++r) {
    uint64_t j = t0 + (uint64_t)r * kThreads + threadIdx.x;
    if (j < Q) atomicAdd(&h[(keys[j] >> shift) & 255u], 1u);
  }
  __syncthreads();
  thist[(uint64_t)threadIdx.x * n_tiles + blockIdx.x] = h[threadIdx.x];
}

__global__ void __launch_bounds__(kThreads) k_sort_scatter(const uint32_t* keys_in, const uint32_t* vals_in,
                                                           uint32_t* keys_out, uint32_t* vals_out,
                                                           const unsigned long long* x, const uint32_t* thist,
                                                           uint32_t shift, uint32_t n_tiles) {
  __shared__ uint32_t run[256];
  __shared__ uint32_t wcnt[kThreads / 32][256];
  const uint32_t tid = threadIdx.x, lane = tid & 31u, warp = tid >> 5;
  const uint64_t Q = x[X_Q];
  const uint64_t t0 = (uint64_t)blockIdx.x * kTile;
  if (t0 >= Q) return;
  run[tid] = thist[(uint64_t)tid * n_tiles + blockIdx.x];  // global start of digit tid in this tile
  const uint32_t lt = (1u << lane) - 1u;
  for (int r = 0; r < kItems; ++r) {
    for (int w = 0; w < kThreads / 32; ++w) wcnt[w][tid] = 0;
    __syncthreads();
    uint64_t j = t0 + (uint64_t)r * kThreads + tid;
    bool valid = j < Q;
    uint32_t key = valid ? keys_in[j] : 0u;
    uint32_t val = valid ? vals_in[j] : 0u;
    uint32_t d = valid ? ((key >> shift) & 255u) : 256u;
    uint32_t peers = __match_any_sync(0xFFFFFFFFu, d);
    uint32_t rank = __popc(peers & lt);
    if (valid && rank == 0) wcnt[warp][d] = __popc(peers);
    __syncthreads();
    {
      uint32_t acc = run[tid];
      for (int w = 0; w < kThreads / 32; ++w) {
        uint32_t c = wcnt[w][tid];
        wcnt[w][tid] = acc;
        acc += c;
      }
      run[tid] = acc;
    }
    __syncthreads();
    if (valid) {
      uint32_t pos = wcnt[warp][d] + rank;
      keys_out[pos] = key;
      vals_out[pos] = val;
    }
    __syncthreads();
  }
}

// ---- 4. costs in sorted order: tile sums, then prefix and the first overflow ------------
__device__ __forceinline__ unsigned long long unit_cost(const PlanLaunch& p, uint32_t u) {
  return (unsigned long long)p.blk_len[u / p.K] * p.elem_size;
}

__global__ void __launch_bounds__(kThreads) k_cost_tiles(const PlanLaunch p, Scratch s, const uint32_t* order) {
  const uint64_t Q = s.x[X_Q];
  const uint64_t t0 = (uint64_t)blockIdx.x * kTile + (uint64_t)threadIdx.x * kItems;
  unsigned long long c = 0;
#pragma unroll
  for (int k = 0; k < kItems; ++k)
    if (t0 + k < Q) c += unit_cost(p, order[t0 + k]);
  unsigned long long tot = block_sum<unsigned long long>(c);
  if (threadIdx.x == 0) s.tile64[blockIdx.x] = tot;
}

__global__ void __launch_bounds__(kThreads) k_cost_prefix(const PlanLaunch p, Scratch s, const uint32_t* order) {
  const uint64_t Q = s.x[X_Q];
  const uint64_t t0 = (uint64_t)blockIdx.x * kTile + (uint64_t)threadIdx.x * kItems;
  unsigned long long c[kItems];
  unsigned long long sum = 0;
#pragma unroll
  for (int k = 0; k < kItems; ++k) {
    c[k] = t0 + k < Q ? unit_cost(p, order[t0 + k]) : 0ull;
    sum += c[k];
  }
  unsigned long long tot;
  unsigned long long run = s.tile64[blockIdx.x] + block_exclusive_scan<unsigned long long>(sum, tot);
#pragma unroll
  for (int k = 0; k < kItems; ++k) {
    uint64_t j = t0 + k;
    if (j >= Q) break;
    unsigned long long before = run;
    run += c[k];
    s.prefix[j] = run;
    if (run > p.budget && before <= p.budget) {  // unique: the prefix is non-decreasing
      s.x[X_P] = j;
      s.x[X_PREFIX_BEFORE_P] = before;
    }
  }
}

// ---- 5. the tail after the first overflow ------------------------------------------------
__device__ __forceinline__ bool tail_candidate(const PlanLaunch& p, const Scratch& s, const uint32_t* order,
                                               uint64_t j, uint64_t Q, uint64_t P, unsigned long long R0) {
  return j < Q && j > P && unit_cost(p, order[j]) <= R0;
}

__global__ void __launch_bounds__(kThreads) k_tail_count(const PlanLaunch p, Scratch s, const uint32_t* order) {
  const uint64_t Q = s.x[X_Q], P = s.x[X_P];
  if (P == kNone || P == 0xFFFFFFFFFFFFFFFFull) {
    if (threadIdx.x == 0) s.tile_a[blockIdx.x] = 0;
    return;
  }
  const unsigned long long R0 = p.budget - s.x[X_PREFIX_BEFORE_P];
  const uint64_t t0 = (uint64_t)blockIdx.x * kTile + (uint64_t)threadIdx.x * kItems;
  uint32_t cnt = 0;
#pragma unroll
  for (int k = 0; k < kItems; ++k) cnt += tail_candidate(p, s, order, t0 + k, Q, P, R0) ? 1u : 0u;
  uint32_t tot = block_sum<uint32_t>(cnt);
  if (threadIdx.x == 0) s.tile_a[blockIdx.x] = tot;
}

__global__ void __launch_bounds__(kThreads) k_tail_compact(const PlanLaunch p, Scratch s, const uint32_t* order) {
  const uint64_t Q = s.x[X_Q], P = s.x[X_P];
  if (P == 0xFFFFFFFFFFFFFFFFull) return;
  const unsigned long long R0 = p.budget - s.x[X_PREFIX_BEFORE_P];
  const uint64_t t0 = (uint64_t)blockIdx.x * kTile + (uint64_t)threadIdx.x * kItems;
  uint32_t cnt = 0;
  bool f[kItems];
#pragma unroll
  for (int k = 0; k < kItems; ++k) {
    f[k] = tail_candidate(p, s, order, t0 + k, Q, P, R0);
    cnt += f[k] ? 1u : 0u;
  }
  uint32_t tot;
  uint32_t pos = s.tile_a[blockIdx.x] + block_exclusive_scan<uint32_t>(cnt, tot);
#pragma unroll
  for (int k = 0; k < kItems; ++k)
    if (f[k]) s.tail[pos++] = (uint32_t)(t0 + k);
}

// one warp: greedy with skip over the compacted tail, in order
__global__ void k_tail_greedy(const PlanLaunch p, Scratch s, const uint32_t* order) {
  const uint32_t lane = threadIdx.x;
  const uint64_t P = s.x[X_P];
  if (P == 0xFFFFFFFFFFFFFFFFull) {
    if (lane == 0) s.x[X_TAILSUM] = 0;
    return;
  }
  const uint64_t L = s.x[X_L];
  const unsigned long long R0 = p.budget - s.x[X_PREFIX_BEFORE_P];
  unsigned long long R = R0;
  for (uint64_t c0 = 0; c0 < L; c0 += 32) {
    uint64_t j = c0 + lane;
    uint32_t pos = j < L ? s.tail[j] : 0u;
    unsigned long long c = j < L ? unit_cost(p, order[pos]) : ~0ull;
    uint32_t done = 0u;
    for (;;) {
      uint32_t m = __ballot_sync(0xFFFFFFFFu, c <= R) & ~done;
      if (m == 0u) break;
      int f = __ffs(m) - 1;
      unsigned long long cf = __shfl_sync(0xFFFFFFFFu, c, f);
      if ((int)lane == f) s.tailsel[pos] = 1;
      R -= cf;
      done = f == 31 ? 0xFFFFFFFFu : ((2u << f) - 1u);
    }
  }
  if (lane == 0) s.x[X_TAILSUM] = R0 - R;
}

// ---- 6. mask, set hash, count; then touched blocks and digest (last CTA) ----------------
__global__ void __launch_bounds__(kThreads) k_mask(const PlanLaunch p, Scratch s, const uint32_t* order) {
  const uint64_t Q = s.x[X_Q], P = s.x[X_P];
  const uint64_t t0 = (uint64_t)blockIdx.x * kTile + (uint64_t)threadIdx.x * kItems;
  unsigned long long h = 0, n = 0;
#pragma unroll
  for (int k = 0; k < kItems; ++k) {
    uint64_t j = t0 + k;
    if (j >= Q) break;
    if (j < P || s.tailsel[j]) {
      uint32_t u = order[j];
      atomicOr(&p.mask[u / p.K], 1u << (u % p.K));
      h += splitmix64(u);
      ++n;
    }
  }
  h = block_sum<unsigned long long>(h);
  n = block_sum<unsigned long long>(n);
  if (threadIdx.x == 0 && n) {
    atomicAdd((unsigned long long*)&p.summary[S_SETHASH], h);
    atomicAdd((unsigned long long*)&p.summary[S_NSEL], n);
  }
}

__device__ __forceinline__ uint64_t fnv_u64(uint64_t h, uint64_t v) {
  for (int k = 0; k < 8; ++k) {
    h ^= (v >> (8 * k)) & 0xFFu;
    h *= 1099511628211ull;
  }
  return h;
}

__global__ void __launch_bounds__(kThreads) k_touched_finalize(const PlanLaunch p, Scratch s) {
  __shared__ bool last;
  unsigned long long cnt = 0;
  for (uint64_t b = (uint64_t)blockIdx.x * kThreads + threadIdx.x; b < p.n_blocks;
       b += (uint64_t)gridDim.x * kThreads)
    cnt += p.mask[b] != 0u ? 1ull : 0ull;
  cnt = block_sum<unsigned long long>(cnt);
  if (threadIdx.x == 0) {
    if (cnt) atomicAdd((unsigned long long*)&p.summary[S_TOUCHED], cnt);
    __threadfence();
    unsigned long long prev = atomicAdd(&s.x[X_DONE], 1ull);
    last = prev == gridDim.x - 1;
  }
  __syncthreads();
  if (!last || threadIdx.x != 0) return;
  __threadfence();
  const uint64_t P = s.x[X_P], Q = s.x[X_Q];
  unsigned long long chat =
      P == 0xFFFFFFFFFFFFFFFFull ? (Q ? s.prefix[Q - 1] : 0ull) : s.x[X_PREFIX_BEFORE_P] + s.x[X_TAILSUM];
  volatile unsigned long long* sum = (volatile unsigned long long*)p.summary;
  unsigned long long nsel = sum[S_NSEL], sh = sum[S_SETHASH];
  uint64_t h = 14695981039346656037ull;
  for (uint32_t k = 0; k < p.hdr_prefix_len; ++k) {
    h ^= p.hdr_prefix[k];
    h *= 1099511628211ull;
  }
  h = fnv_u64(h, chat);
  h = fnv_u64(h, nsel);
  h = fnv_u64(h, sh);
  sum[S_CHAT] = chat;
  sum[S_NCAND] = Q;
  sum[S_DIGEST] = h;
  sum[S_ERR] = *p.index_err;
}

}  // namespace

size_t plan_scratch_bytes(uint64_t n_units) { return carve_bytes(n_units); }

cudaError_t launch_plan(const PlanLaunch& p, void* scratch, cudaStream_t st) {
  const uint64_t U = (uint64_t)p.K * p.n_blocks;
  const uint64_t nt64 = (U + kTile - 1) / kTile;
  if (nt64 > 0x7FFFFFFFull || U > 0xFFFFFFFFull) return cudaErrorInvalidValue;
  const uint32_t nt = (uint32_t)nt64;
  Scratch s = carve(scratch, U);
  cudaError_t e;
  if ((e = cudaMemsetAsync(p.summary, 0, 8 * sizeof(uint64_t), st)) != cudaSuccess) return e;
  if ((e = cudaMemsetAsync(p.mask, 0, p.n_blocks * sizeof(uint32_t), st)) != cudaSuccess) return e;
  if ((e = cudaMemsetAsync(s.tailsel, 0, U, st)) != cudaSuccess) return e;
  if ((e = cudaMemsetAsync(s.x, 0, X_COUNT * 8, st)) != cudaSuccess) return e;
  if ((e = cudaMemsetAsync(&s.x[X_P], 0xFF, 8, st)) != cudaSuccess) return e;

  uint32_t* vals_a = p.order;
  k_score<<<nt, kThreads, 0, st>>>(p, s, U);
  k_scan_single<uint32_t><<<1, 1024, 0, st>>>(s.tile_a, nt, &s.x[X_Q]);
  k_compact<<<nt, kThreads, 0, st>>>(s, vals_a, U);
  // four passes: a -> b -> a -> b -> a, final order in vals_a (= the plan's order array)
  uint32_t *kin = s.keys_a, *vin = vals_a, *kout = s.keys_b, *vout = s.vals_b;
  for (uint32_t pass = 0; pass < 4; ++pass) {
    k_sort_hist<<<nt, kThreads, 0, st>>>(kin, s.x, s.thist, 8u * pass, nt);
    k_scan_single<uint32_t><<<1, 1024, 0, st>>>(s.thist, (uint64_t)nt * 256u, nullptr);
    k_sort_scatter<<<nt, kThreads, 0, st>>>(kin, vin, kout, vout, s.x, s.thist, 8u * pass, nt);
    uint32_t* t;
    t = kin, kin = kout, kout = t;
    t = vin, vin = vout, vout = t;
  }
  const uint32_t* order = vals_a;
  k_cost_tiles<<<nt, kThreads, 0, st>>>(p, s, order);
  k_scan_single<unsigned long long><<<1, 1024, 0, st>>>(s.tile64, nt, nullptr);
  k_cost_prefix<<<nt, kThreads, 0, st>>>(p, s, order);
  k_tail_count<<<nt, kThreads, 0, st>>>(p, s, order);
  k_scan_single<uint32_t><<<1, 1024, 0, st>>>(s.tile_a, nt, &s.x[X_L]);
  k_tail_compact<<<nt, kThreads, 0, st>>>(p, s, order);
  k_tail_greedy<<<1, 32, 0, st>>>(p, s, order);
  k_mask<<<nt, kThreads, 0, st>>>(p, s, order);
  uint64_t tb = (p.n_blocks + kThreads - 1) / kThreads;
  unsigned tgrid = (unsigned)(tb < 1024 ? (tb ? tb : 1) : 1024);
  k_touched_finalize<<<tgrid, kThreads, 0, st>>>(p, s);
  count_launches(3 + 4 * 3 + 9);
  return cudaGetLastError();
}

}  // namespace mp
