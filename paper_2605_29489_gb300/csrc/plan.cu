// Alg. 1 PlanGen on the device, as one cooperative persistent kernel.
//
// The grid's CTAs all stay resident (cooperative launch) and move through the phases
// below together, separated by grid barriers whose waits are bounded.  Every phase
// gives CTA c a contiguous slice of the data, so order is preserved wherever it matters.
//
//  0  tensor-level fallback (only for catalogs with entries lacking statistics, nnz =
//     kNnzMissing): flag every (expert, tensor) pair holding one; then one warp per flagged
//     pair computes its unit's cost (the whole tensor's bytes) and score (|coef_i| times
//     the norm of the tensor's known blocks: an fp32 fma chain in block order, then sqrt).
//     The pair's unit is b0(t)*K + i; the tensor's other units are not candidates.
//  A  score: unit u = b*K + i is a candidate iff nnz > 0 (TIES: and key(maxabs) >= tau);
//     score = |coef_i| * norm (fp32), divided by the block's bytes in the score-per-byte
//     mode; sort key = ~bits(score), so ascending key order is
//     decreasing score.  Each CTA counts the candidates of its unit slice.
//  B  stable compaction of the candidates in unit order (so equal scores stay in
//     ascending unit order).
//  C  stable LSD radix sort of (key, unit) pairs, four 8-bit digits; a digit that is the
//     same for every key is skipped.  Stability plus the unit-ordered input gives the
//     total order (score desc, unit asc).
//  D  costs in that order: every position before the first prefix sum > B is selected.
//  E  after that first overflow only candidates with cost <= the remaining budget R0 can
//     ever be taken (R only shrinks): they are compacted, then one warp of CTA 0 runs the
//     greedy with skip over them in order, from shared memory.
//  F  the mask, the set hash and the count are scattered from the selected positions
//     (a taken fallback unit sets its expert's bit in a per-tensor word, which the
//     touched-block pass ORs into every block of the tensor); the last CTA computes the
//     digest.
#include "mp_internal.cuh"

namespace mp {
namespace {

constexpr int kPT = 256;            // threads per CTA
constexpr uint32_t kMaxGrid = 1024;  // upper bound of the cooperative grid (scratch sizing)
constexpr uint32_t kTailChunk = 4096;
constexpr uint32_t kBarrierLimit = 1u << 24;

// summary words (plan handle)
enum { S_CHAT = 0, S_NSEL = 1, S_NCAND = 2, S_SETHASH = 3, S_DIGEST = 4, S_TOUCHED = 5, S_ERR = 6 };
// scratch scalars
enum { X_BAR_COUNT = 0, X_BAR_GEN = 1, X_P = 2, X_PBP = 3, X_TAILSUM = 4, X_DONE = 5, X_TOTAL = 6, X_MISSING = 7,
       X_TAILMIN = 8, X_BADORDER = 9, X_COUNT = 16 };

constexpr unsigned long long kNoP = ~0ull;

struct Scratch {
  uint32_t* keys_a;             // [U]
  uint32_t* keys_b;             // [U]
  uint32_t* vals_b;             // [U]
  uint32_t* tail_pos;           // [U]
  unsigned long long* tail_cost;  // [U] costs of the compacted tail, in order
  uint8_t* tailsel;             // [U]
  uint32_t* hist;               // [256][kMaxGrid]
  uint32_t* tot;                // [256]
  unsigned long long* cta_a;    // [kMaxGrid]
  unsigned long long* cta_b;    // [kMaxGrid]
  unsigned long long* x;        // [X_COUNT]
  uint32_t* pair_flag;          // [K * n_tensors] (fallback only; cleared by the host)
  uint32_t* pair_key;           // [K * n_tensors]
  unsigned long long* pair_cost;  // [K * n_tensors]
  uint32_t* sel_bits;           // [n_tensors] experts whose fallback unit of the tensor was taken (cleared by the host)
};

inline size_t align_up(size_t v) { return (v + 255) & ~(size_t)255; }

size_t carve(void* base, uint64_t U, uint64_t n_pairs, Scratch* s) {
  char* p = static_cast<char*>(base);
  size_t o = 0;
  auto take = [&](size_t bytes) { char* r = p + o; o += align_up(bytes); return r; };
  Scratch t;
  t.keys_a = (uint32_t*)take(U * 4);
  t.keys_b = (uint32_t*)take(U * 4);
  t.vals_b = (uint32_t*)take(U * 4);
  t.tail_pos = (uint32_t*)take(U * 4);
  t.tail_cost = (unsigned long long*)take(U * 8);
  t.tailsel = (uint8_t*)take(U);
  t.hist = (uint32_t*)take((size_t)256 * kMaxGrid * 4);
  t.tot = (uint32_t*)take(256 * 4);
  t.cta_a = (unsigned long long*)take(kMaxGrid * 8);
  t.cta_b = (unsigned long long*)take(kMaxGrid * 8);
  t.x = (unsigned long long*)take(X_COUNT * 8);
  t.pair_flag = (uint32_t*)take(n_pairs * 4);
  t.pair_key = (uint32_t*)take(n_pairs * 4);
  t.pair_cost = (unsigned long long*)take(n_pairs * 8);
  t.sel_bits = (uint32_t*)take(n_pairs * 4);  // n_tensors words used (n_pairs >= n_tensors)
  if (s) *s = t;
  return o;
}

__device__ __forceinline__ uint32_t ties_key(float d) {
  // bits(bf16_rne(|d|)) & 0x7FFF by integer rounding; |d| is finite and non-negative here
  uint32_t u = __float_as_uint(fabsf(d));
  return ((u + 0x7FFFu + ((u >> 16) & 1u)) >> 16) & 0x7FFFu;
}

__device__ __forceinline__ uint64_t splitmix64(uint64_t state) {
  uint64_t z = state + 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

__device__ __forceinline__ unsigned ld_acquire(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return (unsigned)v;
}

// grid barrier: the last CTA to arrive bumps the generation; the others wait for it with
// a bounded number of polls.  Returns false (uniformly inside the CTA) if the wait expired.
__device__ __forceinline__ bool grid_sync(unsigned long long* x, unsigned& gen, uint64_t* summary) {
  __shared__ int s_ok;
  __syncthreads();
  if (threadIdx.x == 0) {
    int ok = 1;
    const unsigned target = gen + 1;
    __threadfence();
    if (atomicAdd(&x[X_BAR_COUNT], 1ull) == (unsigned long long)(gridDim.x - 1)) {
      x[X_BAR_COUNT] = 0;
      __threadfence();
      atomicExch(&x[X_BAR_GEN], (unsigned long long)target);
    } else {
      uint32_t k = 0;
      while (ld_acquire(&x[X_BAR_GEN]) != target) {
        if (++k > kBarrierLimit) {
          ok = 0;
          atomicOr((unsigned long long*)&summary[S_ERR], (unsigned long long)kErrTimeout);
          break;
        }
        __nanosleep(32);
      }
    }
    __threadfence();
    gen = target;
    s_ok = ok;
  }
  __syncthreads();
  return s_ok != 0;
}

// block-wide exclusive scan (256 threads) with total
template <typename T>
__device__ __forceinline__ T block_scan(T v, T& total) {
  __shared__ T s_w[kPT / 32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  T x = v;
#pragma unroll
  for (int s = 1; s < 32; s <<= 1) {
    T y = __shfl_up_sync(0xFFFFFFFFu, x, s);
    if (lane >= s) x += y;
  }
  if (lane == 31) s_w[warp] = x;
  __syncthreads();
  if (warp == 0) {
    T t = lane < kPT / 32 ? s_w[lane] : T(0);
#pragma unroll
    for (int s = 1; s < kPT / 32; s <<= 1) {
      T y = __shfl_up_sync(0xFFFFFFFFu, t, s);
      if (lane >= s) t += y;
    }
    if (lane < kPT / 32) s_w[lane] = t;
  }
  __syncthreads();
  const T before = warp > 0 ? s_w[warp - 1] : T(0);
  total = s_w[kPT / 32 - 1];
  __syncthreads();
  return before + x - v;
}

template <typename T>
__device__ __forceinline__ T block_sum(T v) {
  T t;
  block_scan<T>(v, t);
  return t;
}

// sum of a[0..n) (n <= kMaxGrid), computed by the whole CTA
__device__ __forceinline__ unsigned long long block_sum_prefix(const unsigned long long* a, uint32_t n) {
  unsigned long long s = 0;
  for (uint32_t k = threadIdx.x; k < n; k += kPT) s += a[k];
  return block_sum<unsigned long long>(s);
}

struct Unit {
  bool cand;
  uint32_t key;
};

__device__ __forceinline__ Unit score_unit(const PlanLaunch& p, const Scratch& s, uint64_t u) {
  const uint64_t b = u / p.K;
  const uint32_t i = (uint32_t)(u % p.K);
  const uint64_t st = (uint64_t)i * p.n_blocks + b;
  if (p.fallback) {
    const uint32_t t = p.blk_tensor[b];
    const uint32_t pr = i * p.n_tensors + t;
    if (s.pair_flag[pr]) return Unit{b == p.t_blk0[t], s.pair_key[pr]};
  }
  const uint32_t nz = p.nnz[st];
  bool cand = nz != 0u && nz != kNnzMissing;
  if (cand && p.op_kind == MP_OP_TIES)
    cand = ties_key(p.maxabs[st]) >= p.tau[(uint64_t)i * p.n_groups + p.blk_group[b]];
  float score = __fmul_rn(p.coef[i], p.norm[st]);
  // score per byte: one IEEE division by the block's byte cost (exact in fp32, <= 2^20)
  if (p.score_mode) score = __fdiv_rn(score, (float)(p.blk_len[b] * p.elem_size));
  return Unit{cand, ~__float_as_uint(score)};
}

__device__ __forceinline__ unsigned long long unit_cost(const PlanLaunch& p, const Scratch& s, uint32_t u) {
  const uint32_t b = u / p.K;
  if (p.fallback) {
    const uint32_t pr = (u % p.K) * p.n_tensors + p.blk_tensor[b];
    if (s.pair_flag[pr]) return s.pair_cost[pr];
  }
  return (unsigned long long)p.blk_len[b] * p.elem_size;
}

// phase 0b for one flagged pair (i, t), by one warp: cost = the tensor's bytes, key from
// |coef_i| * sqrt(ss), ss the fp32 chain fma(n, n, ss) over the known blocks in block order.
// The lanes load a batch of kFbChunks chunks of 32 consecutive entries at once (one load
// latency per batch); every lane then runs the same chain over them in block order.
constexpr int kFbChunks = 8;

__device__ __forceinline__ void fallback_pair(const PlanLaunch& p, const Scratch& s, uint32_t pr, uint32_t lane) {
  const uint32_t i = pr / p.n_tensors, t = pr % p.n_tensors;
  const uint32_t b0 = p.t_blk0[t], b1 = p.t_blk0[t + 1];
  const float* nrm = p.norm + (uint64_t)i * p.n_blocks;
  const uint32_t* nz = p.nnz + (uint64_t)i * p.n_blocks;
  float ss = 0.0f;
  unsigned long long cost = 0;
  for (uint32_t bb = b0; bb < b1; bb += 32u * kFbChunks) {
    float n[kFbChunks];
    bool known[kFbChunks];
#pragma unroll
    for (int c = 0; c < kFbChunks; ++c) {
      const uint32_t b = bb + 32u * c + lane;
      n[c] = 0.0f;
      known[c] = false;
      if (b < b1) {
        n[c] = __ldg(nrm + b);
        known[c] = __ldg(nz + b) != kNnzMissing;
        cost += (unsigned long long)__ldg(p.blk_len + b) * p.elem_size;
      }
    }
#pragma unroll
    for (int c = 0; c < kFbChunks; ++c) {
      // an entry without statistics adds fma(0, 0, ss) = ss exactly (ss >= +0)
      const float nv = known[c] ? n[c] : 0.0f;
#pragma unroll
      for (int j = 0; j < 32; ++j) {
        const float nj = __shfl_sync(0xFFFFFFFFu, nv, j);
        ss = __fmaf_rn(nj, nj, ss);
      }
    }
  }
#pragma unroll
  for (int sh = 16; sh > 0; sh >>= 1) cost += __shfl_xor_sync(0xFFFFFFFFu, cost, sh);
  float score = __fmul_rn(p.coef[i], __fsqrt_rn(ss));
  if (p.score_mode) score = __fdiv_rn(score, __ull2float_rn(cost));
  if (lane == 0) {
    s.pair_key[pr] = ~__float_as_uint(score);
    s.pair_cost[pr] = cost;
  }
}

__device__ __forceinline__ void slice(uint64_t n, uint64_t& a, uint64_t& b) {
  a = n * blockIdx.x / gridDim.x;
  b = n * (blockIdx.x + 1) / gridDim.x;
}

__global__ void __launch_bounds__(kPT) plan_kernel(const PlanLaunch p, Scratch s) {
  __shared__ uint32_t s_run[256];
  __shared__ uint32_t s_wcnt[kPT / 32][256];
  __shared__ unsigned long long s_cost[kTailChunk];
  __shared__ unsigned long long s_bcast[1];
  const uint32_t tid = threadIdx.x, lane = tid & 31u, warp = tid >> 5;
  const uint32_t G = gridDim.x, c = blockIdx.x;
  const uint64_t U = (uint64_t)p.K * p.n_blocks;
  unsigned gen = 0;

  // ---- zero the outputs; A: count the candidates of this CTA's unit slice ----
  for (uint64_t k = (uint64_t)c * kPT + tid; k < p.n_blocks; k += (uint64_t)G * kPT) p.mask[k] = 0u;
  for (uint64_t k = (uint64_t)c * kPT + tid; k < U; k += (uint64_t)G * kPT) s.tailsel[k] = 0;
  if (c == 0 && tid < 8) p.summary[tid] = 0;
  if (c == 0 && tid == 0) {
    s.x[X_P] = kNoP;
    s.x[X_TAILMIN] = ~0ull;
  }
  uint64_t Q = 0, q0 = 0, q1 = 0;
  if (p.cache_q_in) {
    // the candidates in traversal order from an earlier plan of this index and operator:
    // phases 0 to C depend on the operator and the catalog, not on the budget
    Q = *p.cache_q_in;
    if (Q > U) {  // the plan that was to leave the order did not finish: report, plan nothing
      if (c == 0 && tid == 0) s.x[X_BADORDER] = 1ull;
      Q = 0;
    }
    slice(Q, q0, q1);
    for (uint64_t j = q0 + tid; j < q1; j += kPT) p.order[j] = p.cache_order_in[j];
    if (!grid_sync(s.x, gen, p.summary)) return;
  } else {
    uint64_t u0, u1;
    slice(U, u0, u1);
    if (p.fallback) {
      // 0a: flag the pairs holding an entry without statistics (one atomic per pair and warp)
      for (uint64_t t0 = u0; t0 < u1; t0 += kPT) {
        const uint64_t u = t0 + tid;
        uint32_t pr = 0xFFFFFFFFu;
        if (u < u1) {
          const uint64_t b = u / p.K;
          const uint32_t i = (uint32_t)(u % p.K);
          if (p.nnz[(uint64_t)i * p.n_blocks + b] == kNnzMissing) pr = i * p.n_tensors + p.blk_tensor[b];
        }
        const uint32_t peers = __match_any_sync(0xFFFFFFFFu, pr);
        if (pr != 0xFFFFFFFFu && lane == (uint32_t)(__ffs(peers) - 1)) atomicOr(&s.pair_flag[pr], 1u);
      }
      if (!grid_sync(s.x, gen, p.summary)) return;
      // 0b: the flagged pairs' units, one warp each
      const uint32_t n_pairs = p.K * p.n_tensors, nw = G * (kPT / 32);
      for (uint32_t pr = c * (kPT / 32) + warp; pr < n_pairs; pr += nw)
        if (s.pair_flag[pr]) fallback_pair(p, s, pr, lane);
      if (!grid_sync(s.x, gen, p.summary)) return;
    }
    {
      // without the fallback an entry lacking statistics cannot be planned: it is reported
      unsigned long long cnt = 0;
      bool miss = false;
      for (uint64_t u = u0 + tid; u < u1; u += kPT) {
        cnt += score_unit(p, s, u).cand ? 1ull : 0ull;
        miss |= !p.fallback && p.nnz[(u % p.K) * p.n_blocks + u / p.K] == kNnzMissing;
      }
      if (__syncthreads_or(miss) && tid == 0) s.x[X_MISSING] = 1ull;
      cnt = block_sum<unsigned long long>(cnt);
      if (tid == 0) s.cta_a[c] = cnt;
    }
    if (!grid_sync(s.x, gen, p.summary)) return;

    // ---- B: stable compaction into (keys_a, order) ----
    {
      const unsigned long long before = block_sum_prefix(s.cta_a, c);
      Q = block_sum_prefix(s.cta_a, G);
      unsigned long long run = before;
      for (uint64_t t0 = u0; t0 < u1; t0 += kPT) {
        const uint64_t u = t0 + tid;
        Unit x = u < u1 ? score_unit(p, s, u) : Unit{false, 0u};
        uint32_t tot;
        const uint32_t pos = block_scan<uint32_t>(x.cand ? 1u : 0u, tot);
        if (x.cand) {
          if (kChecked && run + pos >= p.n_blocks * p.K) {  // checked build: a compaction slot past U
            atomicOr((unsigned long long*)&p.summary[S_ERR], (unsigned long long)kErrBounds);
          } else {
            s.keys_a[run + pos] = x.key;
            p.order[run + pos] = (uint32_t)u;
          }
        }
        run += tot;
      }
    }
    if (!grid_sync(s.x, gen, p.summary)) return;

    // ---- C: stable LSD radix sort, 8-bit digits ----
    uint32_t *kin = s.keys_a, *vin = p.order, *kout = s.keys_b, *vout = s.vals_b;
    slice(Q, q0, q1);
    for (uint32_t pass = 0; pass < 4; ++pass) {
      const uint32_t shift = 8u * pass;
      // C1: digit histogram of this CTA's slice
      s_run[tid] = 0;
      __syncthreads();
      for (uint64_t j = q0 + tid; j < q1; j += kPT) atomicAdd(&s_run[(kin[j] >> shift) & 255u], 1u);
      __syncthreads();
      s.hist[(uint64_t)tid * G + c] = s_run[tid];
      if (!grid_sync(s.x, gen, p.summary)) return;
      // C2: per digit, exclusive prefix over the CTAs (one warp per digit) and the total
      for (uint32_t d = c + warp * G; d < 256u; d += (kPT / 32) * G) {
        uint32_t* h = s.hist + (uint64_t)d * G;
        uint32_t carry = 0;
        for (uint32_t k0 = 0; k0 < G; k0 += 32) {
          const uint32_t v = k0 + lane < G ? h[k0 + lane] : 0u;
          uint32_t x = v;
  #pragma unroll
          for (int sh = 1; sh < 32; sh <<= 1) {
            const uint32_t y = __shfl_up_sync(0xFFFFFFFFu, x, sh);
            if ((int)lane >= sh) x += y;
          }
          if (k0 + lane < G) h[k0 + lane] = carry + x - v;
          carry += __shfl_sync(0xFFFFFFFFu, x, 31);
        }
        if (lane == 0) s.tot[d] = carry;
      }
      if (!grid_sync(s.x, gen, p.summary)) return;
      // C3: digit starts; skip the pass if one digit holds every key; stable scatter
      uint32_t total;
      const uint32_t t_d = s.tot[tid];
      const uint32_t start = block_scan<uint32_t>(t_d, total);
      const bool skip = __syncthreads_or(t_d == (uint32_t)Q && Q > 0) != 0 || Q == 0;
      if (skip) continue;  // uniform over the grid: every CTA reads the same totals
      s_run[tid] = start + s.hist[(uint64_t)tid * G + c];
      const uint32_t lt = (1u << lane) - 1u;
      for (uint64_t t0 = q0; t0 < q1; t0 += kPT) {
        for (int w = 0; w < kPT / 32; ++w) s_wcnt[w][tid] = 0;
        __syncthreads();
        const uint64_t j = t0 + tid;
        const bool valid = j < q1;
        const uint32_t key = valid ? kin[j] : 0u;
        const uint32_t val = valid ? vin[j] : 0u;
        const uint32_t d = valid ? ((key >> shift) & 255u) : 256u;
        const uint32_t peers = __match_any_sync(0xFFFFFFFFu, d);
        const uint32_t rank = __popc(peers & lt);
        if (valid && rank == 0) s_wcnt[warp][d] = __popc(peers);
        __syncthreads();
        {
          uint32_t acc = s_run[tid];
          for (int w = 0; w < kPT / 32; ++w) {
            const uint32_t cw = s_wcnt[w][tid];
            s_wcnt[w][tid] = acc;
            acc += cw;
          }
          s_run[tid] = acc;
        }
        __syncthreads();
        if (valid) {
          const uint32_t pos = s_wcnt[warp][d] + rank;
          kout[pos] = key;
          vout[pos] = val;
        }
        __syncthreads();  // every warp has read its offsets before the next tile clears them
      }
      if (!grid_sync(s.x, gen, p.summary)) return;
      uint32_t* t;
      t = kin, kin = kout, kout = t;
      t = vin, vin = vout, vout = t;
    }
    // the sorted units end in p.order, or in vals_b if an odd number of passes ran (a
    // uniform fact: every CTA made the same skip decisions)
    if (vin != p.order) {
      for (uint64_t j = q0 + tid; j < q1; j += kPT) p.order[j] = vin[j];
      if (!grid_sync(s.x, gen, p.summary)) return;
    }
    if (p.cache_order_out) {  // keep the order for later plans with the same operator
      for (uint64_t j = q0 + tid; j < q1; j += kPT) p.cache_order_out[j] = p.order[j];
      if (c == 0 && tid == 0) *p.cache_q_out = Q;
    }
  }
  const uint32_t* order = p.order;

  // ---- D: cost prefix in sorted order; the first position where it exceeds B ----
  {
    unsigned long long sum = 0;
    for (uint64_t j = q0 + tid; j < q1; j += kPT) sum += unit_cost(p, s, order[j]);
    sum = block_sum<unsigned long long>(sum);
    if (tid == 0) s.cta_b[c] = sum;
  }
  if (!grid_sync(s.x, gen, p.summary)) return;
  {
    unsigned long long run = block_sum_prefix(s.cta_b, c);
    const unsigned long long total_cost = block_sum_prefix(s.cta_b, G);
    if (c == 0 && tid == 0) s.x[X_TOTAL] = total_cost;
    for (uint64_t t0 = q0; t0 < q1; t0 += kPT) {
      const uint64_t j = t0 + tid;
      const unsigned long long cj = j < q1 ? unit_cost(p, s, order[j]) : 0ull;
      unsigned long long tot;
      const unsigned long long before = run + block_scan<unsigned long long>(cj, tot);
      if (j < q1 && before + cj > p.budget && before <= p.budget) {  // unique: prefixes only grow
        s.x[X_P] = j;
        s.x[X_PBP] = before;
      }
      run += tot;
    }
  }
  if (!grid_sync(s.x, gen, p.summary)) return;
  const unsigned long long P = s.x[X_P];
  const unsigned long long R0 = P == kNoP ? 0ull : p.budget - s.x[X_PBP];

  // ---- E: the tail after the first overflow ----
  if (P != kNoP) {
    {
      unsigned long long cnt = 0;
      for (uint64_t j = q0 + tid; j < q1; j += kPT) cnt += (j > P && unit_cost(p, s, order[j]) <= R0) ? 1ull : 0ull;
      cnt = block_sum<unsigned long long>(cnt);
      if (tid == 0) s.cta_a[c] = cnt;
    }
    if (!grid_sync(s.x, gen, p.summary)) return;
    const unsigned long long L = block_sum_prefix(s.cta_a, G);
    {
      unsigned long long run = block_sum_prefix(s.cta_a, c);
      unsigned long long cmin = ~0ull;
      for (uint64_t t0 = q0; t0 < q1; t0 += kPT) {
        const uint64_t j = t0 + tid;
        const unsigned long long cj = j < q1 ? unit_cost(p, s, order[j]) : ~0ull;
        const bool f = j < q1 && j > P && cj <= R0;
        uint32_t tot;
        const uint32_t pos = block_scan<uint32_t>(f ? 1u : 0u, tot);
        if (f) {
          s.tail_pos[run + pos] = (uint32_t)j;
          s.tail_cost[run + pos] = cj;
          cmin = cj < cmin ? cj : cmin;
        }
        run += tot;
      }
#pragma unroll
      for (int sh = 16; sh > 0; sh >>= 1) {
        const unsigned long long o = __shfl_xor_sync(0xFFFFFFFFu, cmin, sh);
        cmin = o < cmin ? o : cmin;
      }
      if (lane == 0 && cmin != ~0ull) atomicMin(&s.x[X_TAILMIN], cmin);
    }
    if (!grid_sync(s.x, gen, p.summary)) return;
    if (c == 0) {
      // greedy with skip over the compacted tail, in order, from shared memory; once R is
      // below the smallest tail cost nothing more can be taken
      const unsigned long long cmin = __ldcg(&s.x[X_TAILMIN]);
      unsigned long long R = R0;
      for (unsigned long long k0 = 0; k0 < L && R >= cmin; k0 += kTailChunk) {
        const uint32_t n = (uint32_t)min((unsigned long long)kTailChunk, L - k0);
        for (uint32_t k = tid; k < n; k += kPT) s_cost[k] = __ldcg(s.tail_cost + k0 + k);
        __syncthreads();
        if (warp == 0) {
          for (uint32_t b0 = 0; b0 < n && R >= cmin; b0 += 32) {
            const uint32_t k = b0 + lane;
            const unsigned long long ck = k < n ? s_cost[k] : ~0ull;
            uint32_t done = 0u;
            for (;;) {
              const uint32_t m = __ballot_sync(0xFFFFFFFFu, ck <= R) & ~done;
              if (m == 0u) break;
              const int f = __ffs(m) - 1;
              if ((int)lane == f) s.tailsel[s.tail_pos[k0 + k]] = 1;
              R -= __shfl_sync(0xFFFFFFFFu, ck, f);
              done = f == 31 ? 0xFFFFFFFFu : ((2u << f) - 1u);
            }
          }
          if (lane == 0) s_bcast[0] = R;
        }
        __syncthreads();
        R = s_bcast[0];
      }
      if (tid == 0) s.x[X_TAILSUM] = R0 - R;
    }
    if (!grid_sync(s.x, gen, p.summary)) return;
  }

  // ---- F: mask, set hash, count; then touched blocks and the digest (last CTA) ----
  {
    unsigned long long h = 0, n = 0;
    for (uint64_t j = q0 + tid; j < q1; j += kPT) {
      if ((P == kNoP || j < P) || s.tailsel[j]) {
        const uint32_t u = order[j];
        if (kChecked && (uint64_t)u >= p.n_blocks * p.K) {  // checked build: a unit id past U
          atomicOr((unsigned long long*)&p.summary[S_ERR], (unsigned long long)kErrBounds);
          continue;
        }
        const uint32_t b = u / p.K, i = u % p.K;
        const uint32_t t = p.fallback ? p.blk_tensor[b] : 0u;
        if (p.fallback && s.pair_flag[i * p.n_tensors + t]) {
          atomicOr(&s.sel_bits[t], 1u << i);  // every block of t gets bit i in the next pass
        } else {
          atomicOr(&p.mask[b], 1u << i);
        }
        h += splitmix64(u);
        ++n;
      }
    }
    h = block_sum<unsigned long long>(h);
    n = block_sum<unsigned long long>(n);
    if (tid == 0 && n) {
      atomicAdd((unsigned long long*)&p.summary[S_SETHASH], h);
      atomicAdd((unsigned long long*)&p.summary[S_NSEL], n);
    }
  }
  if (!grid_sync(s.x, gen, p.summary)) return;
  {
    uint64_t b0, b1;
    slice(p.n_blocks, b0, b1);
    unsigned long long t = 0;
    for (uint64_t b = b0 + tid; b < b1; b += kPT) {
      uint32_t m = p.mask[b];
      if (p.fallback) {
        const uint32_t sb = __ldcg(s.sel_bits + p.blk_tensor[b]);
        if (sb) {
          m |= sb;
          p.mask[b] = m;  // one thread per block in this pass
        }
      }
      t += m != 0u ? 1ull : 0ull;
    }
    t = block_sum<unsigned long long>(t);
    __shared__ bool last;
    if (tid == 0) {
      if (t) atomicAdd((unsigned long long*)&p.summary[S_TOUCHED], t);
      __threadfence();
      last = atomicAdd(&s.x[X_DONE], 1ull) == (unsigned long long)(G - 1);
    }
    __syncthreads();
    if (!last || tid != 0) return;
  }
  // the digest: FNV-1a 64 over the host-built prefix and C_hat, n_sel, set_hash
  __threadfence();
  volatile unsigned long long* sum = (volatile unsigned long long*)p.summary;
  const unsigned long long chat = P == kNoP ? s.x[X_TOTAL] : s.x[X_PBP] + s.x[X_TAILSUM];
  const unsigned long long nsel = sum[S_NSEL], sh = sum[S_SETHASH];
  uint64_t h = 14695981039346656037ull;
  for (uint32_t k = 0; k < p.hdr_prefix_len; ++k) {
    h ^= p.hdr_prefix[k];
    h *= 1099511628211ull;
  }
  const unsigned long long tail[3] = {chat, nsel, sh};
  for (int w = 0; w < 3; ++w)
    for (int k = 0; k < 8; ++k) {
      h ^= (tail[w] >> (8 * k)) & 0xFFu;
      h *= 1099511628211ull;
    }
  sum[S_CHAT] = chat;
  sum[S_NCAND] = Q;
  sum[S_DIGEST] = h;
  sum[S_ERR] = sum[S_ERR] | (unsigned long long)*p.index_err | (s.x[X_MISSING] ? (unsigned long long)kErrMissing : 0ull) |
               (s.x[X_BADORDER] ? (unsigned long long)kErrInternal : 0ull);
}

}  // namespace

size_t plan_scratch_bytes(uint64_t n_units, uint64_t n_pairs) { return carve(nullptr, n_units, n_pairs, nullptr); }

cudaError_t launch_plan(const PlanLaunch& p, void* scratch, cudaStream_t st) {
  const uint64_t U = (uint64_t)p.K * p.n_blocks;
  if (U > 0xFFFFFFFFull) return cudaErrorInvalidValue;
  const uint64_t n_pairs = p.fallback ? (uint64_t)p.K * p.n_tensors : 0ull;
  if (p.fallback && (!p.blk_tensor || !p.t_blk0 || n_pairs == 0)) return cudaErrorInvalidValue;
  Scratch s;
  carve(scratch, U, n_pairs, &s);
  int dev = 0, sms = 0, per_sm = 0;
  cudaError_t e;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
  if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, plan_kernel, kPT, 0)) != cudaSuccess) return e;
  // about 512 units per CTA (two tiles), at most one CTA per SM, all co-resident
  if (per_sm < 1) return cudaErrorInvalidConfiguration;
  uint64_t grid = (U + 511) / 512;
  const uint64_t cap = (uint64_t)sms;
  if (grid > cap) grid = cap;
  if (grid > kMaxGrid) grid = kMaxGrid;
  if (grid < 1) grid = 1;
  if ((e = launch_fill(s.x, 0, X_COUNT * sizeof(unsigned long long), st)) != cudaSuccess) return e;
  if (n_pairs && (e = launch_fill(s.pair_flag, 0, n_pairs * 4, st)) != cudaSuccess) return e;
  if (n_pairs && (e = launch_fill(s.sel_bits, 0, (size_t)p.n_tensors * 4, st)) != cudaSuccess) return e;
  PlanLaunch pc = p;
  void* args[] = {&pc, &s};
  if ((e = cudaLaunchCooperativeKernel((const void*)plan_kernel, dim3((unsigned)grid), dim3(kPT), args, 0, st)) !=
      cudaSuccess)
    return e;
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace mp
