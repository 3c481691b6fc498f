// Alg. 2 ExecuteMerge on the device: M_A[t,b] = M_0[t,b] + Psi_op(A_{.,t,b}, Delta_{.,t,b})
// (Eq. 4) for every block, reading only the experts the access mask selects.
//
// Pipeline (persistent CTAs, 2 or 3 per SM, 256 consumer threads + 1 producer warp):
//  * work unit = one chunk of a block (8 KiB for AVG/TA, 4 KiB for TIES/DARE); chunks are
//    handed out dynamically through a global counter, GRAB at a time;
//  * the producer warp takes a grab: its lanes load the chunks' block metadata (and, for
//    TIES, every expert's trim threshold) in parallel into shared memory, and the counter
//    value of the next grab is requested before this one is issued, so that no fill waits
//    on a global-memory round trip;
//  * lane 0 then walks each chunk's fills — the base chunk, then every selected expert's
//    chunk in ascending expert order — and streams each fill into the next slot of a ring
//    of NS shared-memory slots with one cp.async.bulk (TMA 1-D bulk copy), completing on
//    the slot's "full" mbarrier; it writes the slot's metadata (chunk, offset, length,
//    mask, TIES threshold) before arming the barrier;
//  * consumers take the slots in the same order: the base fill loads M_0 into registers,
//    each expert fill folds Delta_i into fp32 accumulators, the last fill of a chunk
//    writes the output with 16-byte streaming stores; every consumer thread arrives on the
//    slot's "empty" mbarrier as soon as it has read it;
//  * the bytes in flight are the ring (NS slots per CTA), independent of registers and of
//    how many experts a block selects.
// Per element, in the fixed ascending expert order:
//   AVG/TA: acc = fma(alpha_i, delta_i, acc)                          out = M_0 + acc
//   DARE:   delta_i kept by a Philox word >= T, scaled by sigma; then as AVG
//   TIES:   trimmed by tau_i; S, P, N, counts;  m = P/c+ | N/c- | 0;   out = fma(lambda, m, M_0)
//   renormalised AVG (App. A.1): as AVG with alpha_i / (sum of alpha over the experts that are
//           selected or have an exactly zero delta block, known from the catalog)
//   DARE-TIES: DARE's keep and rescale, then TIES's election and mean without trimming
// An omitted expert contributes exactly zero to every accumulator, so skipping it equals
// reading a zero-completed tuple (App. A.1) and it is never dereferenced; a chunk that
// selects no expert is M_0 plus the zero the operator adds, or, in the touched-only mode
// (Alg. 2 WriteBlockOrReference), not produced at all: the output keeps its contents there.
// Every mbarrier wait is bounded: on expiry the CTA records kErrTimeout, stops, waits
// (bounded) for its own copies in flight and returns.
#include <cuda_bf16.h>

#include <type_traits>

#include "mp_internal.cuh"
#include "philox.cuh"
#include "small_div.cuh"
#include "tma.cuh"

namespace mp {
namespace {

constexpr uint32_t kEnd = 0xFFFFFFFFu;

enum { OP_ADD = 0, OP_TIES = 1, OP_DARE = 2, OP_RENORM = 3, OP_DTIES = 4 };

// TIES and DARE-TIES share the sign election and disjoint mean (DARE and DARE-TIES share
// the random keep mask); AVG/TA and the renormalised AVG share the additive geometry
template <int OPC>
constexpr bool kTiesLike = OPC == OP_TIES || OPC == OP_DTIES;
template <int OPC>
constexpr bool kAddGeo = OPC == OP_ADD || OPC == OP_RENORM;

// slot geometry per operator.  The additive merges are bound by HBM: two CTAs per SM with a
// 96 KiB ring each (two 16-byte vectors per consumer thread and fill).  TIES, DARE and
// DARE-TIES spend more arithmetic per byte, so they run more warps per SM to hide latency
// (measured better than fewer consumer threads with more work each), with 4 KiB slots (one
// vector per consumer thread and fill, so that their state fits the register budget): TIES
// and DARE four CTAs per SM with a 44 KiB ring (their state fits 56 registers), DARE-TIES
// three with a 64 KiB ring (it would spill at 56).
template <int OPC>
struct Geo {
  static constexpr int kConsumers = 256;
  static constexpr int kThreads = kConsumers + 32;  // + one producer warp
  static constexpr int kCtasPerSm = kAddGeo<OPC> ? 2 : (OPC == OP_DTIES ? 3 : 4);
  static constexpr uint32_t kRingBytes = kAddGeo<OPC> ? 98304u : (OPC == OP_DTIES ? 65536u : 45056u);
  static constexpr uint32_t kSlotBytes = kAddGeo<OPC> ? 8192u : 4096u;  // one chunk of one checkpoint
  static constexpr int kSlots = (int)(kRingBytes / kSlotBytes);
  static constexpr uint32_t kGrab = 8;  // chunks taken per counter increment (<= 32)
};

struct SlotMeta {
  uint64_t off;   // element offset of the chunk in the flat buffers
  uint32_t q;     // chunk id, or kEnd
  uint32_t n;     // elements in the chunk
  uint32_t m;     // the block's access mask
  uint32_t aux;   // TIES: bits threshold of this (expert, trim group); renormalised AVG: the
                  // experts counted in the normaliser (selected or with a zero delta block)
};

// block metadata of one chunk of a grab, staged by the producer warp
struct ChunkMeta {
  uint64_t off;  // element offset of the chunk
  uint32_t n;    // elements (0: nothing to do)
  uint32_t m;    // access mask
};

template <int NS, uint32_t SB, uint32_t G>
struct __align__(128) Smem {
  uint8_t slot[NS][SB];
  SlotMeta meta[NS];
  ChunkMeta chunk[G];
  uint32_t thr[G][kMaxK];  // TIES: bits threshold of (chunk, expert)
  uint32_t zmask[G];       // renormalised AVG: experts whose delta block is exactly zero
  uint64_t full[NS];
  uint64_t empty[NS];
  unsigned long long realized[kMaxK];
  float2 ctab[kMaxK + 1];  // TIES: {c, RN(1/c)} for the counts c = 0..kMaxK (entry 0: {1, 1})
  int abort;
};

// packed fp32x2 arithmetic (two independent IEEE round-to-nearest operations per
// instruction): (d0, d1) = (a0 op b0, a1 op b1)
__device__ __forceinline__ void f2_sub(float a0, float a1, float b0, float b1, float& d0, float& d1) {
  asm("{\n .reg .b64 ra, rb, rd;\n mov.b64 ra, {%2, %3};\n mov.b64 rb, {%4, %5};\n sub.rn.f32x2 rd, ra, rb;\n"
      " mov.b64 {%0, %1}, rd;\n}"
      : "=f"(d0), "=f"(d1)
      : "f"(a0), "f"(a1), "f"(b0), "f"(b1));
}

__device__ __forceinline__ void f2_mul(float a0, float a1, float b0, float b1, float& d0, float& d1) {
  asm("{\n .reg .b64 ra, rb, rd;\n mov.b64 ra, {%2, %3};\n mov.b64 rb, {%4, %5};\n mul.rn.f32x2 rd, ra, rb;\n"
      " mov.b64 {%0, %1}, rd;\n}"
      : "=f"(d0), "=f"(d1)
      : "f"(a0), "f"(a1), "f"(b0), "f"(b1));
}

__device__ __forceinline__ void f2_add(float a0, float a1, float b0, float b1, float& d0, float& d1) {
  asm("{\n .reg .b64 ra, rb, rd;\n mov.b64 ra, {%2, %3};\n mov.b64 rb, {%4, %5};\n add.rn.f32x2 rd, ra, rb;\n"
      " mov.b64 {%0, %1}, rd;\n}"
      : "=f"(d0), "=f"(d1)
      : "f"(a0), "f"(a1), "f"(b0), "f"(b1));
}

// (d0, d1) = (a0 * b0 + c0, a1 * b1 + c1), each a single fused rounding
__device__ __forceinline__ void f2_fma(float a0, float a1, float b0, float b1, float c0, float c1, float& d0,
                                       float& d1) {
  asm("{\n .reg .b64 ra, rb, rc, rd;\n mov.b64 ra, {%2, %3};\n mov.b64 rb, {%4, %5};\n mov.b64 rc, {%6, %7};\n"
      " fma.rn.f32x2 rd, ra, rb, rc;\n mov.b64 {%0, %1}, rd;\n}"
      : "=f"(d0), "=f"(d1)
      : "f"(a0), "f"(a1), "f"(b0), "f"(b1), "f"(c0), "f"(c1));
}

// The TIES trim compares the 15-bit key bits(bf16_rne(|d|)) & 0x7FFF with tau.  For
// |d| >= 0 the key reaches tau >= 1 exactly when bits(|d|) >= (tau << 16) - 0x8000 +
// (tau & 1): the halfway point below tau rounds up to tau only when tau is even.  tau = 0
// keeps everything; tau = 0x8000 ("keep nothing") gives 0x7FFF8000, a NaN pattern, so a
// float compare against it is never true.
__host__ __device__ __forceinline__ uint32_t ties_bits_threshold(uint32_t tau) {
  return tau == 0u ? 0u : (tau << 16) - 0x8000u + (tau & 1u);
}

// One expert's contribution to an element's TIES tally, with predicated adds: the delta d
// is kept when |d| >= thr; a kept d goes into P (with count +1) when positive or into N
// (count + 0x10000) otherwise.  thr is at least the smallest subnormal, so a kept d is
// never zero and "not positive" means negative; one compare with two destination
// predicates splits the kept entries by sign.  A skipped add is the same as adding the +0
// of a trimmed entry: P and N are never -0, so +0 leaves them unchanged.  The elected
// sign is that of P + N (compared exactly at the end).
__device__ __forceinline__ void ties_tally(float d, float thr, float& P, float& N, uint32_t& cnt) {
  asm("{\n"
      " .reg .pred pk, pp, pn;\n"
      " .reg .f32 ad;\n"
      " abs.f32 ad, %3;\n"
      " setp.ge.f32 pk, ad, %4;\n"
      " setp.gt.and.f32 pp|pn, %3, 0f00000000, pk;\n"
      " @pp add.rn.f32 %0, %0, %3;\n"
      " @pn add.rn.f32 %1, %1, %3;\n"
      " @pp add.u32 %2, %2, 1;\n"
      " @pn add.u32 %2, %2, 65536;\n"
      "}\n"
      : "+f"(P), "+f"(N), "+r"(cnt)
      : "f"(d), "f"(thr));
}

// One expert's contribution to an element's DARE-TIES tally: the rescaled delta s enters
// when its keep word kw (the 16-bit word in the upper half of a 32-bit register) reaches
// T16 and s is nonzero, into P (count +1) when positive or N (count + 0x10000) when
// negative; no magnitude trim.  A dropped or zero entry adds nothing (the +0 of Eq. 4's
// dropped delta leaves P and N unchanged).
__device__ __forceinline__ void dties_tally(float s, uint32_t kw, uint32_t T16, float& P, float& N, uint32_t& cnt) {
  asm("{\n"
      " .reg .pred pk, pp, pn;\n"
      " setp.ge.u32 pk, %4, %5;\n"
      " setp.gt.and.f32 pp, %3, 0f00000000, pk;\n"
      " setp.lt.and.f32 pn, %3, 0f00000000, pk;\n"
      " @pp add.rn.f32 %0, %0, %3;\n"
      " @pn add.rn.f32 %1, %1, %3;\n"
      " @pp add.u32 %2, %2, 1;\n"
      " @pn add.u32 %2, %2, 65536;\n"
      "}\n"
      : "+f"(P), "+f"(N), "+r"(cnt)
      : "f"(s), "r"(kw), "r"(T16));
}

// bf16 -> fp32: the upper element by a mask, the lower one moved up by a multiply (which runs
// on the FMA pipe and leaves the ALU pipe to the compares)
template <bool BF16>
__device__ __forceinline__ void unpack(const uint4 r, float* x) {
  if constexpr (BF16) {
    x[0] = __uint_as_float(r.x * 65536u);
    x[1] = __uint_as_float(r.x & 0xFFFF0000u);
    x[2] = __uint_as_float(r.y * 65536u);
    x[3] = __uint_as_float(r.y & 0xFFFF0000u);
    x[4] = __uint_as_float(r.z * 65536u);
    x[5] = __uint_as_float(r.z & 0xFFFF0000u);
    x[6] = __uint_as_float(r.w * 65536u);
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

// the raw 16-byte vector at element k0 of a fill, as read_vec reads it (zeros past the chunk)
template <bool BF16>
__device__ __forceinline__ uint4 read_raw(const uint8_t* slot, const void* gsrc, uint64_t off, uint32_t k0,
                                          uint32_t n, uint32_t n_tma) {
  constexpr uint32_t V = BF16 ? 8u : 4u;
  if (k0 + V <= n_tma) return *reinterpret_cast<const uint4*>(slot + k0 * (BF16 ? 2u : 4u));
  uint32_t w[4] = {0u, 0u, 0u, 0u};
#pragma unroll
  for (uint32_t e = 0; e < V; ++e) {
    if (k0 + e < n) {
      if constexpr (BF16) w[e >> 1] |= (uint32_t)(static_cast<const uint16_t*>(gsrc)[off + k0 + e]) << (16u * (e & 1u));
      else w[e] = static_cast<const uint32_t*>(gsrc)[off + k0 + e];
    }
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}

// elements 2k and 2k + 1 of a raw vector as fp32 (k is a compile-time index)
template <bool BF16, int k>
__device__ __forceinline__ void pair_of(const uint4 r, float& a, float& b) {
  if constexpr (BF16) {
    const uint32_t w = k == 0 ? r.x : (k == 1 ? r.y : (k == 2 ? r.z : r.w));
    a = __uint_as_float(w * 65536u);
    b = __uint_as_float(w & 0xFFFF0000u);
  } else {
    a = __uint_as_float(k == 0 ? r.x : r.z);
    b = __uint_as_float(k == 0 ? r.y : r.w);
  }
}

// the tail loops are unrolled over the vector with a predicate, so that h and y stay in
// registers (a loop bounded by navail would index them at run time, through local memory)
template <bool BF16>
__device__ __forceinline__ void store_vec(void* ptr, uint64_t elem, uint32_t navail, const float* y) {
  constexpr uint32_t V = BF16 ? 8u : 4u;
  if constexpr (BF16) {
    // two elements per conversion, each rounded to nearest-even: element 2k in the low half
    uint32_t w[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const __nv_bfloat162 h2 = __floats2bfloat162_rn(y[2 * k], y[2 * k + 1]);
      w[k] = *reinterpret_cast<const uint32_t*>(&h2);
    }
    if (navail >= V) {
      __stcs(reinterpret_cast<uint4*>(static_cast<char*>(ptr) + elem * 2u), make_uint4(w[0], w[1], w[2], w[3]));
    } else {
#pragma unroll
      for (uint32_t e = 0; e < V; ++e)
        if (e < navail) static_cast<uint16_t*>(ptr)[elem + e] = (uint16_t)(w[e >> 1] >> (16u * (e & 1u)));
    }
  } else {
    if (navail >= V) {
      __stcs(reinterpret_cast<float4*>(static_cast<char*>(ptr) + elem * 4u), make_float4(y[0], y[1], y[2], y[3]));
    } else {
#pragma unroll
      for (uint32_t e = 0; e < V; ++e)
        if (e < navail) static_cast<float*>(ptr)[elem + e] = y[e];
    }
  }
}

// Checked build: a chunk's block must lie in the launch's block range before the block table
// is read for it, and the chunk (its elements, buffers, alignment, experts and TIES trim
// group) must pass chunk_in_bounds before anything is copied; a failure is recorded in the
// call's error word and the chunk is skipped.  Both are constant true in the default build.
__device__ __forceinline__ bool checked_block(const MergeLaunch& p, uint64_t b) {
  if constexpr (!kChecked) return true;
  if (b >= p.b_begin && b < p.b_end && b < p.n_blocks) return true;
  atomicOr(p.err, kErrBounds);
  return false;
}

template <bool TIES>
__device__ __forceinline__ bool checked_chunk(const MergeLaunch& p, uint64_t b, const ChunkMeta& cm, uint32_t grp,
                                              uint32_t es) {
  if constexpr (!kChecked) return true;
  if (cm.n == 0u) return true;
  if ((!TIES || grp < p.n_groups) &&
      chunk_in_bounds(b, p.b_begin, p.b_end, p.blk_off[b], p.blk_len[b], cm.off, cm.n, cm.m, p.K, es,
                      p.expert_origin, p.ext))
    return true;
  atomicOr(p.err, kErrBounds);
  return false;
}

// DARE keep words of the vector at flat element j0 for expert i: element j keeps its delta
// iff 16-bit word j mod 8 of the Philox4x32-10 output for counter j / 8 is >= T.  A bf16
// vector is exactly the 8 words of one call (chunk and tensor offsets are multiples of 8
// elements); an fp32 vector is half of one.  Word j mod 8 of element j is returned in the
// upper half of a 32-bit register: the upper word as it stands, the lower one moved up by a
// multiply (FMA pipe; the ALU pipe is the busy one); it is kept iff that register >= T << 16.
template <bool BF16>
__device__ __forceinline__ void dare_keep_words(const MergeLaunch& p, uint32_t i, uint64_t j0,
                                                uint32_t (&kw)[BF16 ? 8 : 4]) {
  constexpr int V = BF16 ? 8 : 4;
  const uint64_t g = j0 >> 3;
  const Philox4 r = philox4x32_10_rk((uint32_t)g, (uint32_t)(g >> 32), i, 0x44415245u, p.dare_rk);
  const uint32_t e0 = (uint32_t)(j0 & 7u);  // 0 for bf16; 0 or 4 for fp32
#pragma unroll
  for (int e = 0; e < V; ++e) {
    const uint32_t wd = BF16 ? r.w[e >> 1] : (e0 ? r.w[2 + (e >> 1)] : r.w[e >> 1]);
    kw[e] = (e & 1) ? wd : wd * 65536u;
  }
}

template <bool BF16, int OPC>
__global__ void __launch_bounds__(Geo<OPC>::kThreads, Geo<OPC>::kCtasPerSm)
    merge_tma_kernel(const MergeLaunch p, uint32_t cpb, uint64_t n_chunks, unsigned long long* work) {
  constexpr int kConsumers = Geo<OPC>::kConsumers;
  constexpr uint32_t ES = BF16 ? 2u : 4u;
  constexpr uint32_t SB = Geo<OPC>::kSlotBytes;
  constexpr int kSlots = Geo<OPC>::kSlots;
  constexpr uint32_t G = Geo<OPC>::kGrab;
  constexpr uint32_t CH = SB / ES;  // elements per chunk
  constexpr int V = BF16 ? 8 : 4;
  constexpr int VPT = (int)(CH / (kConsumers * V));  // vectors per consumer thread per chunk
  static_assert(CH == (uint32_t)(kConsumers * VPT * V), "chunk geometry");
  extern __shared__ __align__(128) uint8_t smem_raw[];
  Smem<kSlots, SB, G>& S = *reinterpret_cast<Smem<kSlots, SB, G>*>(smem_raw);
  const uint32_t tid = threadIdx.x, warp = tid >> 5, lane = tid & 31u;
  volatile int* abort_flag = &S.abort;
  const uint32_t wl = wait_limit_of(p.wait_limit);

  if (tid == 0) {
    for (int s = 0; s < kSlots; ++s) {
      mbar_init(&S.full[s], 1);
      mbar_init(&S.empty[s], kConsumers);  // every consumer thread arrives
    }
    S.abort = 0;
    mbar_fence_init();
  }
  if (tid < (uint32_t)kMaxK) S.realized[tid] = 0;
  if (tid <= (uint32_t)kMaxK) {
    const float c = tid == 0 ? 1.0f : (float)tid;
    S.ctab[tid] = make_float2(c, __fdiv_rn(1.0f, c));
  }
  __syncthreads();

  if (warp == kConsumers / 32) {
    // ---------------- producer ----------------
    uint32_t fill = 0;
    bool ok = true;
    // lane 0 arms slot `fill` with the given chunk data and starts its bulk copy
    auto produce = [&](uint32_t q, uint64_t off, uint32_t n, uint32_t m, uint32_t aux,
                       const char* src_row, uint32_t bytes) -> bool {
      const uint32_t s = fill % kSlots, r = fill / kSlots;
      if (fill == 0 && p.stall) {  // test hook: slot 0 is never armed, so its wait runs out
        ++fill;
        return true;
      }
      if (r > 0 && !mbar_wait<true>(&S.empty[s], (r - 1) & 1u, abort_flag, wl)) return false;
      if (r > 0) fence_proxy_async_smem();
      S.meta[s].off = off;
      S.meta[s].q = q;
      S.meta[s].n = n;
      S.meta[s].m = m;
      S.meta[s].aux = aux;
      mbar_arrive_expect_tx(&S.full[s], bytes);
      if (bytes) tma_load_1d(S.slot[s], src_row, bytes, &S.full[s]);
      ++fill;
      return true;
    };
    unsigned long long q_next = 0;
    if (lane == 0) q_next = atomicAdd(work, (unsigned long long)G);
    for (;;) {
      const unsigned long long q0 = __shfl_sync(0xFFFFFFFFu, q_next, 0);
      if (q0 >= n_chunks || !ok) break;
      if (lane == 0) q_next = atomicAdd(work, (unsigned long long)G);  // used by the next grab
      // lanes c < G: metadata of chunk q0 + c
      uint32_t grp = 0;
      uint64_t bq = 0;  // block of chunk q0 + lane
      if (lane < G) {
        const unsigned long long q = q0 + lane;
        ChunkMeta cm{0, 0, 0};
        if (q < n_chunks && checked_block(p, p.b_begin + q / cpb)) {
          const uint64_t b = p.b_begin + q / cpb;
          bq = b;
          const uint32_t start = (uint32_t)(q % cpb) * CH;
          const uint32_t len = p.blk_len[b];
          cm.off = p.blk_off[b] + start;
          cm.m = p.mask[b];
          cm.n = start < len ? min(CH, len - start) : 0u;
          if (p.touched_only && cm.m == 0u) cm.n = 0u;  // left as it is: a reference to M_0
          if constexpr (OPC == OP_TIES) grp = p.blk_group[b];
          if (!checked_chunk<OPC == OP_TIES>(p, b, cm, grp, ES)) cm.n = 0u, grp = 0u;
        }
        S.chunk[lane] = cm;
      }
      if constexpr (OPC == OP_TIES) {
        // lane i < K: the trim thresholds of expert i for every chunk of the grab, at least
        // the smallest subnormal (a zero delta is never kept: it would add nothing)
#pragma unroll
        for (uint32_t c = 0; c < G; ++c) {
          const uint32_t g = __shfl_sync(0xFFFFFFFFu, grp, c);
          if (lane < p.K) S.thr[c][lane] = max(ties_bits_threshold(p.tau[(uint64_t)lane * p.n_groups + g]), 1u);
        }
      }
      if constexpr (OPC == OP_RENORM) {
        // lane i < K: is expert i's delta block exactly zero (catalog nnz = 0)?  Such an
        // expert is counted in the normaliser without being read.
#pragma unroll
        for (uint32_t c = 0; c < G; ++c) {
          const uint64_t b = __shfl_sync(0xFFFFFFFFu, bq, c);
          const bool z = lane < p.K && p.nnz[(uint64_t)lane * p.n_blocks + b] == 0u;
          const uint32_t zb = __ballot_sync(0xFFFFFFFFu, z);
          if (lane == 0) S.zmask[c] = zb;
        }
      }
      __syncwarp();
      if (lane == 0) {
        const uint32_t nq = (uint32_t)min((unsigned long long)G, n_chunks - q0);
        for (uint32_t c = 0; c < nq && ok; ++c) {
          const ChunkMeta cm = S.chunk[c];
          if (cm.n == 0) continue;
          const uint32_t q = (uint32_t)(q0 + c);
          const uint32_t bytes = (cm.n * ES) & ~15u;
          const uint32_t aux0 = OPC == OP_RENORM ? (cm.m | S.zmask[c]) : 0u;
          ok = produce(q, cm.off, cm.n, cm.m, aux0, static_cast<const char*>(p.base) + cm.off * ES, bytes);
          for (uint32_t mm = cm.m; ok && mm; mm &= mm - 1) {
            const uint32_t i = __ffs(mm) - 1;
            // DARE-TIES keeps every nonzero rescaled delta: threshold = the smallest subnormal
            ok = produce(q, cm.off, cm.n, cm.m, OPC == OP_TIES ? S.thr[c][i] : 1u,
                         static_cast<const char*>(p.experts.p[i]) + (cm.off - p.expert_origin) * ES, bytes);
            S.realized[i] += (unsigned long long)cm.n * ES;
          }
        }
      }
      ok = __shfl_sync(0xFFFFFFFFu, ok, 0);
      __syncwarp();
    }
    if (lane == 0) {
      if (ok) ok = produce(kEnd, 0, 0, 0, 0u, nullptr, 0);
      if (!ok) {
        atomicOr(p.err, kErrTimeout);
        S.abort = 1;
      }
      // drain: the last fill of every slot must have landed before the CTA may exit
      for (uint32_t s = 0; s < (uint32_t)kSlots && s < fill; ++s) {
        const uint32_t last = fill - 1 - ((fill - 1 + kSlots - s) % kSlots);
        if (last == 0 && p.stall) continue;  // never armed: nothing in flight
        mbar_wait_drain(&S.full[s], (last / kSlots) & 1u);
      }
      for (uint32_t i = 0; i < p.K; ++i)
        if (S.realized[i])
          atomicAdd(p.realized + (uint64_t)(blockIdx.x % kCounterSlots) * p.K + i, S.realized[i]);
    }
    return;
  }

  // ---------------- consumers ----------------
  float x0[VPT][V], acc[VPT][V], Pp[VPT][V], Nn[VPT][V];
  uint32_t cnt[VPT][V];  // TIES: positive count | negative count << 16
  uint64_t off = 0;
  uint32_t n = 0, n_tma = 0, remaining = 0;
  uint32_t m_chunk = 0, m_rest = 0;  // the chunk's access mask; its experts still to come
  float s_sel = 0.0f;  // renormalised AVG: sum of the counted experts' alpha (ascending)
  // DARE keep decisions of the vector's elements (dare_keep_words)
  auto dare_words = [&](uint32_t i, uint64_t j0, uint32_t (&kw)[V]) { dare_keep_words<BF16>(p, i, j0, kw); };
  auto dare_kept = [&](uint32_t i, uint64_t j0, bool (&kept)[V]) {
    uint32_t kw[V];
    dare_words(i, j0, kw);
#pragma unroll
    for (int e = 0; e < V; ++e) kept[e] = kw[e] >= p.dare_T16;
  };
  for (uint32_t fill = 0;; ++fill) {
    const uint32_t s = fill % kSlots, r = fill / kSlots;
    if (!warp_wait<true>(&S.full[s], r & 1u, abort_flag, wl)) {
      atomicOr(p.err, kErrTimeout);
      S.abort = 1;
      break;
    }
    const uint8_t* slot = S.slot[s];
    // fills come as the base chunk, then its selected experts in ascending order: only a
    // base fill needs the slot's metadata; an expert fill's expert is the next set bit
    if (remaining == 0) {
      const SlotMeta mt = S.meta[s];
      if (mt.q == kEnd) break;
      off = mt.off;
      n = mt.n;
      n_tma = ((n * ES) & ~15u) / ES;
      m_chunk = m_rest = mt.m;
      remaining = __popc(mt.m);
      if constexpr (OPC == OP_RENORM) {
        s_sel = 0.0f;
        for (uint32_t mm = mt.aux; mm; mm &= mm - 1) s_sel = __fadd_rn(s_sel, p.alpha[__ffs(mm) - 1]);
      }
#pragma unroll
      for (int u = 0; u < VPT; ++u) {
        const uint32_t k0 = (tid + (uint32_t)u * kConsumers) * V;
        read_vec<BF16>(slot, p.base, off, k0, n, n_tma, x0[u]);
        if (remaining) {
#pragma unroll
          for (int e = 0; e < V; ++e) {
            acc[u][e] = 0.0f;
            Pp[u][e] = 0.0f;
            Nn[u][e] = 0.0f;
            cnt[u][e] = 0u;
          }
        }
      }
    } else {
      const uint32_t i = __ffs(m_rest) - 1;
      m_rest &= m_rest - 1;
      const void* src = p.experts.p[i];
      if constexpr (kTiesLike<OPC>) {
        // TIES: trim test on the magnitude's bits: key(|d|) >= tau exactly when bits(|d|) >=
        // the producer's threshold (a NaN pattern, never true, when nothing is kept).
        // DARE-TIES: the delta is rescaled, and it enters when its keep word passes and the
        // result is nonzero (no magnitude trim).
        const float thr = __uint_as_float(OPC == OP_TIES ? S.meta[s].aux : 1u);
#pragma unroll
        for (int u = 0; u < VPT; ++u) {
          const uint32_t k0 = (tid + (uint32_t)u * kConsumers) * V;
          float xe[V];
          read_vec<BF16>(slot, src, off - p.expert_origin, k0, n, n_tma, xe);
          uint32_t kw[V];
          if constexpr (OPC == OP_DTIES) dare_words(i, off + k0, kw);
#pragma unroll
          for (int e = 0; e < V; e += 2) {
            // the deltas of an element pair in one packed fp32x2 subtract
            float d0, d1;
            f2_sub(xe[e], xe[e + 1], x0[u][e], x0[u][e + 1], d0, d1);
            if constexpr (OPC == OP_DTIES) {
              float s0, s1;
              f2_mul(d0, d1, p.sigma, p.sigma, s0, s1);
              dties_tally(s0, kw[e], p.dare_T16, Pp[u][e], Nn[u][e], cnt[u][e]);
              dties_tally(s1, kw[e + 1], p.dare_T16, Pp[u][e + 1], Nn[u][e + 1], cnt[u][e + 1]);
            } else {
              ties_tally(d0, thr, Pp[u][e], Nn[u][e], cnt[u][e]);
              ties_tally(d1, thr, Pp[u][e + 1], Nn[u][e + 1], cnt[u][e + 1]);
            }
          }
        }
      } else {
        // renormalised AVG: beta_i = alpha_i / (sum of the selected alpha), one IEEE division
        const float a = OPC == OP_RENORM ? __fdiv_rn(p.alpha[i], s_sel) : p.alpha[i];
#pragma unroll
        for (int u = 0; u < VPT; ++u) {
          const uint32_t k0 = (tid + (uint32_t)u * kConsumers) * V;
          float xe[V];
          read_vec<BF16>(slot, src, off - p.expert_origin, k0, n, n_tma, xe);
          bool kept[V];
          if constexpr (OPC == OP_DARE) dare_kept(i, off + k0, kept);
#pragma unroll
          for (int e = 0; e < V; e += 2) {
            float d0, d1;
            f2_sub(xe[e], xe[e + 1], x0[u][e], x0[u][e + 1], d0, d1);
            if constexpr (OPC == OP_DARE) {  // a dropped entry is omitted from the sum
              float s0, s1;
              f2_mul(d0, d1, p.sigma, p.sigma, s0, s1);
              if (kept[e]) acc[u][e] = __fmaf_rn(a, s0, acc[u][e]);
              if (kept[e + 1]) acc[u][e + 1] = __fmaf_rn(a, s1, acc[u][e + 1]);
            } else {
              f2_fma(a, a, d0, d1, acc[u][e], acc[u][e + 1], acc[u][e], acc[u][e + 1]);
            }
          }
        }
      }
      --remaining;
    }
    mbar_arrive(&S.empty[s]);  // every consumer thread: its own reads of the slot are done
    if (remaining == 0) {
#pragma unroll
      for (int u = 0; u < VPT; ++u) {
        // every lane of the warp runs the finalisation (a lane past the chunk's end holds
        // zeros) so that the warp vote below is reached by all of them; only the store is
        // limited to the chunk
        const uint32_t k0 = (tid + (uint32_t)u * kConsumers) * V;
        const bool live = k0 < n;
        float y[V];
        if (m_chunk == 0) {  // uniform over the warp
          // no expert selected: every accumulator is +0, so the output is M_0 plus the
          // zero the operator adds (lambda * +0 for TIES, +0 otherwise)
          const float z = kTiesLike<OPC> ? __fmul_rn(p.lambda, 0.0f) : 0.0f;
#pragma unroll
          for (int e = 0; e < V; ++e) y[e] = __fadd_rn(x0[u][e], z);
          if (live) store_vec<BF16>(p.out, off + k0, n - k0, y);
          continue;
        }
        if constexpr (kTiesLike<OPC>) {
          // one division per element: the mean of the entries whose sign was elected, the
          // sign of P + N taken exactly as P > -N or P < -N (then that side holds at least
          // one entry, so c >= 1; otherwise +0 / 1 = +0).  The rare numerators that need the
          // IEEE division take it under one warp vote.
          auto num_c = [&](int e, float& num, uint32_t& c) {
            const bool pos = Pp[u][e] > -Nn[u][e], any = Pp[u][e] != -Nn[u][e];
            num = any ? (pos ? Pp[u][e] : Nn[u][e]) : 0.0f;
            c = any ? (pos ? (cnt[u][e] & 0xFFFFu) : (cnt[u][e] >> 16)) : 0u;
          };
          bool exact = false;
#pragma unroll
          for (int e = 0; e < V; ++e) {
            float num;
            uint32_t c;
            num_c(e, num, c);
            const float2 cy = S.ctab[c];
            y[e] = div_small_fast(num, cy.x, cy.y);
            exact = exact || div_small_needs_ieee(num);
          }
          if (__any_sync(0xFFFFFFFFu, exact)) {
#pragma unroll
            for (int e = 0; e < V; ++e) {
              float num;
              uint32_t c;
              num_c(e, num, c);
              if (div_small_needs_ieee(num)) y[e] = __fdiv_rn(num, S.ctab[c].x);
            }
          }
#pragma unroll
          for (int e = 0; e < V; ++e) y[e] = __fmaf_rn(p.lambda, y[e], x0[u][e]);
        } else {
#pragma unroll
          for (int e = 0; e < V; ++e) y[e] = __fadd_rn(x0[u][e], acc[u][e]);
        }
        if (live) store_vec<BF16>(p.out, off + k0, n - k0, y);
      }
    }
  }
}

// ---------------- TIES (at most 8 experts) and DARE (at most 16): whole-chunk consumers ----------------
//
// The same TMA ring, but a chunk (its base fill and its selected experts' fills, which sit in
// consecutive ring slots) is published as one unit: one "full" mbarrier per chunk counts the
// bytes of all its fills, one "empty" mbarrier per chunk counts the consumers' releases.
// A consumer thread waits once per chunk, folds every selected expert of its vector in the
// fixed ascending order while all of them are in shared memory, releases the chunk and only
// then finalises: the per-element state (M_0 and P, N, counts for TIES, the accumulator for
// DARE) lives for one chunk and the per-fill waits, arrivals and metadata reads of the
// streaming kernel disappear.  The ring must hold every fill of one chunk (1 + K slots), so
// this kernel serves TIES with K <= 8 and DARE with K <= 16; the streaming kernel above
// serves the other operators and larger expert counts.
constexpr uint32_t kTcSlotBytes = 4096u;
constexpr uint32_t kTcMaxK = 16;

// ring slots and CTAs per SM by expert count: K <= 4 holds two chunks of 5 fills in 11
// slots at four CTAs per SM (three for DARE-TIES, whose state needs more registers); K <= 8
// two chunks of 9 fills in 18 slots at three; K <= 16 one chunk of 17 fills, or several of
// the usual few selected experts, in 17 slots at three
template <int OPC, int KC>
struct TcGeo {
  static constexpr int kSlots = KC <= 4 ? 11 : (KC <= 8 ? 18 : 17);
  static constexpr int kCtasPerSm = KC <= 4 && OPC != OP_DTIES ? 4 : 3;
  static constexpr int kConsumers = 256;
  static constexpr int kThreads = kConsumers + 32;
  static constexpr uint32_t kGrab = 8;
};

template <int KC>
struct TcEntry {
  uint64_t off;          // element offset of the chunk
  uint32_t q;            // chunk id, or kEnd
  uint32_t n;            // elements in the chunk
  uint32_t m;            // the block's access mask
  uint32_t s0;           // ring slot of the base fill; expert fill j sits in slot s0 + 1 + j (mod NS)
  uint32_t nsel;         // selected experts
  uint32_t fast;         // 1: every selected threshold is >= 2^-100 (no numerator needs the IEEE division)
  float thr[KC];         // TIES: trim thresholds (as floats) in fill order
  uint8_t ex[KC];        // the selected experts in fill order
};

// sized by the expert count KC so that three CTAs of 18 slots fit one SM's 228 KB
template <int NS, uint32_t G, int KC>
struct __align__(128) TcSmem {
  uint8_t slot[NS][kTcSlotBytes];
  TcEntry<KC> ce[NS];
  ChunkMeta chunk[G];
  uint32_t thr[G][KC];  // bits threshold of (chunk of the grab, expert)
  uint64_t full[NS];
  uint64_t empty[NS];
  unsigned long long realized[KC];
  float2 ntab[kTcMaxK + 1];  // {-c, RN(1/c)} for the counts c = 0..16 (entry 0: {-1, 1})
  uint32_t nf[NS];           // producer only: fills held by the chunk of each entry
  int abort;
};

template <bool BF16, int OPC, int KC>
__global__ void __launch_bounds__(TcGeo<OPC, KC>::kThreads, TcGeo<OPC, KC>::kCtasPerSm)
    merge_chunk_kernel(const MergeLaunch p, uint32_t cpb, uint64_t n_chunks, unsigned long long* work) {
  static_assert(OPC == OP_TIES || OPC == OP_DARE || OPC == OP_DTIES, "whole-chunk consumers: TIES, DARE, DARE-TIES");
  // the packed counts C = 2^23 + c+ + 2^CB c-: CB = 4 bits for up to 8 experts, 5 for 16
  constexpr uint32_t CB = KC <= 8 ? 4u : 5u;
  constexpr int NS = TcGeo<OPC, KC>::kSlots;
  constexpr int kConsumers = TcGeo<OPC, KC>::kConsumers;
  constexpr uint32_t G = TcGeo<OPC, KC>::kGrab;
  constexpr uint32_t ES = BF16 ? 2u : 4u;
  constexpr uint32_t CH = kTcSlotBytes / ES;  // elements per chunk
  constexpr int V = BF16 ? 8 : 4;
  static_assert(CH == (uint32_t)(kConsumers * V), "one vector per consumer thread and chunk");
  static_assert(NS >= KC + 1, "the ring holds every fill of a chunk");
  extern __shared__ __align__(128) uint8_t smem_raw[];
  TcSmem<NS, G, KC>& S = *reinterpret_cast<TcSmem<NS, G, KC>*>(smem_raw);
  const uint32_t tid = threadIdx.x, warp = tid >> 5, lane = tid & 31u;
  volatile int* abort_flag = &S.abort;
  const uint32_t wl = wait_limit_of(p.wait_limit);

  if (tid == 0) {
    for (int s = 0; s < NS; ++s) {
      mbar_init(&S.full[s], 1);
      mbar_init(&S.empty[s], kConsumers);  // every consumer thread arrives once per chunk
    }
    S.abort = 0;
    mbar_fence_init();
  }
  if (tid < (uint32_t)KC) S.realized[tid] = 0;
  if (tid <= kTcMaxK) {
    const float c = tid == 0 ? 1.0f : (float)tid;
    S.ntab[tid] = make_float2(-c, __fdiv_rn(1.0f, c));
  }
  __syncthreads();

  if (warp == kConsumers / 32) {
    // ---------------- producer ----------------
    uint32_t fill = 0;  // ring slots used so far (monotonic)
    uint32_t seq = 0;   // chunks published
    uint32_t head = 0;  // oldest published chunk not yet seen released
    uint32_t used = 0;  // slots held by chunks head .. seq - 1
    bool ok = true;
    // lane 0: wait until entry seq % NS is free and nfill slots are free; chunks are
    // released in order, so the oldest one is the next to free its slots
    auto reserve = [&](uint32_t nfill) -> bool {
      while (seq - head >= (uint32_t)NS || used + nfill > (uint32_t)NS) {
        const uint32_t he = head % NS;
        if (!mbar_wait<true>(&S.empty[he], (head / NS) & 1u, abort_flag, wl)) return false;
        used -= S.nf[he];
        ++head;
      }
      return true;
    };
    unsigned long long q_next = 0;
    if (lane == 0) q_next = atomicAdd(work, (unsigned long long)G);
    for (;;) {
      const unsigned long long q0 = __shfl_sync(0xFFFFFFFFu, q_next, 0);
      if (q0 >= n_chunks || !ok) break;
      if (lane == 0) q_next = atomicAdd(work, (unsigned long long)G);  // used by the next grab
      uint32_t grp = 0;
      if (lane < G) {
        const unsigned long long q = q0 + lane;
        ChunkMeta cm{0, 0, 0};
        if (q < n_chunks && checked_block(p, p.b_begin + q / cpb)) {
          const uint64_t b = p.b_begin + q / cpb;
          const uint32_t start = (uint32_t)(q % cpb) * CH;
          const uint32_t len = p.blk_len[b];
          cm.off = p.blk_off[b] + start;
          cm.m = p.mask[b];
          cm.n = start < len ? min(CH, len - start) : 0u;
          if (p.touched_only && cm.m == 0u) cm.n = 0u;  // left as it is: a reference to M_0
          if (OPC == OP_TIES) grp = p.blk_group[b];
          if (!checked_chunk<OPC == OP_TIES>(p, b, cm, grp, ES)) cm.n = 0u, grp = 0u;
        }
        S.chunk[lane] = cm;
      }
      if constexpr (OPC == OP_TIES) {
        // lane i < K: the trim thresholds of expert i for every chunk of the grab, at least the
        // smallest subnormal (a zero delta is never kept: it would add nothing)
#pragma unroll
        for (uint32_t c = 0; c < G; ++c) {
          const uint32_t g = __shfl_sync(0xFFFFFFFFu, grp, c);
          if (lane < p.K) S.thr[c][lane] = max(ties_bits_threshold(p.tau[(uint64_t)lane * p.n_groups + g]), 1u);
        }
      }
      __syncwarp();
      if (lane == 0) {
        const uint32_t nq = (uint32_t)min((unsigned long long)G, n_chunks - q0);
        for (uint32_t c = 0; c < nq && ok; ++c) {
          const ChunkMeta cm = S.chunk[c];
          if (cm.n == 0) continue;
          const uint32_t nsel = __popc(cm.m);
          if (!(ok = reserve(1u + nsel))) break;
          if (fill >= (uint32_t)NS) fence_proxy_async_smem();  // slots the consumers have read are refilled
          const uint32_t e = seq % NS;
          const uint32_t bytes = (cm.n * ES) & ~15u;
          TcEntry<KC>& ce = S.ce[e];
          ce.off = cm.off;
          ce.q = (uint32_t)(q0 + c);
          ce.n = cm.n;
          ce.m = cm.m;
          ce.s0 = fill % NS;
          ce.nsel = nsel;
          uint32_t fast = 1u, j = 0;
          for (uint32_t mm = cm.m; mm; mm &= mm - 1, ++j) {
            const uint32_t i = __ffs(mm) - 1;
            ce.ex[j] = (uint8_t)i;
            if constexpr (OPC == OP_TIES) {
              const uint32_t t = S.thr[c][i];
              ce.thr[j] = __uint_as_float(t);
              fast &= t >= 0x0D800000u ? 1u : 0u;  // bits of 2^-100
            }
          }
          ce.fast = OPC == OP_TIES ? fast : 0u;  // DARE-TIES: rescaled deltas may be tiny
          S.nf[e] = 1u + nsel;
          // test hook: the first chunk is never armed, so the consumers' wait for it runs out
          const bool arm = !(seq == 0 && p.stall);
          if (arm) mbar_arrive_expect_tx(&S.full[e], (1u + nsel) * bytes);
          if (bytes && arm)
            tma_load_1d(S.slot[fill % NS], static_cast<const char*>(p.base) + cm.off * ES, bytes, &S.full[e]);
          ++fill;
          for (uint32_t mm = cm.m; mm; mm &= mm - 1) {
            const uint32_t i = __ffs(mm) - 1;
            if (bytes && arm)
              tma_load_1d(S.slot[fill % NS],
                          static_cast<const char*>(p.experts.p[i]) + (cm.off - p.expert_origin) * ES, bytes,
                          &S.full[e]);
            ++fill;
            S.realized[i] += (unsigned long long)cm.n * ES;
          }
          used += 1u + nsel;
          ++seq;
        }
      }
      ok = __shfl_sync(0xFFFFFFFFu, ok, 0);
      __syncwarp();
    }
    if (lane == 0) {
      if (ok && (ok = reserve(0u))) {
        const uint32_t e = seq % NS;
        S.ce[e].q = kEnd;
        S.nf[e] = 0u;
        if (!(seq == 0 && p.stall)) mbar_arrive_expect_tx(&S.full[e], 0u);
        ++seq;
      }
      if (!ok) {
        atomicOr(p.err, kErrTimeout);
        S.abort = 1;
      }
      // drain: the last chunk of every entry must have landed before the CTA may exit
      for (uint32_t e = 0; e < (uint32_t)NS && e < seq; ++e) {
        const uint32_t last = seq - 1 - ((seq - 1 + NS - e) % NS);
        if (last == 0 && p.stall) continue;  // never armed: nothing in flight
        mbar_wait_drain(&S.full[e], (last / NS) & 1u);
      }
      for (uint32_t i = 0; i < p.K; ++i)
        if (S.realized[i])
          atomicAdd(p.realized + (uint64_t)(blockIdx.x % kCounterSlots) * p.K + i, S.realized[i]);
    }
    return;
  }
  // ---------------- consumers: thread t owns vector t of every chunk ----------------
  const uint32_t k0 = tid * (uint32_t)V;
  for (uint32_t c = 0;; ++c) {
    const uint32_t e = c % NS;
    if (!warp_wait<true>(&S.full[e], (c / NS) & 1u, abort_flag, wl)) {
      atomicOr(p.err, kErrTimeout);
      S.abort = 1;
      break;
    }
    const TcEntry<KC>& ce = S.ce[e];
    if (ce.q == kEnd) break;
    uint32_t s = ce.s0;
    const uint32_t nsel = ce.nsel;
    float x0[V];
    bool in_slot;  // the thread's vector lies inside the bulk-copied bytes
    {
      const uint32_t n = ce.n, n_tma = ((n * ES) & ~15u) / ES;
      in_slot = k0 + V <= n_tma;
      read_vec<BF16>(S.slot[s], p.base, ce.off, k0, n, n_tma, x0);
    }
    float y[V];
    if (nsel == 0) {  // uniform over the CTA
      // no expert selected: the output is M_0 plus the zero the operator adds (lambda * +0
      // for TIES, +0 for DARE)
      const float z = kTiesLike<OPC> ? __fmul_rn(p.lambda, 0.0f) : 0.0f;
#pragma unroll
      for (int v = 0; v < V; ++v) y[v] = __fadd_rn(x0[v], z);
      const uint64_t off = ce.off;
      const uint32_t n = ce.n;
      mbar_arrive(&S.empty[e]);
      if (k0 < n) store_vec<BF16>(p.out, off + k0, n - k0, y);
      continue;
    }
    if constexpr (OPC == OP_DARE) {
      // acc = fma(alpha_i, v_i, acc) over the selected experts whose keep word passes, in
      // ascending order, with v_i = delta_i * sigma (a dropped entry is omitted)
      float acc[V];
#pragma unroll
      for (int v = 0; v < V; ++v) acc[v] = 0.0f;
#pragma unroll 1
      for (uint32_t j = 0; j < nsel; ++j) {
        s = s + 1 == (uint32_t)NS ? 0u : s + 1;
        const uint32_t i = ce.ex[j];
        const float a = p.alpha[i];
        uint4 r;
        if (in_slot) {
          r = *reinterpret_cast<const uint4*>(S.slot[s] + k0 * ES);
        } else {  // the ragged tail of a tensor, from global memory
          const uint32_t n = ce.n;
          r = read_raw<BF16>(S.slot[s], p.experts.p[i], ce.off - p.expert_origin, k0, n, ((n * ES) & ~15u) / ES);
        }
        uint32_t kw[V];
        dare_keep_words<BF16>(p, i, ce.off + k0, kw);
        auto fold_pair = [&](int v, float e0, float e1) {
          float d0, d1, s0, s1;
          f2_sub(e0, e1, x0[v], x0[v + 1], d0, d1);
          f2_mul(d0, d1, p.sigma, p.sigma, s0, s1);
          // a dropped entry is omitted from the sum, as an unselected one is
          if (kw[v] >= p.dare_T16) acc[v] = __fmaf_rn(a, s0, acc[v]);
          if (kw[v + 1] >= p.dare_T16) acc[v + 1] = __fmaf_rn(a, s1, acc[v + 1]);
        };
        float e0, e1;
        pair_of<BF16, 0>(r, e0, e1);
        fold_pair(0, e0, e1);
        pair_of<BF16, 1>(r, e0, e1);
        fold_pair(2, e0, e1);
        if constexpr (BF16) {
          pair_of<BF16, 2>(r, e0, e1);
          fold_pair(4, e0, e1);
          pair_of<BF16, 3>(r, e0, e1);
          fold_pair(6, e0, e1);
        }
      }
      const uint64_t off = ce.off;
      const uint32_t n = ce.n;
      mbar_arrive(&S.empty[e]);  // every read of the chunk's slots and entry is done
#pragma unroll
      for (int v = 0; v < V; v += 2) f2_add(x0[v], x0[v + 1], acc[v], acc[v + 1], y[v], y[v + 1]);
      if (k0 < n) store_vec<BF16>(p.out, off + k0, n - k0, y);
      continue;
    }
    // Per element: P and N, the sums of the kept positive and negative deltas, and both
    // counts in one float C = 2^23 + c+ + 2^CB c- (exact: every value is an integer below
    // 2^24, so the low bits of C hold c+ and c-).  DARE-TIES keeps, instead, every nonzero
    // rescaled delta s = d sigma whose keep word passes (no magnitude trim).  A delta d is kept positive when d >= thr and kept
    // negative when d <= -thr (thr > 0: |d| >= thr and the sign in one compare each); the
    // keep factors k+ and k- are 1 or 0, and P = fma(k+, d, P), N = fma(k-, d, N): a factor 1
    // adds d with the one rounding of P + d, a factor 0 adds a zero, which leaves P and N
    // unchanged (they start at +0 and are never -0).  Two elements per packed instruction.
    float Pp[V], Nn[V], Cc[V];
#pragma unroll
    for (int v = 0; v < V; ++v) {
      Pp[v] = 0.0f;
      Nn[v] = 0.0f;
      Cc[v] = 8388608.0f;  // 2^23
    }
    // the selected experts in ascending order: fill j of the chunk sits in slot s0 + 1 + j
#pragma unroll 1
    for (uint32_t j = 0; j < nsel; ++j) {
      s = s + 1 == (uint32_t)NS ? 0u : s + 1;
      const float thr = OPC == OP_TIES ? ce.thr[j] : 0.0f;
      uint32_t kw[V];
      if constexpr (OPC == OP_DTIES) dare_keep_words<BF16>(p, ce.ex[j], ce.off + k0, kw);
      uint4 r;
      if (in_slot) {
        r = *reinterpret_cast<const uint4*>(S.slot[s] + k0 * ES);
      } else {  // the ragged tail of a tensor, from global memory (expert = j-th selected)
        const uint32_t i = __fns(ce.m, 0, (int)j + 1), n = ce.n;
        r = read_raw<BF16>(S.slot[s], p.experts.p[i], ce.off - p.expert_origin, k0, n, ((n * ES) & ~15u) / ES);
      }
      // one element pair at a time, so that only the raw vector stays live
      auto tally_pair = [&](int v, float e0, float e1) {
        float d0, d1, t0, t1, kp0, kp1, kn0, kn1;
        f2_sub(e0, e1, x0[v], x0[v + 1], d0, d1);
        if constexpr (OPC == OP_DTIES) {
          f2_mul(d0, d1, p.sigma, p.sigma, d0, d1);
          // keep factors as 1.0 / 0.0 straight from compares joined with the keep test
          asm("{\n .reg .pred q;\n setp.ge.u32 q, %4, %5;\n set.gt.and.f32.f32 %0, %6, 0f00000000, q;\n"
              " set.lt.and.f32.f32 %1, %6, 0f00000000, q;\n setp.ge.u32 q, %7, %5;\n"
              " set.gt.and.f32.f32 %2, %8, 0f00000000, q;\n set.lt.and.f32.f32 %3, %8, 0f00000000, q;\n}"
              : "=f"(kp0), "=f"(kn0), "=f"(kp1), "=f"(kn1)
              : "r"(kw[v]), "r"(p.dare_T16), "f"(d0), "r"(kw[v + 1]), "f"(d1));
        } else {
          kp0 = d0 >= thr ? 1.0f : 0.0f;
          kp1 = d1 >= thr ? 1.0f : 0.0f;
          kn0 = d0 <= -thr ? 1.0f : 0.0f;
          kn1 = d1 <= -thr ? 1.0f : 0.0f;
        }
        f2_fma(kp0, kp1, d0, d1, Pp[v], Pp[v + 1], Pp[v], Pp[v + 1]);
        f2_fma(kn0, kn1, d0, d1, Nn[v], Nn[v + 1], Nn[v], Nn[v + 1]);
        f2_fma(kn0, kn1, (float)(1u << CB), (float)(1u << CB), kp0, kp1, t0, t1);
        f2_add(Cc[v], Cc[v + 1], t0, t1, Cc[v], Cc[v + 1]);
      };
      float e0, e1;
      pair_of<BF16, 0>(r, e0, e1);
      tally_pair(0, e0, e1);
      pair_of<BF16, 1>(r, e0, e1);
      tally_pair(2, e0, e1);
      if constexpr (BF16) {
        pair_of<BF16, 2>(r, e0, e1);
        tally_pair(4, e0, e1);
        pair_of<BF16, 3>(r, e0, e1);
        tally_pair(6, e0, e1);
      }
    }
    const uint64_t off = ce.off;
    const uint32_t n = ce.n, fast = ce.fast;
    mbar_arrive(&S.empty[e]);  // every read of the chunk's slots and entry is done
    // the elected side's sum and count: the sign of P + N taken exactly as P > -N or P < -N
    // (then that side holds at least one entry, so c >= 1); otherwise the numerator +0, whose
    // quotient is +0 whatever count (<= 16, a valid table entry) is paired with it
    auto num_c = [&](int v, float& num, uint32_t& cv) {
      const bool pos = Pp[v] > -Nn[v], any = Pp[v] != -Nn[v];
      num = any ? (pos ? Pp[v] : Nn[v]) : 0.0f;
      const uint32_t cb = __float_as_uint(Cc[v]);
      cv = (pos ? cb : cb >> CB) & ((1u << CB) - 1u);
    };
    // q = RN(num * y), then Markstein's correction q + RN(num - q c) * y, and the output
    // fma(lambda, q, M_0), two elements per instruction; `checked` also notes the numerators
    // 0 < |num| < 2^-100, which then take the IEEE division under one warp vote
    auto finalise = [&](auto checked) {
      // 2 |bits| - 2 wraps the zeros to the top: its minimum over the vector is below
      // 2 * bits(2^-100) - 2 exactly when some numerator has 0 < |num| < 2^-100
      uint32_t lowest = 0xFFFFFFFFu;
#pragma unroll
      for (int v = 0; v < V; v += 2) {
        float a0, a1, q0, q1, r0, r1;
        uint32_t c0, c1;
        num_c(v, a0, c0);
        num_c(v + 1, a1, c1);
        if constexpr (decltype(checked)::value)
          lowest = min(lowest, min(__float_as_uint(a0) * 2u - 2u, __float_as_uint(a1) * 2u - 2u));
        const float2 t0 = S.ntab[c0], t1 = S.ntab[c1];
        f2_mul(a0, a1, t0.y, t1.y, q0, q1);
        f2_fma(q0, q1, t0.x, t1.x, a0, a1, r0, r1);
        f2_fma(r0, r1, t0.y, t1.y, q0, q1, q0, q1);
        f2_fma(p.lambda, p.lambda, q0, q1, x0[v], x0[v + 1], y[v], y[v + 1]);
      }
      static_assert(0x0D800000u * 2u - 2u == 0x1AFFFFFEu, "bits of 2^-100");
      const bool exact = decltype(checked)::value && lowest < 0x1AFFFFFEu;
      if (decltype(checked)::value && __any_sync(0xFFFFFFFFu, exact)) {
#pragma unroll
        for (int v = 0; v < V; ++v) {
          float a;
          uint32_t cv;
          num_c(v, a, cv);
          if (div_small_needs_ieee(a)) y[v] = __fmaf_rn(p.lambda, __fdiv_rn(a, -S.ntab[cv].x), x0[v]);
        }
      }
    };
    if constexpr (OPC == OP_DTIES) {
      finalise(std::true_type{});  // rescaled deltas may be tiny: always checked
    } else if (fast) {             // uniform over the CTA: every nonzero numerator >= 2^-100
      finalise(std::false_type{});
    } else {
      // TIES chunks with a threshold below 2^-100 (rare): one element at a time
      bool exact = false;
#pragma unroll
      for (int v = 0; v < V; ++v) {
        float a;
        uint32_t cv;
        num_c(v, a, cv);
        const float2 t = S.ntab[cv];
        y[v] = div_small_fast(a, -t.x, t.y);
        exact = exact || div_small_needs_ieee(a);
      }
      if (__any_sync(0xFFFFFFFFu, exact)) {
#pragma unroll
        for (int v = 0; v < V; ++v) {
          float a;
          uint32_t cv;
          num_c(v, a, cv);
          if (div_small_needs_ieee(a)) y[v] = __fdiv_rn(a, -S.ntab[cv].x);
        }
      }
#pragma unroll
      for (int v = 0; v < V; ++v) y[v] = __fmaf_rn(p.lambda, y[v], x0[v]);
    }
    if (k0 < n) store_vec<BF16>(p.out, off + k0, n - k0, y);
  }
}

template <bool BF16, int OPC, int KC>
cudaError_t launch_chunk(const MergeLaunch& p, cudaStream_t st) {
  constexpr uint32_t chunk = kTcSlotBytes / (BF16 ? 2u : 4u);
  const uint32_t cpb = (p.block_elems + chunk - 1) / chunk;
  const uint64_t n_chunks = (p.b_end - p.b_begin) * cpb;
  if (n_chunks == 0) return cudaSuccess;
  if (n_chunks >= 0xFFFFFFFFull) return cudaErrorInvalidValue;
  int dev = 0, sms = 0;
  cudaError_t e;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
  using Smem = TcSmem<TcGeo<OPC, KC>::kSlots, TcGeo<OPC, KC>::kGrab, KC>;
  // every CTA also holds 1 KB of the SM's 228 KB for the system
  static_assert(TcGeo<OPC, KC>::kCtasPerSm * (sizeof(Smem) + 1024) <= 228u * 1024u,
                "the CTAs per SM that the grid assumes fit one SM's shared memory");
  const size_t smem = sizeof(Smem);
  auto kern = merge_chunk_kernel<BF16, OPC, KC>;
  if ((e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)) != cudaSuccess)
    return e;
  uint64_t grid = (uint64_t)sms * TcGeo<OPC, KC>::kCtasPerSm;
  if (grid > n_chunks) grid = n_chunks;
  if ((e = launch_fill(p.work, 0, sizeof(unsigned long long), st)) != cudaSuccess) return e;
  kern<<<(unsigned)grid, TcGeo<OPC, KC>::kThreads, smem, st>>>(p, cpb, n_chunks, p.work);
  count_launches(1);
  return cudaGetLastError();
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
  const size_t smem = sizeof(Smem<Geo<OPC>::kSlots, Geo<OPC>::kSlotBytes, Geo<OPC>::kGrab>);
  if ((e = cudaFuncSetAttribute(merge_tma_kernel<BF16, OPC>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)) !=
      cudaSuccess)
    return e;
  uint64_t grid = (uint64_t)sms * Geo<OPC>::kCtasPerSm;
  if (grid > n_chunks) grid = n_chunks;
  if ((e = launch_fill(p.work, 0, sizeof(unsigned long long), st)) != cudaSuccess) return e;
  merge_tma_kernel<BF16, OPC><<<(unsigned)grid, Geo<OPC>::kThreads, smem, st>>>(p, cpb, n_chunks, p.work);
  count_launches(1);
  return cudaGetLastError();
}

template <bool BF16>
cudaError_t launch_dtype(const MergeLaunch& p, cudaStream_t st) {
  switch (p.op_kind) {
    case MP_OP_AVG:
    case MP_OP_TA: return launch_op<BF16, OP_ADD>(p, st);
    case MP_OP_TIES:
      if (p.K <= 4) return launch_chunk<BF16, OP_TIES, 4>(p, st);
      if (p.K <= 8) return launch_chunk<BF16, OP_TIES, 8>(p, st);
      return launch_op<BF16, OP_TIES>(p, st);
    case MP_OP_DARE:
      if (p.K <= 4) return launch_chunk<BF16, OP_DARE, 4>(p, st);
      if (p.K <= 8) return launch_chunk<BF16, OP_DARE, 8>(p, st);
      if (p.K <= 16) return launch_chunk<BF16, OP_DARE, 16>(p, st);
      return launch_op<BF16, OP_DARE>(p, st);
    case MP_OP_AVG_RENORM: return launch_op<BF16, OP_RENORM>(p, st);
    case MP_OP_DARE_TIES:
      if (p.K <= 4) return launch_chunk<BF16, OP_DTIES, 4>(p, st);
      if (p.K <= 8) return launch_chunk<BF16, OP_DTIES, 8>(p, st);
      if (p.K <= 16) return launch_chunk<BF16, OP_DTIES, 16>(p, st);
      return launch_op<BF16, OP_DTIES>(p, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

cudaError_t launch_merge(const MergeLaunch& p, cudaStream_t st) {
  return p.dtype == MP_BF16 ? launch_dtype<true>(p, st) : launch_dtype<false>(p, st);
}

}  // namespace mp
