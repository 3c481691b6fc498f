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
#include "tma.cuh"

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
    // the lower element moved up by a multiply (FMA pipe), the upper one by a mask (ALU)
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

__device__ __forceinline__ uint32_t ties_key(float d) {
  return (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(fabsf(d))) & 0x7FFFu;
}

// ---- the catalog pass: TMA producer / consumer pipeline ---------------------------------
//
// Work item = (block, group of up to KG experts); items are handed out through a global
// counter.  The producer thread streams every chunk of the item's block — the base chunk,
// then each expert's chunk — into a ring of shared-memory slots (cp.async.bulk, completion
// on the slot's "full" mbarrier).  Consumer thread l (0..255) is lane l of the fixed
// summation order: a chunk of VPT * 256 vectors starts at vector VPT * 256 * c, and thread
// l takes its vectors VPT * 256 * c + 256 u + l (u < VPT), i.e. exactly its own vectors l,
// l + 256, ... in increasing order.  At the end of the block the 256 lane sums are
// combined by the xor butterfly.
constexpr int kIxConsumers = 256;
constexpr int kIxThreads = kIxConsumers + 32;
static_assert(kIxConsumers == 256, "one consumer thread per coarse TIES bin at the end of a block");
constexpr uint32_t kIxEnd = 0xFFFFFFFFu;

// ring geometry.  The plain catalog is bound by HBM: two CTAs per SM with twelve 8 KiB
// slots.  The TIES catalog also bins every delta, which makes it bound by instruction
// latency: four CTAs per SM (more warps to hide it; the state fits 56 registers) with twelve
// 4 KiB slots (one vector per consumer thread and fill).  With eight experts per item the
// histograms make a CTA too large for four per SM: three run, with the registers of three.
template <bool TIES, int KG = 1>
struct IxGeo {
  static constexpr int kCtasPerSm = TIES ? (KG > 4 ? 3 : 4) : 2;
  static constexpr uint32_t kSlotBytes = TIES ? 4096u : 8192u;
  static constexpr int kSlots = 12;
};

struct IxMeta {
  uint64_t off;    // element offset of the chunk
  uint32_t item;   // work item, or kIxEnd
  uint32_t n;      // elements in the chunk
  uint32_t last;   // 1 on the block's last chunk
  uint32_t s0;     // whole-chunk publication: ring slot of the base fill (experts follow)
  int32_t wlo[4];  // whole-chunk publication, window bins: L - 1 of the item's experts' windows
};

// How the TIES catalog bins the keys of the deltas:
//  * kBinCoarse: 256 bins of the upper 8 key bits (the two-level select: a second pass then
//    counts the lower 7 bits inside the chosen bin);
//  * kBinWindow: the 384 keys [L, L + 384) of a window predicted from a sample (three
//    coarse bins at full resolution), one bin below and one above it, so that the
//    threshold is found without a second pass whenever it lies inside the window.
enum { kBinNone = 0, kBinCoarse = 1, kBinWindow = 2 };
constexpr uint32_t kWinKeys = 384;           // keys of the window
constexpr uint32_t kWinBins = kWinKeys + 2;  // + below + above

template <int KG, int NS, uint32_t SB, uint32_t NB>
struct __align__(128) IxSmem {
  uint32_t hist[KG][NB];  // first: its byte addresses stay below 2^16 (ties_win2k packs two)
  alignas(128) uint8_t slot[NS][SB];
  IxMeta meta[NS];
  uint64_t full[NS];
  uint64_t empty[NS];
  uint32_t nf[NS];  // whole-chunk publication: fills held by the chunk of each entry
  float red_ss[KG][8];
  float red_mx[KG][8];
  uint32_t red_nz[KG][8];
  uint64_t cbar;  // consumer-only barrier (one arrival per consumer warp)
  int abort;
};

// raw 16-byte vector at element k0 of a fill: from the slot when inside the bulk-copied
// bytes, else (the ragged tail of a tensor) from global memory, zero past the chunk
template <bool BF16>
__device__ __forceinline__ uint4 ix_read_raw(const uint8_t* slot, const void* gsrc, uint64_t off, uint32_t k0,
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

__device__ __forceinline__ bool same_vec(const uint4 a, const uint4 b) {
  return a.x == b.x && a.y == b.y && a.z == b.z && a.w == b.w;
}

// TIES coarse bins of two deltas: bin = upper 8 bits of the 15-bit key bits(bf16(|d|)),
// i.e. bits 7..14 of the round-to-nearest-even bf16 of d (the sign bit 15 is masked off);
// both are converted by one packed cvt.  A nonzero delta adds 1 to its bin of the
// shared histogram at hist (byte address in the shared window); a zero delta adds
// nothing, so the histogram's total is the block's nonzero count.  Predicated, so that no
// branch is taken per element.
__device__ __forceinline__ void ties_bin2(float d0, float d1, uint32_t hist) {
  asm volatile(
      "{\n"
      " .reg .pred p0, p1;\n"
      " .reg .b32 w, a0, a1;\n"
      " cvt.rn.bf16x2.f32 w, %2, %1;\n"
      " setp.ne.f32 p0, %1, 0f00000000;\n"
      " setp.ne.f32 p1, %2, 0f00000000;\n"
      " shr.b32 a0, w, 5;\n"
      " and.b32 a0, a0, 1020;\n"
      " add.u32 a0, a0, %0;\n"
      " shr.b32 a1, w, 21;\n"
      " and.b32 a1, a1, 1020;\n"
      " add.u32 a1, a1, %0;\n"
      " @p0 red.shared.add.u32 [a0], 1;\n"
      " @p1 red.shared.add.u32 [a1], 1;\n"
      "}\n" ::"r"(hist),
      "f"(d0), "f"(d1)
      : "memory");
}

// (d0, d1) = (a0 - b0, a1 - b1), each rounded to nearest: one packed subtract
__device__ __forceinline__ void f2_sub(float a0, float a1, float b0, float b1, float& d0, float& d1) {
  asm("{\n .reg .b64 ra, rb, rd;\n mov.b64 ra, {%2, %3};\n mov.b64 rb, {%4, %5};\n sub.rn.f32x2 rd, ra, rb;\n"
      " mov.b64 {%0, %1}, rd;\n}"
      : "=f"(d0), "=f"(d1)
      : "f"(a0), "f"(a1), "f"(b0), "f"(b1));
}

// TIES window bins of two deltas: a nonzero delta with key k adds 1 to bin
// clamp(k - lo, 0, 385) of the shared histogram at hist0, with lo = L - 1: bin 0 below the
// window, bins 1..384 for the keys L..L + 383, bin 385 above it.  Both keys at once in
// 16-bit lanes: one add and one clamp at zero and 385 (k - lo lies in [-32383, 32768]; it
// wraps only for the NaN key 0x7FFF at lo = -1, whose bin the clamp still keeps in range and
// whose NaN the statistics report).  Predicated, no branch.
__device__ __forceinline__ void ties_win2(float d0, float d1, int32_t lo, uint32_t hist0) {
  const __nv_bfloat162 h2 = __floats2bfloat162_rn(d0, d1);
  const uint32_t w = *reinterpret_cast<const uint32_t*>(&h2) & 0x7FFF7FFFu;
  static_assert(kWinKeys + 1u == 0x181u, "the clamp bound is the above-window bin");
  const uint32_t nlo2 = ((uint32_t)(-lo) & 0xFFFFu) * 0x00010001u;
  uint32_t kk;
  asm("{\n .reg .b32 t;\n add.s16x2 t, %1, %2;\n min.s16x2.relu %0, t, %3;\n}"
      : "=r"(kk)
      : "r"(w), "r"(nlo2), "r"(0x01810181u));
  // byte addresses by multiply-add (FMA pipe; the ALU pipe carries the rest)
  uint32_t a0, a1;
  asm("mad.lo.u32 %0, %1, 4, %2;" : "=r"(a0) : "r"(kk & 0xFFFFu), "r"(hist0));
  asm("mad.lo.u32 %0, %1, 4, %2;" : "=r"(a1) : "r"(kk >> 16), "r"(hist0));
  asm volatile(
      "{\n"
      " .reg .pred p0, p1;\n"
      " setp.ne.f32 p0, %2, 0f00000000;\n"
      " setp.ne.f32 p1, %3, 0f00000000;\n"
      " @p0 red.shared.add.u32 [%0], 1;\n"
      " @p1 red.shared.add.u32 [%1], 1;\n"
      "}\n" ::"r"(a0),
      "r"(a1), "f"(d0), "f"(d1)
      : "memory");
}

// The same bins for deltas of two bf16 checkpoints, where key 0 holds exactly the zero
// deltas (the difference of two distinct bf16 values is at least the smallest bf16
// subnormal, whose key is 1).  Every delta adds 1 to its bin, zeros included: a zero has
// key 0 and lands below the window, in bin 0, which no threshold reads (with the window at
// the bottom, L = 0 and lo = -1, it lands in key 0's bin, where it can only decide a
// threshold of key 0, the one that an uncounted zero gives too).  The nonzero deltas are
// counted from the returned key word instead (nz_halves).  Both byte addresses come from one
// multiply-add in 16-bit lanes: h2 = the histogram's byte address in both lanes, which the
// caller keeps below 2^16 - 4 * 385.  No predicate and no branch.
__device__ __forceinline__ uint32_t ties_win2k(float d0, float d1, int32_t lo, uint32_t h2) {
  const __nv_bfloat162 hb = __floats2bfloat162_rn(d0, d1);
  const uint32_t w = *reinterpret_cast<const uint32_t*>(&hb) & 0x7FFF7FFFu;
  const uint32_t nlo2 = ((uint32_t)(-lo) & 0xFFFFu) * 0x00010001u;
  uint32_t kk;
  asm("{\n .reg .b32 t;\n add.s16x2 t, %1, %2;\n min.s16x2.relu %0, t, %3;\n}"
      : "=r"(kk)
      : "r"(w), "r"(nlo2), "r"(0x01810181u));
  const uint32_t a2 = kk * 4u + h2;  // lanes: h + 4 b0 and h + 4 b1 (no carry between them)
  asm volatile(
      "{\n"
      " .reg .b32 a0, a1;\n"
      " and.b32 a0, %0, 65535;\n"
      " shr.u32 a1, %0, 16;\n"
      " red.shared.add.u32 [a0], 1;\n"
      " red.shared.add.u32 [a1], 1;\n"
      "}\n" ::"r"(a2)
      : "memory");
  return w;
}

// number of nonzero keys among the four key words of a vector, in two 16-bit lanes
__device__ __forceinline__ uint32_t nz_halves(uint32_t w0, uint32_t w1, uint32_t w2, uint32_t w3) {
  uint32_t m0, m1, m2, m3;
  asm("min.u16x2 %0, %1, %2;" : "=r"(m0) : "r"(w0), "r"(0x00010001u));
  asm("min.u16x2 %0, %1, %2;" : "=r"(m1) : "r"(w1), "r"(0x00010001u));
  asm("min.u16x2 %0, %1, %2;" : "=r"(m2) : "r"(w2), "r"(0x00010001u));
  asm("min.u16x2 %0, %1, %2;" : "=r"(m3) : "r"(w3), "r"(0x00010001u));
  return m0 + m1 + m2 + m3;
}

// TIES fine bins of two deltas: a nonzero delta whose coarse bin (key bits 7..14) is es
// adds 1 to fine bin (key & 127) of the shared histogram at hist; predicated, no branch
__device__ __forceinline__ void ties_fine2(float d0, float d1, uint32_t es, uint32_t hist) {
  asm volatile(
      "{\n"
      " .reg .pred p0, p1;\n"
      " .reg .b32 w, k0, k1, e0, e1, a0, a1;\n"
      " cvt.rn.bf16x2.f32 w, %2, %1;\n"
      " and.b32 k0, w, 32767;\n"
      " shr.b32 k1, w, 16;\n"
      " and.b32 k1, k1, 32767;\n"
      " shr.b32 e0, k0, 7;\n"
      " shr.b32 e1, k1, 7;\n"
      " setp.ne.f32 p0, %1, 0f00000000;\n"
      " setp.ne.f32 p1, %2, 0f00000000;\n"
      " setp.eq.and.u32 p0, e0, %3, p0;\n"
      " setp.eq.and.u32 p1, e1, %3, p1;\n"
      " and.b32 a0, k0, 127;\n"
      " and.b32 a1, k1, 127;\n"
      " shl.b32 a0, a0, 2;\n"
      " shl.b32 a1, a1, 2;\n"
      " add.u32 a0, a0, %0;\n"
      " add.u32 a1, a1, %0;\n"
      " @p0 red.shared.add.u32 [a0], 1;\n"
      " @p1 red.shared.add.u32 [a1], 1;\n"
      "}\n" ::"r"(hist),
      "f"(d0), "f"(d1), "r"(es)
      : "memory");
}

// Checked build: a work item (block b, experts i0 .. i0 + kc - 1) must lie in the launch's
// block range before the block table is read for it, and the whole block, read from the
// base and those experts, must pass chunk_in_bounds (with its TIES trim group below
// n_groups) before anything is copied or loaded; a failure is recorded in the call's error
// word and the item is skipped.  Constant true in the default build.
template <bool TIES>
__device__ __forceinline__ bool checked_item(const IndexLaunch& p, uint64_t b, uint32_t i0, uint32_t kc,
                                             uint32_t es) {
  if constexpr (!kChecked) return true;
  if (b >= p.b_begin && b < p.b_end && b < p.n_blocks && i0 < p.K && (!TIES || p.blk_group[b] < p.n_groups) &&
      chunk_in_bounds(b, p.b_begin, p.b_end, p.blk_off[b], p.blk_len[b], p.blk_off[b], p.blk_len[b],
                      expert_run(i0, kc), p.K, es, p.expert_origin, p.ext))
    return true;
  atomicOr(p.err, kErrBounds);
  return false;
}

template <bool BF16, int KG, int BM>
__global__ void __launch_bounds__(kIxThreads, IxGeo<BM != kBinNone, KG>::kCtasPerSm)
    index_tma_kernel(const IndexLaunch p, uint32_t G, uint64_t n_items, unsigned long long* work) {
  constexpr bool TIES = BM != kBinNone;
  constexpr uint32_t NB = BM == kBinNone ? 1u : (BM == kBinWindow ? kWinBins : 256u);  // key bins per expert
  // The TIES catalog with up to 4 experts per item publishes whole chunks: the base fill and
  // the item's expert fills of one chunk sit in consecutive ring slots under one "full"
  // mbarrier (counting all their bytes) and one "empty" mbarrier, so that a consumer waits
  // and releases once per chunk instead of once per fill.
  constexpr bool CW = TIES && KG <= 4;
  // window bins of bf16 deltas: the nonzero count comes from the keys (ties_win2k,
  // nz_halves) and the zeros share the below-window bin
  constexpr bool KNZ = BM == kBinWindow && BF16;
  constexpr int kIxSlots = IxGeo<TIES, KG>::kSlots;
  static_assert(!CW || kIxSlots >= 2 * (KG + 1), "two whole chunks fit the ring");
  constexpr uint32_t kIxSlotBytes = IxGeo<TIES, KG>::kSlotBytes;
  constexpr uint32_t ES = BF16 ? 2u : 4u;
  constexpr uint32_t CH = kIxSlotBytes / ES;
  constexpr int V = BF16 ? 8 : 4;
  constexpr int VPT = (int)(CH / (kIxConsumers * V));
  static_assert(VPT >= 1 && CH == (uint32_t)(VPT * kIxConsumers * V), "chunk geometry");
  extern __shared__ __align__(128) uint8_t smem_raw[];
  using Sm = IxSmem<KG, kIxSlots, kIxSlotBytes, NB>;
  Sm& S = *reinterpret_cast<Sm*>(smem_raw);
  const uint32_t tid = threadIdx.x, warp = tid >> 5, lane = tid & 31u;
  // the fallback pass of the windowed catalog runs only when some threshold left its window
  if (BM == kBinCoarse && p.miss && *p.miss == 0u) return;
  if constexpr (KNZ) {  // the packed bin addresses need the histogram below 2^16 - 4 * 385
    if (su32(&S.hist[KG - 1][NB - 1]) >= 65536u - 4u * (kWinKeys + 1u)) {
      if (threadIdx.x == 0) atomicOr(p.err, kErrInternal);
      return;
    }
  }
  volatile int* abort_flag = &S.abort;
  const uint32_t wl = wait_limit_of(p.wait_limit);

  if (tid == 0) {
    for (int s = 0; s < kIxSlots; ++s) {
      mbar_init(&S.full[s], 1);
      mbar_init(&S.empty[s], kIxConsumers);  // every consumer thread arrives
    }
    mbar_init(&S.cbar, kIxConsumers / 32);
    S.abort = 0;
    mbar_fence_init();
  }
  for (uint32_t x = tid; x < (uint32_t)KG * NB; x += blockDim.x) (&S.hist[0][0])[x] = 0u;
  __syncthreads();

  if (warp == kIxConsumers / 32) {
    // ---------------- producer ----------------
    if (lane == 0) {
      uint32_t fill = 0;
      bool ok = true;
      // whole-chunk publication: chunks published (seq), the oldest one not yet seen released
      // (head) and the ring slots held by chunks head .. seq - 1 (used)
      uint32_t seq = 0, head = 0, used = 0;
      auto reserve = [&](uint32_t nfill) -> bool {
        while (seq - head >= (uint32_t)kIxSlots || used + nfill > (uint32_t)kIxSlots) {
          const uint32_t he = head % kIxSlots;
          if (!mbar_wait(&S.empty[he], (head / kIxSlots) & 1u, abort_flag, wl)) return false;
          used -= S.nf[he];
          ++head;
        }
        return true;
      };
      // publishes one chunk: the base fill and kc expert fills in consecutive slots
      int32_t item_wlo[4] = {0, 0, 0, 0};  // window bins: L - 1 of the current item's experts
      auto publish = [&](uint32_t item, uint64_t off, uint32_t n, uint32_t last, uint32_t i0,
                         uint32_t kc) -> bool {
        const uint32_t nfill = item == kIxEnd ? 0u : 1u + kc;
        if (!reserve(nfill)) return false;
        if (fill >= (uint32_t)kIxSlots) fence_proxy_async_smem();  // slots the consumers have read are refilled
        const uint32_t e = seq % kIxSlots;
        const uint32_t bytes = (n * ES) & ~15u;
        S.meta[e].off = off;
        S.meta[e].item = item;
        S.meta[e].n = n;
        S.meta[e].last = last;
        S.meta[e].s0 = fill % kIxSlots;
        if constexpr (BM == kBinWindow) {
#pragma unroll
          for (int k = 0; k < 4; ++k) S.meta[e].wlo[k] = item_wlo[k];
        }
        S.nf[e] = nfill;
        const bool arm = !(seq == 0 && p.stall);  // test hook: the first chunk is never armed
        if (arm) mbar_arrive_expect_tx(&S.full[e], nfill * bytes);
        if (nfill) {
          if (bytes && arm)
            tma_load_1d(S.slot[fill % kIxSlots], static_cast<const char*>(p.base) + off * ES, bytes, &S.full[e]);
          ++fill;
          for (uint32_t k = 0; k < kc; ++k) {
            if (bytes && arm)
              tma_load_1d(S.slot[fill % kIxSlots],
                          static_cast<const char*>(p.experts.p[i0 + k]) + (off - p.expert_origin) * ES, bytes,
                          &S.full[e]);
            ++fill;
          }
        }
        used += nfill;
        ++seq;
        return true;
      };
      auto produce = [&](uint32_t item, uint64_t off, uint32_t n, uint32_t last, const char* src_row,
                         uint32_t bytes) -> bool {
        const uint32_t s = fill % kIxSlots, r = fill / kIxSlots;
        if (fill == 0 && p.stall) {  // test hook: slot 0 is never armed, so its wait runs out
          ++fill;
          return true;
        }
        if (r > 0 && !mbar_wait(&S.empty[s], (r - 1) & 1u, abort_flag, wl)) return false;
        if (r > 0) fence_proxy_async_smem();
        S.meta[s].off = off;
        S.meta[s].item = item;
        S.meta[s].n = n;
        S.meta[s].last = last;
        mbar_arrive_expect_tx(&S.full[s], bytes);
        if (bytes) tma_load_1d(S.slot[s], src_row, bytes, &S.full[s]);
        ++fill;
        return true;
      };
      while (ok) {
        const unsigned long long it = atomicAdd(work, 1ull);
        if (it >= n_items) break;
        const uint64_t b = p.b_begin + it / G;
        const uint32_t i0 = (uint32_t)(it % G) * KG;
        const uint32_t kc = min((uint32_t)KG, p.K - i0);
        if (!checked_item<TIES>(p, b, i0, kc, ES)) continue;
        if (BM == kBinCoarse && p.gmiss) {  // windowed fallback: the marked pairs' groups only
          const uint32_t grp = p.blk_group[b];
          bool any = false;
          for (uint32_t k = 0; k < kc; ++k) any = any || p.gmiss[(uint64_t)(i0 + k) * p.n_groups + grp] != 0u;
          if (!any) continue;
        }
        const uint32_t len = p.blk_len[b];
        const uint64_t off0 = p.blk_off[b];
        const uint32_t nch = (len + CH - 1) / CH;
        if constexpr (CW && BM == kBinWindow) {
          const uint32_t grp = p.blk_group[b];
#pragma unroll
          for (int k = 0; k < 4; ++k)
            item_wlo[k] = (uint32_t)k < kc ? (int32_t)p.wlo[(uint64_t)(i0 + k) * p.n_groups + grp] - 1 : 0;
        }
        for (uint32_t c = 0; c < nch && ok; ++c) {
          const uint32_t n = min(CH, len - c * CH);
          const uint64_t off = off0 + (uint64_t)c * CH;
          const uint32_t bytes = (n * ES) & ~15u;
          const uint32_t last = c + 1 == nch ? 1u : 0u;
          if constexpr (CW) {
            ok = publish((uint32_t)it, off, n, last, i0, kc);
          } else {
            ok = produce((uint32_t)it, off, n, last, static_cast<const char*>(p.base) + off * ES, bytes);
            for (uint32_t k = 0; k < kc && ok; ++k)
              ok = produce((uint32_t)it, off, n, last,
                           static_cast<const char*>(p.experts.p[i0 + k]) + (off - p.expert_origin) * ES, bytes);
          }
        }
      }
      if (ok) ok = CW ? publish(kIxEnd, 0, 0, 0, 0, 0) : produce(kIxEnd, 0, 0, 0, nullptr, 0);
      if (!ok) {
        atomicOr(p.err, kErrTimeout);
        S.abort = 1;
      }
      // drain: the last use of every slot (entry, when publishing whole chunks) must have
      // landed before the CTA may exit
      const uint32_t nuse = CW ? seq : fill;
      for (uint32_t s = 0; s < (uint32_t)kIxSlots && s < nuse; ++s) {
        const uint32_t lastf = nuse - 1 - ((nuse - 1 + kIxSlots - s) % kIxSlots);
        if (lastf == 0 && p.stall) continue;  // never armed: nothing in flight
        mbar_wait_drain(&S.full[s], (lastf / kIxSlots) & 1u);
      }
    }
    return;
  }

  // ---------------- consumers (lane l of the summation order) ----------------
  float ss[KG], mx[KG];
  uint32_t nz[KG];
#pragma unroll
  for (int k = 0; k < KG; ++k) {
    ss[k] = 0.0f;
    mx[k] = 0.0f;
    nz[k] = 0u;
  }
  uint32_t fill = 0, cphase = 0;
  bool alive = true;
  auto wait_full = [&](uint32_t f) -> bool {
    if (!warp_wait(&S.full[f % kIxSlots], (f / kIxSlots) & 1u, abort_flag, wl)) {
      atomicOr(p.err, kErrTimeout);
      S.abort = 1;
      return false;
    }
    return true;
  };
  auto release = [&](uint32_t f) {
    mbar_arrive(&S.empty[f % kIxSlots]);  // every consumer thread: its own reads of the slot are done
  };
  while (alive) {
    if (!wait_full(fill)) break;
    const IxMeta mt = S.meta[fill % kIxSlots];
    if (mt.item == kIxEnd) break;
    const uint64_t b = p.b_begin + mt.item / G;
    const uint32_t i0 = (mt.item % G) * KG;
    const uint32_t kc = min((uint32_t)KG, p.K - i0);
    const uint32_t n = mt.n, n_tma = ((n * ES) & ~15u) / ES;
    const uint64_t off = mt.off;
    float xb[VPT][V];
    uint4 rb[VPT];     // the base vectors as read, for the equality test
    bool bfin = true;  // every base element finite (Inf - Inf and NaN - NaN are not zero)
    const uint32_t s0 = mt.s0;  // whole-chunk publication: the base fill's slot
    {
      const uint8_t* slot = S.slot[CW ? s0 : fill % kIxSlots];
#pragma unroll
      for (int u = 0; u < VPT; ++u) {
        rb[u] = ix_read_raw<BF16>(slot, p.base, off, (tid + (uint32_t)u * kIxConsumers) * V, n, n_tma);
        unpack<BF16>(rb[u], xb[u]);
#pragma unroll
        for (int e = 0; e < V; ++e) bfin = bfin && fabsf(xb[u][e]) < __int_as_float(0x7F800000);
      }
      if constexpr (!CW) {
        release(fill);
        ++fill;
      }
    }
#pragma unroll
    for (int k = 0; k < KG; ++k) {
      if ((uint32_t)k >= kc) break;
      if constexpr (!CW) {
        if (!wait_full(fill)) {
          alive = false;
          break;
        }
      }
      const uint8_t* slot = S.slot[CW ? (s0 + 1u + (uint32_t)k) % kIxSlots : fill % kIxSlots];
      uint4 re[VPT];
      // the equality test pays off only for TIES, whose per-element binning it skips; for
      // the other operators the comparison and vote cost more than the arithmetic they save
      bool same = TIES && bfin;
#pragma unroll
      for (int u = 0; u < VPT; ++u) {
        re[u] = ix_read_raw<BF16>(slot, p.experts.p[i0 + k], off - p.expert_origin,
                                  (tid + (uint32_t)u * kIxConsumers) * V, n, n_tma);
        same = same && same_vec(re[u], rb[u]);
      }
      // a finite vector equal bit for bit to the base gives deltas of exactly +0, which
      // change neither the sum of squares (>= +0), the max (>= +0), the count nor the bins:
      // a warp whose vectors all match skips them (warp-uniform, so the summation order is
      // untouched)
      if (!__all_sync(0xFFFFFFFFu, same)) {
        // kBinWindow: L - 1 of this expert's window in the block's trim group
        int32_t wlo_k = 0;
        if constexpr (BM == kBinWindow) {
          if constexpr (CW) wlo_k = mt.wlo[k < 4 ? k : 0];
          else wlo_k = (int32_t)__ldg(p.wlo + (uint64_t)(i0 + k) * p.n_groups + __ldg(p.blk_group + b)) - 1;
        }
#pragma unroll
        for (int u = 0; u < VPT; ++u) {
          float xe[V];
          unpack<BF16>(re[u], xe);
          float d[V];
#pragma unroll
          for (int e = 0; e < V; e += 2) f2_sub(xe[e], xe[e + 1], xb[u][e], xb[u][e + 1], d[e], d[e + 1]);
          // the sum of squares is one fma chain in element order (the canonical order);
          // max |d| and the counts are exact in any order, so they take a tree
#pragma unroll
          for (int e = 0; e < V; ++e) ss[k] = __fmaf_rn(d[e], d[e], ss[k]);
          float m[V / 2];
#pragma unroll
          for (int e = 0; e < V / 2; ++e) m[e] = fmaxf(fabsf(d[2 * e]), fabsf(d[2 * e + 1]));
#pragma unroll
          for (int w = V / 4; w >= 1; w >>= 1)
#pragma unroll
            for (int e = 0; e < w; ++e) m[e] = fmaxf(m[e], m[e + w]);
          mx[k] = fmaxf(mx[k], m[0]);
          if constexpr (KNZ) {
            const uint32_t h2 = su32(&S.hist[k][0]) * 0x00010001u;
            uint32_t wk[V / 2];
#pragma unroll
            for (int e = 0; e < V; e += 2) wk[e / 2] = ties_win2k(d[e], d[e + 1], wlo_k, h2);
            nz[k] += nz_halves(wk[0], wk[1], wk[2], wk[3]);
          } else {
#pragma unroll
            for (int e = 0; e < V; e += 2) {
              if constexpr (BM == kBinWindow) {
                ties_win2(d[e], d[e + 1], wlo_k, su32(&S.hist[k][0]));
              } else if constexpr (BM == kBinCoarse) {
                ties_bin2(d[e], d[e + 1], su32(&S.hist[k][0]));
              } else {
                nz[k] += d[e] != 0.0f ? 1u : 0u;
                nz[k] += d[e + 1] != 0.0f ? 1u : 0u;
              }
            }
          }
        }
      }
      if constexpr (!CW) {
        release(fill);
        ++fill;
      }
    }
    if constexpr (CW) {  // every read of the chunk's slots and entry is done
      release(fill);
      ++fill;
    }
    if (!alive || !mt.last) continue;

    // end of the block: the canonical combine, then the statistics (and TIES bins)
#pragma unroll
    for (int k = 0; k < KG; ++k) {
      if constexpr (KNZ) nz[k] = (nz[k] & 0xFFFFu) + (nz[k] >> 16);  // the two 16-bit lanes
#pragma unroll
      for (int s = 16; s >= 1; s >>= 1) {
        ss[k] = __fadd_rn(ss[k], __shfl_xor_sync(0xFFFFFFFFu, ss[k], s));
        mx[k] = fmaxf(mx[k], __shfl_xor_sync(0xFFFFFFFFu, mx[k], s));
        nz[k] += __shfl_xor_sync(0xFFFFFFFFu, nz[k], s);
      }
      if (lane == 0) {
        S.red_ss[k][warp] = ss[k];
        S.red_mx[k][warp] = mx[k];
        S.red_nz[k][warp] = nz[k];
      }
      ss[k] = 0.0f;
      mx[k] = 0.0f;
      nz[k] = 0u;
    }
    if (!consumer_barrier(&S.cbar, cphase, abort_flag, wl)) {
      atomicOr(p.err, kErrTimeout);
      S.abort = 1;
      break;
    }
    if (warp == 0) {
      uint32_t bad = 0u;
#pragma unroll
      for (int k = 0; k < KG; ++k) {
        float a = lane < 8 ? S.red_ss[k][lane] : 0.0f;
        float m = lane < 8 ? S.red_mx[k][lane] : 0.0f;
        uint32_t c = lane < 8 ? S.red_nz[k][lane] : 0u;
#pragma unroll
        for (int s = 4; s >= 1; s >>= 1) {
          a = __fadd_rn(a, __shfl_xor_sync(0xFFFFFFFFu, a, s));
          m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, s));
          c += __shfl_xor_sync(0xFFFFFFFFu, c, s);
        }
        if (lane == 0 && (uint32_t)k < kc) {
          const uint64_t u = (uint64_t)(i0 + k) * p.n_blocks + b;
          p.norm[u] = __fsqrt_rn(a);
          p.maxabs[u] = m;
          if constexpr (!TIES || KNZ) p.nnz[u] = c;
          // a NaN delta makes the sum of squares NaN; an infinite one makes max |delta| infinite
          if (isnan(a) || isinf(m)) bad = 1u;
        }
      }
      if (lane == 0 && bad) atomicOr(p.err, kErrNonfinite);
    }
    if constexpr (TIES) {
      // every nonzero delta added 1 to exactly one bin: the histogram's total is nnz (not
      // for KNZ, whose nonzero deltas were counted by key and whose bin 0 holds the zeros too)
      if (!consumer_barrier(&S.cbar, cphase, abort_flag, wl)) {
        atomicOr(p.err, kErrTimeout);
        S.abort = 1;
        break;
      }
      // thread t holds bin t (and, for the window bins, bin t + 256)
      uint32_t hc[KG], hd[KG];
#pragma unroll
      for (int k = 0; k < KG; ++k) {
        hc[k] = S.hist[k][tid];
        S.hist[k][tid] = 0u;
        hd[k] = 0u;
        if (BM == kBinWindow && tid + 256u < NB) {
          hd[k] = S.hist[k][tid + 256u];
          S.hist[k][tid + 256u] = 0u;
        }
        if constexpr (!KNZ) {
          uint32_t w = hc[k] + hd[k];
#pragma unroll
          for (int s = 16; s >= 1; s >>= 1) w += __shfl_xor_sync(0xFFFFFFFFu, w, s);
          if (lane == 0) S.red_nz[k][warp] = w;
        }
      }
      if constexpr (!KNZ) {
        if (!consumer_barrier(&S.cbar, cphase, abort_flag, wl)) {
          atomicOr(p.err, kErrTimeout);
          S.abort = 1;
          break;
        }
      }
      const uint32_t grp = p.blk_group[b];
      const uint32_t len = p.blk_len[b];
#pragma unroll
      for (int k = 0; k < KG; ++k) {
        if ((uint32_t)k >= kc) break;
        uint32_t nzk = 0;
        if constexpr (!KNZ) {
#pragma unroll
          for (int w = 0; w < kIxConsumers / 32; ++w) nzk += S.red_nz[k][w];
          if (tid == 0) p.nnz[(uint64_t)(i0 + k) * p.n_blocks + b] = nzk;
        }
        const uint64_t x = (uint64_t)(i0 + k) * p.n_groups + grp;
        if constexpr (BM == kBinCoarse) {
          unsigned long long c = hc[k];
          if (tid == 0) c += len - nzk;  // zero deltas have key 0
          if (p.unit_hist) p.unit_hist[(((uint64_t)(i0 + k) * p.n_blocks + b) << 8) + tid] = (uint32_t)c;
          if (c) atomicAdd(&p.coarse[x * 256u + tid], c);
        } else {
          // bin 0 (below the window) only counts toward nnz; bins 1..384 are the window's
          // keys; bin 385 is above it
          if (tid > 0 && hc[k]) atomicAdd(&p.wfine[x * kWinKeys + tid - 1u], (unsigned long long)hc[k]);
          const uint32_t j = tid + 256u;
          if (j <= kWinKeys && hd[k]) atomicAdd(&p.wfine[x * kWinKeys + j - 1u], (unsigned long long)hd[k]);
          if (j == kWinKeys + 1u && hd[k]) atomicAdd(&p.wabove[x], (unsigned long long)hd[k]);
        }
      }
    }
    if (!consumer_barrier(&S.cbar, cphase, abort_flag, wl)) {
      atomicOr(p.err, kErrTimeout);
      S.abort = 1;
      break;
    }
  }
}

// coarse select: bin e* of the upper 8 key bits holding the k-th largest key, and the
// rank of that key inside the bin
__global__ void ties_coarse_select(const IndexLaunch p) {
  uint64_t x = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (x >= (uint64_t)p.K * p.n_groups) return;
  if (p.gmiss && p.gmiss[x] == 0u) return;  // its window already gave the threshold
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
  if (p.miss && *p.miss == 0u) return;  // windowed thresholds: no pair needs this pass
  const uint32_t G = (p.K + KG - 1) / KG;
  const uint64_t n_items = p.n_blocks * G;
  const uint32_t tid = threadIdx.x;
  // items (block, group of KG experts) in a grid-stride loop: a grid of resident CTAs
  for (uint64_t it = blockIdx.x; it < n_items; it += gridDim.x) {
    const uint64_t b = it / G;
    const uint32_t i0 = (uint32_t)(it % G) * KG;
    const uint32_t kc = min((uint32_t)KG, p.K - i0);
    if (!checked_item<true>(p, b, i0, kc, BF16 ? 2u : 4u)) continue;  // uniform over the CTA
    const uint32_t grp = p.blk_group[b];

    uint32_t estar[KG];
    uint32_t want = 0u;  // bit k: expert i0+k may hold keys in its bin e*
#pragma unroll
    for (int k = 0; k < KG; ++k) {
      estar[k] = kNoBin;
      if ((uint32_t)k < kc) {
        uint32_t i = i0 + k;
        uint32_t es = p.estar[(uint64_t)i * p.n_groups + grp];
        uint64_t u = (uint64_t)i * p.n_blocks + b;
        const bool read = (!p.mask || ((p.mask[b] >> i) & 1u)) &&  // TIES_MASKED: selected blocks only
                          (!p.gmiss || p.gmiss[(uint64_t)i * p.n_groups + grp] != 0u);  // windowed: missed pairs only
        if (read && es != kNoBin && p.nnz[u] != 0u && (ties_key(p.maxabs[u]) >> 7) >= es) {
          estar[k] = es;
          want |= 1u << k;
        }
      }
    }
    if (want == 0u) continue;  // uniform over the CTA
    if (p.thr_reads && threadIdx.x == 0)
      atomicAdd(p.thr_reads, (unsigned long long)__popc(want) * p.blk_len[b] * (BF16 ? 2u : 4u));
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
        for (int e = 0; e < V; e += 2)
          ties_fine2(__fsub_rn(xe[e], xb[e]), __fsub_rn(xe[e + 1], xb[e + 1]), estar[k], su32(&s_fine[k][0]));
      }
    }
    __syncthreads();
    for (uint32_t x = tid; x < (uint32_t)KG * 128u; x += 256u) {
      uint32_t k = x >> 7, m = x & 127u;
      if (!((want >> k) & 1u)) continue;
      uint32_t c = s_fine[k][m];
      if (c) atomicAdd(&p.fine[((uint64_t)(i0 + k) * p.n_groups + grp) * 128u + m], (unsigned long long)c);
    }
    __syncthreads();  // the next item clears s_fine
  }
}

__global__ void ties_fine_select(const IndexLaunch p) {
  uint64_t x = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (x >= (uint64_t)p.K * p.n_groups) return;
  if (p.gmiss && p.gmiss[x] == 0u) return;  // its window already gave the threshold
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

// TIES after masking: the coarse bins of (expert i, group) summed over a window of blocks:
// a selected block adds its catalog histogram, an unselected one adds its elements to bin 0
// (omitted entries are zeros).  One CTA per (expert, window of kMaskWin blocks); thread e
// owns bin e and adds its sum for each group the window touches.
constexpr uint32_t kMaskWin = 256;

__global__ void __launch_bounds__(256) ties_masked_coarse(const IndexLaunch p, uint32_t n_win) {
  const uint32_t i = blockIdx.x / n_win;
  const uint64_t b0 = (uint64_t)(blockIdx.x % n_win) * kMaskWin;
  const uint64_t b1 = b0 + kMaskWin < p.n_blocks ? b0 + kMaskWin : p.n_blocks;
  const uint32_t e = threadIdx.x;
  const uint32_t* uh = p.unit_hist + ((uint64_t)i * p.n_blocks << 8);
  uint32_t grp = p.blk_group[b0];
  unsigned long long acc = 0;
  for (uint64_t b = b0; b < b1; ++b) {
    const uint32_t g = p.blk_group[b];
    if (g != grp) {
      if (acc) atomicAdd(&p.coarse[((uint64_t)i * p.n_groups + grp) * 256u + e], acc);
      acc = 0;
      grp = g;
    }
    if ((p.mask[b] >> i) & 1u) acc += uh[(b << 8) + e];
    else if (e == 0) acc += p.blk_len[b];
  }
  if (acc) atomicAdd(&p.coarse[((uint64_t)i * p.n_groups + grp) * 256u + e], acc);
}

// ---- TIES thresholds with a predicted window ----------------------------------------------
//
// The threshold of a trim group is the k-th largest key of its deltas.  A sample predicts
// the coarse bin e (upper 8 key bits) that holds it: from every block of the group, 32
// vectors at jittered, evenly spaced positions (every vector of a block of at most 4096
// elements), binned like the coarse catalog — every block contributes because the scale of
// the deltas changes from block to block; e is the bin of the k_s-th largest sampled key,
// k_s = max(1, floor(rho * sampled elements)).  The catalog pass then counts the 384 keys
// of the window starting at L = 128 clamp(e - 1, 0, 253) at full resolution, plus the keys
// above it, and ties_window_finish takes the threshold from those counts.  A pair whose
// threshold lies outside its window is marked, and the two-level select (coarse pass over
// the marked pairs' groups, coarse select, fine pass, fine select) runs for the marked
// pairs only; it does nothing when none is marked.  The prediction affects only which of
// the two exact paths gives a threshold, never its value.
constexpr uint32_t kSampleSpan = 64;  // blocks of one group per sampling CTA

template <bool BF16, int KG>
__global__ void __launch_bounds__(256) ties_sample_kernel(const IndexLaunch p) {
  constexpr uint32_t V = BF16 ? 8u : 4u;
  __shared__ uint32_t hist[KG][256];
  __shared__ unsigned long long s_n;  // sampled elements
  const uint2 span = p.samp_span[blockIdx.x];  // {group, first block}: up to kSampleSpan blocks
  const uint32_t g = span.x, i0 = blockIdx.y * KG;
  const uint32_t kc = min((uint32_t)KG, p.K - i0);
  if (kChecked && (g >= p.n_groups || i0 >= p.K)) {  // uniform over the CTA
    if (threadIdx.x == 0) atomicOr(p.err, kErrBounds);
    return;
  }
  const uint32_t tid = threadIdx.x, warp = tid >> 5, lane = tid & 31u;
  for (uint32_t x = tid; x < (uint32_t)KG * 256u; x += blockDim.x) (&hist[0][0])[x] = 0u;
  if (tid == 0) s_n = 0;
  __syncthreads();
  const uint64_t gb1 = p.n_groups == 1 ? p.n_blocks : p.grp_blk0[g + 1];
  const uint64_t b1 = min((uint64_t)span.y + kSampleSpan, gb1);
  unsigned long long my_n = 0;
  for (uint64_t b = span.y + warp; b < b1; b += 8) {
    if (!checked_item<false>(p, b, i0, kc, BF16 ? 2u : 4u)) continue;  // uniform over the warp
    const uint32_t len = p.blk_len[b];
    const uint64_t off = p.blk_off[b];
    const uint32_t nvec = (len + V - 1) / V;
    const bool every = len <= 4096u;
    const uint32_t per = every ? 1u : nvec / 32u;
    for (uint32_t v0 = lane; v0 < (every ? nvec : 32u); v0 += 32u) {
      uint32_t v = v0;
      if (!every) {  // a position in stretch v0 from a hash of (block, stretch)
        uint32_t h = (uint32_t)b * 0x9E3779B1u ^ (v0 + 1u) * 0x85EBCA77u;
        h ^= h >> 15;
        h *= 0x2C1B3C6Du;
        h ^= h >> 12;
        v = v0 * per + h % per;
      }
      my_n += min(V, len - v * V);
      // every checkpoint's vector in flight at once: one memory round trip per position
      const uint4 rb = load_vec_raw(p.base, BF16, off, v, len);
      uint4 re[KG];
#pragma unroll
      for (int k = 0; k < KG; ++k)
        if ((uint32_t)k < kc) re[k] = load_vec_raw(p.experts.p[i0 + k], BF16, off, v, len);
      float xb[V];
      unpack<BF16>(rb, xb);
#pragma unroll
      for (int k = 0; k < KG; ++k) {
        if ((uint32_t)k >= kc) break;
        float xe[V];
        unpack<BF16>(re[k], xe);
#pragma unroll
        for (uint32_t e = 0; e < V; ++e) {
          const float d = __fsub_rn(xe[e], xb[e]);
          if (d != 0.0f) atomicAdd(&hist[k][ties_key(d) >> 7], 1u);
        }
      }
    }
  }
#pragma unroll
  for (int s = 16; s >= 1; s >>= 1) my_n += __shfl_xor_sync(0xFFFFFFFFu, my_n, s);
  if (lane == 0) atomicAdd(&s_n, my_n);
  __syncthreads();
  for (uint32_t x = tid; x < kc * 256u; x += blockDim.x) {
    const uint32_t k = x >> 8, e = x & 255u;
    if (hist[k][e]) atomicAdd(&p.shist[((uint64_t)(i0 + k) * p.n_groups + g) * 256u + e], (unsigned long long)hist[k][e]);
  }
  if (tid == 0 && blockIdx.y == 0) atomicAdd(&p.scnt[g], s_n);
}

// the window of each (expert, group) from its sampled coarse bins
__global__ void ties_window_select(const IndexLaunch p) {
  const uint64_t x = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (x >= (uint64_t)p.K * p.n_groups) return;
  const uint32_t g = (uint32_t)(x % p.n_groups);
  unsigned long long ks = (unsigned long long)floor((double)p.density * (double)p.scnt[g]);
  if (ks == 0) ks = 1;
  const unsigned long long* h = p.shist + x * 256u;
  uint32_t e = 0;
  unsigned long long cum = 0;
  for (int j = 255; j >= 0; --j) {
    cum += h[j];
    if (cum >= ks) {
      e = (uint32_t)j;
      break;
    }
  }
  const uint32_t lo = e == 0 ? 0u : min(e - 1u, 253u);
  p.wlo[x] = lo << 7;
}

// the threshold of each (expert, group) from its window counts, or a mark for the
// two-level select when it lies outside the window
__global__ void ties_window_finish(const IndexLaunch p) {
  const uint64_t x = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (x >= (uint64_t)p.K * p.n_groups) return;
  const uint32_t g = (uint32_t)(x % p.n_groups);
  const unsigned long long k = p.kth[g];
  if (k == 0) {
    p.tau[x] = kTauNone;
    return;
  }
  const unsigned long long above = p.wabove[x];
  const uint32_t L = p.wlo[x];
  if (above < k) {
    const unsigned long long r = k - above;
    const unsigned long long* f = p.wfine + x * kWinKeys;
    unsigned long long cum = 0;
    for (int j = (int)kWinKeys - 1; j >= 0; --j) {
      cum += f[j];
      if (cum >= r) {
        p.tau[x] = L + (uint32_t)j;
        return;
      }
    }
    if (L == 0) {  // every uncounted delta is an exact zero, key 0
      p.tau[x] = 0;
      return;
    }
  }
  p.gmiss[x] = 1u;
  atomicOr(p.miss, 1u);
}

// the TIES threshold from the coarse bins of the whole family: select the bin, count
// the lower key bits inside it (a second pass over the blocks that can reach it; experts
// addressed with origin 0), select the threshold
template <bool BF16, int KG>
cudaError_t ties_finish_t(const IndexLaunch& p, cudaStream_t st) {
  const uint32_t G = (p.K + KG - 1) / KG;
  const uint64_t nsel = (uint64_t)p.K * p.n_groups;
  const unsigned sgrid = (unsigned)((nsel + 127) / 128);
  int dev = 0, sms = 0;
  cudaError_t e;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
  int per_sm = 0;  // resident CTAs of 256 threads; items by grid stride
  if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, ties_fine_kernel<BF16, KG>, 256, 0)) != cudaSuccess)
    return e;
  uint64_t fgrid = (uint64_t)sms * (per_sm > 0 ? per_sm : 1);
  if (fgrid > p.n_blocks * G) fgrid = p.n_blocks * G;
  if (fgrid == 0) fgrid = 1;
  ties_coarse_select<<<sgrid, 128, 0, st>>>(p);
  ties_fine_kernel<BF16, KG><<<(unsigned)fgrid, 256, 0, st>>>(p);
  ties_fine_select<<<sgrid, 128, 0, st>>>(p);
  count_launches(3);
  return cudaGetLastError();
}

// one persistent launch of the catalog kernel with binning mode BM
template <bool BF16, int KG, int BM>
cudaError_t launch_pass(const IndexLaunch& p, uint32_t G, uint64_t n_items, int sms, cudaStream_t st) {
  constexpr bool ties = BM != kBinNone;
  constexpr uint32_t NB = BM == kBinNone ? 1u : (BM == kBinWindow ? kWinBins : 256u);
  const size_t smem = sizeof(IxSmem<KG, IxGeo<ties, KG>::kSlots, IxGeo<ties, KG>::kSlotBytes, NB>);
  static_assert(IxGeo<ties, KG>::kCtasPerSm *
                        (sizeof(IxSmem<KG, IxGeo<ties, KG>::kSlots, IxGeo<ties, KG>::kSlotBytes, NB>) + 1024) <=
                    228u * 1024u,
                "the CTAs per SM that the grid assumes fit one SM's shared memory");
  uint64_t grid = (uint64_t)sms * IxGeo<ties, KG>::kCtasPerSm;
  if (grid > n_items) grid = n_items;
  cudaError_t e;
  if ((e = launch_fill(p.work, 0, sizeof(unsigned long long), st)) != cudaSuccess) return e;
  auto k = index_tma_kernel<BF16, KG, BM>;
  if ((e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)) != cudaSuccess) return e;
  k<<<(unsigned)grid, kIxThreads, smem, st>>>(p, G, n_items, p.work);
  count_launches(1);
  return cudaGetLastError();
}

template <bool BF16, int KG>
cudaError_t launch_t(const IndexLaunch& p, cudaStream_t st) {
  const uint32_t G = (p.K + KG - 1) / KG;
  const uint64_t n_items = (p.b_end - p.b_begin) * G;
  if (n_items == 0) return cudaSuccess;
  if (n_items > 0x7FFFFFFFull) return cudaErrorInvalidValue;
  const bool ties = p.coarse != nullptr;
  int dev = 0, sms = 0;
  cudaError_t e;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
  if (!ties) return launch_pass<BF16, KG, kBinNone>(p, G, n_items, sms, st);
  if (!p.wlo) {  // the two-level select for every pair
    if ((e = launch_pass<BF16, KG, kBinCoarse>(p, G, n_items, sms, st)) != cudaSuccess) return e;
    if (p.defer_ties_select) return cudaSuccess;
    return ties_finish_t<BF16, KG>(p, st);
  }
  // predicted windows: sample, windowed catalog pass, thresholds from the windows, then the
  // two-level select for the pairs whose threshold left its window (a no-op when none did)
  const uint64_t nsel = (uint64_t)p.K * p.n_groups;
  ties_sample_kernel<BF16, KG><<<dim3(p.n_samp_spans, G), 256, 0, st>>>(p);
  ties_window_select<<<(unsigned)((nsel + 127) / 128), 128, 0, st>>>(p);
  count_launches(2);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  if ((e = launch_pass<BF16, KG, kBinWindow>(p, G, n_items, sms, st)) != cudaSuccess) return e;
  ties_window_finish<<<(unsigned)((nsel + 127) / 128), 128, 0, st>>>(p);
  count_launches(1);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  if ((e = launch_pass<BF16, KG, kBinCoarse>(p, G, n_items, sms, st)) != cudaSuccess) return e;
  return ties_finish_t<BF16, KG>(p, st);
}

template <bool BF16, int KG>
cudaError_t window_begin_t(const IndexLaunch& p, cudaStream_t st) {
  const uint32_t G = (p.K + KG - 1) / KG;
  const uint64_t nsel = (uint64_t)p.K * p.n_groups;
  if (p.n_samp_spans == 0 || nsel == 0) return cudaSuccess;
  ties_sample_kernel<BF16, KG><<<dim3(p.n_samp_spans, G), 256, 0, st>>>(p);
  ties_window_select<<<(unsigned)((nsel + 127) / 128), 128, 0, st>>>(p);
  count_launches(2);
  return cudaGetLastError();
}

template <bool BF16, int KG>
cudaError_t pass_t(const IndexLaunch& p, bool window, cudaStream_t st) {
  const uint32_t G = (p.K + KG - 1) / KG;
  const uint64_t n_items = (p.b_end - p.b_begin) * G;
  if (n_items == 0) return cudaSuccess;
  if (n_items > 0x7FFFFFFFull) return cudaErrorInvalidValue;
  int dev = 0, sms = 0;
  cudaError_t e;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
  return window ? launch_pass<BF16, KG, kBinWindow>(p, G, n_items, sms, st)
                : launch_pass<BF16, KG, kBinCoarse>(p, G, n_items, sms, st);
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

cudaError_t launch_ties_window_begin(const IndexLaunch& p, cudaStream_t st) {
  if (!p.wlo || !p.coarse) return cudaErrorInvalidValue;
  const bool bf = p.dtype == MP_BF16;
  if (p.K <= 1) return bf ? window_begin_t<true, 1>(p, st) : window_begin_t<false, 1>(p, st);
  if (p.K <= 2) return bf ? window_begin_t<true, 2>(p, st) : window_begin_t<false, 2>(p, st);
  if (p.K <= 4) return bf ? window_begin_t<true, 4>(p, st) : window_begin_t<false, 4>(p, st);
  return bf ? window_begin_t<true, 8>(p, st) : window_begin_t<false, 8>(p, st);
}

cudaError_t launch_index_pass(const IndexLaunch& p, bool window, cudaStream_t st) {
  if (!p.wlo || !p.coarse) return cudaErrorInvalidValue;
  const bool bf = p.dtype == MP_BF16;
  if (p.K <= 1) return bf ? pass_t<true, 1>(p, window, st) : pass_t<false, 1>(p, window, st);
  if (p.K <= 2) return bf ? pass_t<true, 2>(p, window, st) : pass_t<false, 2>(p, window, st);
  if (p.K <= 4) return bf ? pass_t<true, 4>(p, window, st) : pass_t<false, 4>(p, window, st);
  return bf ? pass_t<true, 8>(p, window, st) : pass_t<false, 8>(p, window, st);
}

cudaError_t launch_ties_window_end(const IndexLaunch& p, cudaStream_t st) {
  if (!p.wlo || !p.coarse) return cudaErrorInvalidValue;
  const uint64_t nsel = (uint64_t)p.K * p.n_groups;
  if (nsel == 0) return cudaSuccess;
  ties_window_finish<<<(unsigned)((nsel + 127) / 128), 128, 0, st>>>(p);
  count_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_ties_masked(const IndexLaunch& p, cudaStream_t st) {
  if (!p.unit_hist || !p.mask || p.n_blocks == 0) return cudaErrorInvalidValue;
  const uint32_t n_win = (uint32_t)((p.n_blocks + kMaskWin - 1) / kMaskWin);
  ties_masked_coarse<<<p.K * n_win, 256, 0, st>>>(p, n_win);
  count_launches(1);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  return launch_ties_finish(p, st);
}

cudaError_t launch_ties_finish(const IndexLaunch& p, cudaStream_t st) {
  const bool bf = p.dtype == MP_BF16;
  if (p.K <= 1) return bf ? ties_finish_t<true, 1>(p, st) : ties_finish_t<false, 1>(p, st);
  if (p.K <= 2) return bf ? ties_finish_t<true, 2>(p, st) : ties_finish_t<false, 2>(p, st);
  if (p.K <= 4) return bf ? ties_finish_t<true, 4>(p, st) : ties_finish_t<false, 4>(p, st);
  return bf ? ties_finish_t<true, 8>(p, st) : ties_finish_t<false, 8>(p, st);
}

}  // namespace mp
