// Inline-PTX helpers for the bulk-copy pipelines: mbarriers with bounded waits and the
// 1-D TMA bulk copy global -> shared (cp.async.bulk, completion counted in bytes on an
// mbarrier).  Every wait here has an iteration limit so that no kernel can hang.
#pragma once

#include <stdint.h>

namespace mp {

// A sleeping wait suspends the thread for up to kSuspendHintNs per try_wait round (it resumes
// as soon as the phase completes), so waiting warps do not spin on the issue slots that working
// warps need; a polling wait returns after each round.  Which one a kernel uses is a measured
// choice (the merge kernel sleeps, the catalog kernel polls).  kWaitLimit rounds bound every
// wait to a few seconds.
constexpr uint32_t kSuspendHintNs = 2000;
constexpr uint32_t kWaitLimit = 1u << 21;  // try_wait rounds before a wait gives up

// the limit a kernel uses for its pipeline waits: the launch's (a test setting) or the default
__device__ __forceinline__ uint32_t wait_limit_of(uint32_t launch_limit) {
  return launch_limit ? launch_limit : kWaitLimit;
}

__device__ __forceinline__ uint32_t su32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(su32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_fence_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(su32(bar)), "r"(bytes) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(su32(bar)) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(su32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// try_wait that may suspend the thread for up to kSuspendHintNs
__device__ __forceinline__ bool mbar_try_wait_sleep(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(su32(bar)), "r"(parity), "r"(kSuspendHintNs)
      : "memory");
  return ok != 0;
}

// bounded wait for the phase with the given parity; false on expiry (after `limit` rounds)
// or when *abort is set
template <bool SLEEP = false>
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, volatile int* abort,
                                          uint32_t limit = kWaitLimit) {
  for (uint32_t k = 0; k < limit; ++k) {
    if (SLEEP ? mbar_try_wait_sleep(bar, parity) : mbar_try_wait(bar, parity)) return true;
    if ((k & 15u) == 15u && *abort) return false;
  }
  return false;
}

// bounded wait that ignores the abort flag (drains copies still in flight before exit)
__device__ __forceinline__ void mbar_wait_drain(uint64_t* bar, uint32_t parity) {
  for (uint32_t k = 0; k < kWaitLimit; ++k)
    if (mbar_try_wait(bar, parity)) return;
}

// Orders the shared-memory accesses this thread has observed before the async-proxy writes
// of a bulk copy it issues next.  The producer calls it after acquiring a slot's "empty"
// mbarrier and before refilling the slot: the consumers' reads of the old contents are
// generic-proxy accesses, the refill an async-proxy write, and only a proxy fence orders
// the two (without it a refill can land before a consumer's read has been performed).
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void tma_load_1d(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(su32(dst)),
      "l"(src), "r"(bytes), "r"(su32(bar))
      : "memory");
}

// every lane of the warp waits (each acquires the barrier); the outcome is made uniform
// across the warp so that a give-up never splits a warp
template <bool SLEEP = false>
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort,
                                          uint32_t limit = kWaitLimit) {
  const bool ok = mbar_wait<SLEEP>(bar, parity, abort, limit);
  return __all_sync(0xFFFFFFFFu, ok);
}

// barrier over the consumer warps only (bar counts one arrival per warp), with a bounded
// wait: a warp that has given up cannot leave the others blocked; phase counts the uses
__device__ __forceinline__ bool consumer_barrier(uint64_t* bar, uint32_t& phase, volatile int* abort,
                                                 uint32_t limit = kWaitLimit) {
  __syncwarp();
  if ((threadIdx.x & 31u) == 0) mbar_arrive(bar);
  const bool ok = warp_wait(bar, phase & 1u, abort, limit);
  ++phase;
  return ok;
}

}  // namespace mp
