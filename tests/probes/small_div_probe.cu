// Exhaustive check of the merge kernel's division by a small count against the CUDA
// IEEE division: every finite fp32 numerator other than -0 (all 2^32 bit patterns but
// Inf, NaN and 0x80000000) and every count c = 1..32.  Reports the number of mismatches
// and one of them.
#include <stdint.h>

#include "small_div.cuh"

namespace {

__global__ void small_div_check(unsigned long long* bad, unsigned int* first) {
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  unsigned long long mine = 0;
  for (uint64_t x = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; x < (1ull << 32); x += stride) {
    const float a = __uint_as_float((uint32_t)x);
    if (!isfinite(a) || (uint32_t)x == 0x80000000u) continue;
    for (uint32_t c = 1; c <= 32; ++c) {
      const float cf = (float)c;
      const float y = __fdiv_rn(1.0f, cf);
      const float got = mp::div_small(a, cf, y);
      const float want = __fdiv_rn(a, cf);
      if (__float_as_uint(got) != __float_as_uint(want)) {
        ++mine;
        if (atomicCAS(first + 2, 0u, 1u) == 0u) {
          first[0] = (uint32_t)x;
          first[1] = c;
        }
      }
    }
  }
  if (mine) atomicAdd(bad, mine);
}

}  // namespace

// bad[0] = mismatches; first[0..1] = (numerator bits, c) of one mismatch, first[2] its
// claim flag; returns the CUDA error code of the run
extern "C" int small_div_probe(unsigned long long* bad, unsigned int* first) {
  int dev = 0, sms = 0;
  cudaError_t e;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return (int)e;
  if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return (int)e;
  small_div_check<<<sms * 8, 256>>>(bad, first);
  return (int)cudaDeviceSynchronize();
}
