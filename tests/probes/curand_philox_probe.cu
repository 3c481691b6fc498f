// Test probe: cuRAND's device Philox4_32_10 generator, used to pin the oracle's Philox.
// curand_init(seed, subsequence, offset) then n calls of curand4(); one thread per request.
#include <curand_kernel.h>
#include <stdint.h>

__global__ void probe(const unsigned long long* seed, const unsigned long long* subseq,
                      const unsigned long long* offset, unsigned n, unsigned count, uint4* out) {
  unsigned t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= count) return;
  curandStatePhilox4_32_10_t st;
  curand_init(seed[t], subseq[t], offset[t], &st);
  for (unsigned k = 0; k < n; ++k) out[(unsigned long long)t * n + k] = curand4(&st);
}

extern "C" int curand_philox_probe(const unsigned long long* d_seed, const unsigned long long* d_subseq,
                                   const unsigned long long* d_offset, unsigned n, unsigned count, void* d_out) {
  probe<<<(count + 127) / 128, 128>>>(d_seed, d_subseq, d_offset, n, count, (uint4*)d_out);
  return cudaDeviceSynchronize() == cudaSuccess ? 0 : -1;
}
