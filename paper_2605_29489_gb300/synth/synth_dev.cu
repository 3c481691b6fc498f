// GPU fill of synthetic checkpoints: the same element recipe as the host fill
// (synth_core.h), launched over the family's block table so that an expert's
// per-block scale is looked up once per CTA.
#include <cuda_runtime.h>
#include <stdint.h>

#include "synth_core.h"

namespace {

__global__ void fill_base_kernel(int dtype, uint64_t key, uint64_t n, void* out) {
  uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  for (uint64_t j = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; j < n; j += stride) {
    float v = syn_base_f32(key, j);
    if (dtype == SYN_BF16) ((uint16_t*)out)[j] = syn_bf16_bits(v);
    else ((float*)out)[j] = v;
  }
}

// one CTA row per block; the expert buffer already holds a copy of the base
__global__ void fill_expert_kernel(int dtype, uint64_t key, uint64_t n_blk, const uint64_t* blk_off,
                                   const uint32_t* blk_len, const float* blk_scale, const void* base,
                                   void* out) {
  for (uint64_t b = blockIdx.y + (uint64_t)blockIdx.z * gridDim.y; b < n_blk;
       b += (uint64_t)gridDim.y * gridDim.z) {
    float s = blk_scale[b];
    if (s == 0.0f) continue;
    uint64_t off = blk_off[b];
    uint32_t len = blk_len[b];
    for (uint32_t k = blockIdx.x * blockDim.x + threadIdx.x; k < len; k += gridDim.x * blockDim.x) {
      uint64_t j = off + k;
      float bv = dtype == SYN_BF16 ? syn_bf16_to_f32(((const uint16_t*)base)[j]) : ((const float*)base)[j];
      float v = syn_expert_f32(key, bv, s, j);
      if (dtype == SYN_BF16) ((uint16_t*)out)[j] = syn_bf16_bits(v);
      else ((float*)out)[j] = v;
    }
  }
}

}  // namespace

extern "C" {

// Fill the first n elements of the base stream into the device buffer out.
int syn_dev_fill_base(int dtype, uint64_t seed, uint64_t n, void* out, void* stream) {
  if ((dtype != SYN_BF16 && dtype != SYN_F32) || (n > 0 && !out)) return -1;
  if (n == 0) return 0;
  cudaStream_t st = (cudaStream_t)stream;
  uint64_t blocks = (n + 255) / 256;
  if (blocks > 152ull * 64) blocks = 152ull * 64;
  fill_base_kernel<<<(unsigned)blocks, 256, 0, st>>>(dtype, syn_stream_key(seed, 0), n, out);
  return cudaGetLastError() == cudaSuccess ? 0 : -2;
}

// Fill expert `expert` (stream 1+expert) of an n-element family into out, given the
// stored base (device) and the device block table (start, length, scale per block).
int syn_dev_fill_expert(int dtype, uint64_t seed, uint32_t expert, uint64_t n, uint64_t n_blk,
                        const uint64_t* blk_off, const uint32_t* blk_len, const float* blk_scale,
                        uint32_t max_blk_len, const void* base, void* out, void* stream) {
  if ((dtype != SYN_BF16 && dtype != SYN_F32) || (n > 0 && (!out || !base))) return -1;
  if (n == 0) return 0;
  cudaStream_t st = (cudaStream_t)stream;
  size_t es = dtype == SYN_BF16 ? 2 : 4;
  if (cudaMemcpyAsync(out, base, n * es, cudaMemcpyDeviceToDevice, st) != cudaSuccess) return -2;
  if (n_blk == 0) return 0;
  unsigned gx = (unsigned)((max_blk_len + 255) / 256);
  if (gx > 64) gx = 64;
  if (gx == 0) gx = 1;
  uint64_t rows = n_blk;
  unsigned gy = (unsigned)(rows < 65535 ? rows : 65535);
  uint64_t gz64 = (rows + gy - 1) / gy;
  unsigned gz = (unsigned)(gz64 < 65535 ? gz64 : 65535);
  dim3 grid(gx, gy, gz);
  fill_expert_kernel<<<grid, 256, 0, st>>>(dtype, syn_stream_key(seed, 1u + expert), n_blk, blk_off, blk_len,
                                           blk_scale, base, out);
  return cudaGetLastError() == cudaSuccess ? 0 : -2;
}

}  // extern "C"
