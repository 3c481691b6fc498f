/*
 * Seeded synthetic checkpoint families: the element-level generator.
 *
 * This header is the one piece of code that both the CPU oracle's test inputs
 * and the GPU path's inputs come from.  It holds none of the merge method's
 * arithmetic: it only turns (seed, stream, element index, block scale) into a
 * base or expert element.  It compiles as plain C (host, gcc) and as CUDA
 * device code (nvcc), and every floating-point step is a single IEEE
 * round-to-nearest operation, so both compilations produce identical bytes.
 *
 * Recipe (one element j of the flat checkpoint, stream 0 = base, 1+i = expert i):
 *   z_j      = Irwin-Hall sum of four 32-bit uniform words, centred and scaled
 *              to unit variance (an approximate N(0,1), |z| <= 2*sqrt(3));
 *   base     = cast(0.02f * z_j^(0))
 *   expert_i = cast(float(base) + s_{i,b} * z_j^(1+i))   (fp32 mul, then add)
 * where cast is bf16 round-to-nearest-even or the fp32 identity and s_{i,b}
 * is the per-(expert, block) scale from the family's scale table.
 *
 * The uniform words come from the SplitMix64 output function (Steele, Lea and
 * Flood, "Fast splittable pseudorandom number generators", OOPSLA 2014)
 * applied to a Weyl sequence keyed by (seed, stream).
 */
#ifndef MP_SYNTH_CORE_H
#define MP_SYNTH_CORE_H

#include <stdint.h>

#ifdef __CUDACC__
#define SYN_FN __host__ __device__ __forceinline__
#else
#define SYN_FN static inline
#endif

#define SYN_GAMMA 0x9E3779B97F4A7C15ULL
/* sqrt(3) * 2^-32 rounded to fp32: maps the centred Irwin-Hall sum to unit variance */
#define SYN_NORM_SCALE 0x1.bb67aep-32f
#define SYN_BASE_STD 0.02f

enum { SYN_BF16 = 0, SYN_F32 = 1 };

SYN_FN uint64_t syn_mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

/* key of one random stream: stream 0 is the base, stream 1+i is expert i */
SYN_FN uint64_t syn_stream_key(uint64_t seed, uint32_t stream) {
  return syn_mix64(seed + SYN_GAMMA * ((uint64_t)stream + 1u));
}

SYN_FN float syn_mul(float a, float b) {
#ifdef __CUDA_ARCH__
  return __fmul_rn(a, b);
#else
  return a * b;
#endif
}

SYN_FN float syn_add(float a, float b) {
#ifdef __CUDA_ARCH__
  return __fadd_rn(a, b);
#else
  return a + b;
#endif
}

SYN_FN float syn_i64_to_f32(int64_t v) {
#ifdef __CUDA_ARCH__
  return __ll2float_rn((long long)v);
#else
  return (float)v;
#endif
}

SYN_FN uint32_t syn_f32_bits(float f) {
#ifdef __CUDA_ARCH__
  return __float_as_uint(f);
#else
  union { float f; uint32_t u; } c;
  c.f = f;
  return c.u;
#endif
}

SYN_FN float syn_bits_f32(uint32_t u) {
#ifdef __CUDA_ARCH__
  return __uint_as_float(u);
#else
  union { float f; uint32_t u; } c;
  c.u = u;
  return c.f;
#endif
}

/* fp32 -> bf16 bits, round to nearest even (quiet NaN kept quiet) */
SYN_FN uint16_t syn_bf16_bits(float f) {
  uint32_t u = syn_f32_bits(f);
  if ((u & 0x7FFFFFFFu) > 0x7F800000u) return (uint16_t)((u >> 16) | 0x40u);
  return (uint16_t)((u + 0x7FFFu + ((u >> 16) & 1u)) >> 16);
}

SYN_FN float syn_bf16_to_f32(uint16_t h) { return syn_bits_f32(((uint32_t)h) << 16); }

/* approximately standard normal variate for element j of the stream with key `key` */
SYN_FN float syn_normal(uint64_t key, uint64_t j) {
  uint64_t w0 = syn_mix64(key + SYN_GAMMA * (2u * j + 1u));
  uint64_t w1 = syn_mix64(key + SYN_GAMMA * (2u * j + 2u));
  uint64_t s = (w0 & 0xFFFFFFFFu) + (w0 >> 32) + (w1 & 0xFFFFFFFFu) + (w1 >> 32);
  int64_t c = (int64_t)s - ((int64_t)1 << 33);
  return syn_mul(syn_i64_to_f32(c), SYN_NORM_SCALE);
}

/* base element j as fp32 (before storage rounding) */
SYN_FN float syn_base_f32(uint64_t base_key, uint64_t j) {
  return syn_mul(SYN_BASE_STD, syn_normal(base_key, j));
}

/* expert element j as fp32 (before storage rounding), from the STORED base value */
SYN_FN float syn_expert_f32(uint64_t expert_key, float base_stored, float scale, uint64_t j) {
  return syn_add(base_stored, syn_mul(scale, syn_normal(expert_key, j)));
}

#endif /* MP_SYNTH_CORE_H */
