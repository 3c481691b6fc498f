/*
 * Host (CPU) fill of synthetic checkpoint ranges, multithreaded with pthreads.
 * The element recipe is in synth_core.h; the GPU fill (synth_dev.cu) produces
 * the same bytes from the same header.
 */
#include <pthread.h>
#include <stddef.h>
#include <stdint.h>
#include <string.h>

#include "synth_core.h"

typedef struct {
  int dtype;
  uint64_t key;
  int is_base;
  uint64_t j0, n;
  const uint64_t* blk_off;
  const uint32_t* blk_len;
  const float* blk_scale;
  uint64_t n_blk;
  const void* base_stored;
  void* out;
} fill_job;

/* index of the last block whose start is <= j (blocks sorted by start), or n_blk if none */
static uint64_t find_block(const uint64_t* off, uint64_t n_blk, uint64_t j) {
  uint64_t lo = 0, hi = n_blk;
  while (lo < hi) {
    uint64_t mid = lo + (hi - lo) / 2;
    if (off[mid] <= j) lo = mid + 1; else hi = mid;
  }
  return lo == 0 ? n_blk : lo - 1;
}

static void fill_span(const fill_job* jb, uint64_t k0, uint64_t k1) {
  if (jb->is_base) {
    for (uint64_t k = k0; k < k1; ++k) {
      float v = syn_base_f32(jb->key, jb->j0 + k);
      if (jb->dtype == SYN_BF16) ((uint16_t*)jb->out)[k] = syn_bf16_bits(v);
      else ((float*)jb->out)[k] = v;
    }
    return;
  }
  uint64_t b = find_block(jb->blk_off, jb->n_blk, jb->j0 + k0);
  for (uint64_t k = k0; k < k1; ++k) {
    uint64_t j = jb->j0 + k;
    while (b + 1 < jb->n_blk && jb->blk_off[b + 1] <= j) ++b;
    float s = 0.0f;
    if (b < jb->n_blk && j >= jb->blk_off[b] && j < jb->blk_off[b] + jb->blk_len[b]) s = jb->blk_scale[b];
    float base = jb->dtype == SYN_BF16 ? syn_bf16_to_f32(((const uint16_t*)jb->base_stored)[k])
                                       : ((const float*)jb->base_stored)[k];
    float v = s == 0.0f ? base : syn_expert_f32(jb->key, base, s, j);
    if (jb->dtype == SYN_BF16) ((uint16_t*)jb->out)[k] = syn_bf16_bits(v);
    else ((float*)jb->out)[k] = v;
  }
}

typedef struct { const fill_job* jb; uint64_t k0, k1; } thread_arg;

static void* thread_main(void* p) {
  thread_arg* a = (thread_arg*)p;
  fill_span(a->jb, a->k0, a->k1);
  return NULL;
}

/*
 * Fill elements [j0, j0+n) of one stream into out[0..n).
 * stream 0 is the base; stream 1+i is expert i, which needs the stored base
 * values of the same range (base_stored[0..n)) and the block table
 * (start offset, length and scale of every block, sorted by start).
 * Elements that lie in no block get the base value (zero delta).
 * Returns 0, or -1 on a bad argument.
 */
int syn_fill_range(int dtype, uint64_t seed, uint32_t stream, uint64_t j0, uint64_t n,
                   const uint64_t* blk_off, const uint32_t* blk_len, const float* blk_scale,
                   uint64_t n_blk, const void* base_stored, void* out, int nthreads) {
  if ((dtype != SYN_BF16 && dtype != SYN_F32) || (n > 0 && out == NULL)) return -1;
  if (stream != 0 && n > 0 && (base_stored == NULL || (n_blk > 0 && (!blk_off || !blk_len || !blk_scale))))
    return -1;
  fill_job jb;
  jb.dtype = dtype;
  jb.key = syn_stream_key(seed, stream);
  jb.is_base = stream == 0;
  jb.j0 = j0;
  jb.n = n;
  jb.blk_off = blk_off;
  jb.blk_len = blk_len;
  jb.blk_scale = blk_scale;
  jb.n_blk = n_blk;
  jb.base_stored = base_stored;
  jb.out = out;
  if (nthreads < 1) nthreads = 1;
  if (nthreads > 256) nthreads = 256;
  if (n < (uint64_t)nthreads * 65536u) nthreads = 1;
  if (nthreads == 1) {
    fill_span(&jb, 0, n);
    return 0;
  }
  pthread_t th[256];
  thread_arg args[256];
  int started = 0;
  for (int t = 0; t < nthreads; ++t) {
    args[t].jb = &jb;
    args[t].k0 = n * (uint64_t)t / (uint64_t)nthreads;
    args[t].k1 = n * (uint64_t)(t + 1) / (uint64_t)nthreads;
    if (pthread_create(&th[t], NULL, thread_main, &args[t]) != 0) {
      fill_span(&jb, args[t].k0, args[t].k1);
      th[t] = 0;
      continue;
    }
    ++started;
  }
  for (int t = 0; t < nthreads; ++t)
    if (th[t]) pthread_join(th[t], NULL);
  (void)started;
  return 0;
}

/* the SplitMix64 output function, exported so the host scale table can use it */
uint64_t syn_mix64_export(uint64_t z) { return syn_mix64(z); }
uint64_t syn_stream_key_export(uint64_t seed, uint32_t stream) { return syn_stream_key(seed, stream); }
