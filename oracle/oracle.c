/*
 * CPU oracle for the budgeted, mask-aware merge.  TEST INFRASTRUCTURE ONLY:
 * the product path never loads this file's library; the tests, the smoke
 * check and the benchmark's CPU baseline do.  Plain single-threaded C, built
 * with -ffp-contract=off so every operation is the one written here.
 *
 * Notation follows the paper: M_0 is the base, M_i (i = 1..K, stored here as
 * i = 0..K-1) the experts, Delta_{i,t,b} = M_i[t,b] - M_0[t,b] (Sec. 2), A the
 * access mask over units (i,t,b) (Eq. 2), c_{i,t,b} the read cost (Eq. 3),
 * B the expert-read budget, Psi_op the budgeted operator (Eq. 4).
 *
 * Pins (tests outside this file that fix each function to something other
 * than itself) are listed per function.  Fidelity metrics (relative l2, P95
 * block deviation) are not computed here.
 */
#include "oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

/* ---------------------------------------------------------------------------------------
 * Element conversion.  bf16 is the upper half of an IEEE binary32; rounding to
 * bf16 is round-to-nearest-even on the dropped 16 bits.
 * Pins: torch's CPU bfloat16 conversion on random and edge values; a NaN stays a NaN,
 * also one whose payload lies only in the dropped bits.
 * ------------------------------------------------------------------------------------- */
static uint32_t f2u(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  return u;
}
static float u2f(uint32_t u) {
  float f;
  memcpy(&f, &u, 4);
  return f;
}

float orc_bf16_to_f32(uint16_t h) { return u2f((uint32_t)h << 16); }

uint16_t orc_f32_to_bf16(float f) {
  uint32_t u = f2u(f);
  if ((u & 0x7FFFFFFFu) > 0x7F800000u) return (uint16_t)((u >> 16) | 0x0040u); /* NaN stays NaN */
  uint32_t lower = u & 0xFFFFu;
  uint32_t upper = u >> 16;
  if (lower > 0x8000u || (lower == 0x8000u && (upper & 1u))) upper += 1u; /* ties to even */
  return (uint16_t)upper;
}

static float load_elem(int dtype, const void* p, uint64_t k) {
  if (dtype == ORC_BF16) return orc_bf16_to_f32(((const uint16_t*)p)[k]);
  return ((const float*)p)[k];
}

static void store_elem(int dtype, void* p, uint64_t k, float v) {
  if (dtype == ORC_BF16) ((uint16_t*)p)[k] = orc_f32_to_bf16(v);
  else ((float*)p)[k] = v;
}

static int is_finite_f(float v) { return (f2u(v) & 0x7F800000u) != 0x7F800000u; }

/* TIES magnitude key: the 15 magnitude bits of |delta| rounded to bf16.  Reading: the
   trim compares magnitudes at bf16 resolution (a radix select over bf16 bit patterns).
   Pin: torch bf16 conversion of |delta|. */
uint32_t orc_ties_key(float delta) { return (uint32_t)orc_f32_to_bf16(fabsf(delta)) & 0x7FFFu; }

/* ---------------------------------------------------------------------------------------
 * Block statistics (the catalog's lightweight statistics, Sec. 3 "Catalog"; the
 * Analyze reads of Sec. 2).  For one expert block:
 *   nnz    = #{k : delta_k != 0}
 *   maxabs = max_k |delta_k|
 *   norm   = ||Delta_{i,t,b}||_2 = sqrt(sum_k delta_k^2)
 * The paper fixes no precision or summation order.  The norm decides the plan (its
 * score), so both implementations use one fp32 order:
 *   - the block is cut into 16-byte vectors of V elements (V = 8 bf16 or 4 fp32); a
 *     partial last vector is padded with zero deltas;
 *   - 256 lanes; lane l owns vectors l, l+256, l+512, ... and accumulates
 *     acc = fma(delta, delta, acc) over its vectors' elements in increasing index order;
 *   - the 256 lane sums are combined by a butterfly inside each group of 32 lanes
 *     (p[l] += p[l^s] for s = 16, 8, 4, 2, 1), then over the 8 group sums
 *     (g[w] += g[w^s] for s = 4, 2, 1);
 *   - norm = correctly rounded sqrt of that sum.
 * Pins: closed form on integer-valued deltas (exact in any order); fp64 sum of squares
 * within the fp32 summation error bound; brute-force nnz and maxabs.
 * ------------------------------------------------------------------------------------- */
#define ORC_LANES 256

int orc_block_stats(int dtype, uint64_t n, const void* base, const void* expert, float* norm,
                    float* maxabs, uint32_t* nnz, double* ss_f64) {
  if ((dtype != ORC_BF16 && dtype != ORC_F32) || (n > 0 && (!base || !expert))) return ORC_EINVAL;
  const uint64_t V = dtype == ORC_BF16 ? 8 : 4;
  const uint64_t nvec = (n + V - 1) / V;

  float mx = 0.0f;
  uint32_t cnt = 0;
  double ss64 = 0.0;
  for (uint64_t k = 0; k < n; ++k) {
    float d = load_elem(dtype, expert, k) - load_elem(dtype, base, k);
    if (!is_finite_f(d)) return ORC_ENONFINITE;
    float a = fabsf(d);
    if (a > mx) mx = a;
    if (d != 0.0f) ++cnt;
    ss64 += (double)d * (double)d;
  }

  float p[ORC_LANES];
  for (int l = 0; l < ORC_LANES; ++l) {
    float acc = 0.0f;
    for (uint64_t v = (uint64_t)l; v < nvec; v += ORC_LANES) {
      for (uint64_t e = 0; e < V; ++e) {
        uint64_t k = v * V + e;
        float d = k < n ? load_elem(dtype, expert, k) - load_elem(dtype, base, k) : 0.0f;
        acc = fmaf(d, d, acc);
      }
    }
    p[l] = acc;
  }
  float q[ORC_LANES];
  for (int s = 16; s >= 1; s >>= 1) {
    for (int l = 0; l < ORC_LANES; ++l) q[l] = p[l] + p[l ^ s];
    memcpy(p, q, sizeof(p));
  }
  float g[8], h[8];
  for (int w = 0; w < 8; ++w) g[w] = p[32 * w];
  for (int s = 4; s >= 1; s >>= 1) {
    for (int w = 0; w < 8; ++w) h[w] = g[w] + g[w ^ s];
    memcpy(g, h, sizeof(g));
  }
  if (norm) *norm = sqrtf(g[0]);
  if (maxabs) *maxabs = mx;
  if (nnz) *nnz = cnt;
  if (ss_f64) *ss_f64 = ss64;
  return ORC_OK;
}

static const void* elem_ptr(int dtype, const void* p, uint64_t off) {
  return (const char*)p + off * (dtype == ORC_BF16 ? 2u : 4u);
}

/* statistics of every unit (i, b); arrays are expert-major [K][n_blocks] */
int orc_index(const orc_family* f, float* norm, float* maxabs, uint32_t* nnz) {
  if (!f || f->K == 0) return ORC_EINVAL;
  for (uint32_t i = 0; i < f->K; ++i) {
    for (uint64_t b = 0; b < f->n_blocks; ++b) {
      uint64_t u = (uint64_t)i * f->n_blocks + b;
      int rc = orc_block_stats(f->dtype, f->blk_len[b], elem_ptr(f->dtype, f->base, f->blk_off[b]),
                               elem_ptr(f->dtype, f->experts[i], f->blk_off[b]), &norm[u], &maxabs[u],
                               &nnz[u], NULL);
      if (rc != ORC_OK) return rc;
    }
  }
  return ORC_OK;
}

/* ---------------------------------------------------------------------------------------
 * TIES trim threshold (App. A.1: TIES trims, elects signs and averages sign-consistent
 * entries).  Reading: for each expert i and trim group (one tensor, or the whole
 * checkpoint), k = floor(rho * numel) computed in double, and tau is the k-th largest
 * magnitude key with multiplicity (ties at tau are all kept); k = 0 keeps nothing.  The
 * threshold comes from the full delta (an operator parameter theta, recorded with the
 * plan), so Psi stays non-anticipatory and equals standard TIES at A = 1.
 * Pins: a full sort of the keys on random tensors; hand-computed examples; a non-finite
 * delta is refused.
 * ------------------------------------------------------------------------------------- */
int orc_key_hist(int dtype, uint64_t n, const void* base, const void* expert, uint64_t* hist) {
  if (!hist || (n > 0 && (!base || !expert))) return ORC_EINVAL;
  for (uint64_t k = 0; k < n; ++k) {
    float d = load_elem(dtype, expert, k) - load_elem(dtype, base, k);
    if (!is_finite_f(d)) return ORC_ENONFINITE;
    hist[orc_ties_key(d)] += 1;
  }
  return ORC_OK;
}

uint32_t orc_tau_from_hist(const uint64_t* hist, uint64_t numel, float density) {
  uint64_t k = (uint64_t)floor((double)density * (double)numel);
  if (k == 0) return ORC_TAU_NONE;
  uint64_t cum = 0;
  for (int key = 0x7FFF; key >= 0; --key) {
    cum += hist[key];
    if (cum >= k) return (uint32_t)key;
  }
  return 0; /* k > numel cannot happen for rho <= 1 */
}

/* tau is expert-major [K][n_groups] */
int orc_ties_thresholds(const orc_family* f, float density, uint32_t* tau) {
  if (!f || !tau || f->n_groups == 0) return ORC_EINVAL;
  uint64_t* hist = (uint64_t*)calloc((size_t)f->n_groups * 32768u, sizeof(uint64_t));
  uint64_t* numel = (uint64_t*)calloc(f->n_groups, sizeof(uint64_t));
  if (!hist || !numel) {
    free(hist);
    free(numel);
    return ORC_EOOM;
  }
  for (uint64_t b = 0; b < f->n_blocks; ++b) numel[f->blk_group[b]] += f->blk_len[b];
  int rc = ORC_OK;
  for (uint32_t i = 0; i < f->K && rc == ORC_OK; ++i) {
    memset(hist, 0, (size_t)f->n_groups * 32768u * sizeof(uint64_t));
    for (uint64_t b = 0; b < f->n_blocks && rc == ORC_OK; ++b)
      rc = orc_key_hist(f->dtype, f->blk_len[b], elem_ptr(f->dtype, f->base, f->blk_off[b]),
                        elem_ptr(f->dtype, f->experts[i], f->blk_off[b]),
                        hist + (size_t)f->blk_group[b] * 32768u);
    for (uint32_t g = 0; g < f->n_groups && rc == ORC_OK; ++g)
      tau[(size_t)i * f->n_groups + g] = orc_tau_from_hist(hist + (size_t)g * 32768u, numel[g], density);
  }
  free(hist);
  free(numel);
  return rc;
}

/* TIES after masking (App. A.1: TIES trims, elects signs and averages sign-consistent
 * entries after masking).  Reading: the trim threshold of each (expert, group) is that of
 * the zero-completed masked deltas A_i Delta_i: the k-th largest key, k = floor(density *
 * numel_group), over the entries of the selected blocks together with a zero (key 0) for
 * every entry of an unselected block.  With every block selected it is orc_ties_thresholds.
 * mask: the access mask, one word per block (bit i = expert i). */
int orc_ties_masked_thresholds(const orc_family* f, float density, const uint32_t* mask, uint32_t* tau) {
  if (!f || !tau || !mask || f->n_groups == 0) return ORC_EINVAL;
  uint64_t* hist = (uint64_t*)calloc((size_t)f->n_groups * 32768u, sizeof(uint64_t));
  uint64_t* numel = (uint64_t*)calloc(f->n_groups, sizeof(uint64_t));
  if (!hist || !numel) {
    free(hist);
    free(numel);
    return ORC_EOOM;
  }
  for (uint64_t b = 0; b < f->n_blocks; ++b) numel[f->blk_group[b]] += f->blk_len[b];
  int rc = ORC_OK;
  for (uint32_t i = 0; i < f->K && rc == ORC_OK; ++i) {
    memset(hist, 0, (size_t)f->n_groups * 32768u * sizeof(uint64_t));
    for (uint64_t b = 0; b < f->n_blocks && rc == ORC_OK; ++b) {
      uint64_t* h = hist + (size_t)f->blk_group[b] * 32768u;
      if ((mask[b] >> i) & 1u)
        rc = orc_key_hist(f->dtype, f->blk_len[b], elem_ptr(f->dtype, f->base, f->blk_off[b]),
                          elem_ptr(f->dtype, f->experts[i], f->blk_off[b]), h);
      else
        h[0] += f->blk_len[b]; /* omitted: zero entries, key 0, never read */
    }
    for (uint32_t g = 0; g < f->n_groups && rc == ORC_OK; ++g)
      tau[(size_t)i * f->n_groups + g] = orc_tau_from_hist(hist + (size_t)g * 32768u, numel[g], density);
  }
  free(hist);
  free(numel);
  return rc;
}

/* ---------------------------------------------------------------------------------------
 * Hashes.  FNV-1a 64 (Fowler, Noll, Vo): offset basis 14695981039346656037, prime
 * 1099511628211.  SplitMix64 output function (Steele, Lea, Flood, OOPSLA 2014).
 * Pins: the published FNV-1a test vectors; the SplitMix64 first output from state 0.
 * ------------------------------------------------------------------------------------- */
uint64_t orc_fnv1a64(const uint8_t* data, size_t n) {
  uint64_t h = 14695981039346656037ULL;
  for (size_t k = 0; k < n; ++k) {
    h ^= data[k];
    h *= 1099511628211ULL;
  }
  return h;
}

uint64_t orc_splitmix64(uint64_t state) {
  uint64_t z = state + 0x9E3779B97F4A7C15ULL;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

/* ---------------------------------------------------------------------------------------
 * Block content hash (Sec. 3 "Catalog": the catalog stores hashes of every block; Alg. 2
 * validates hashes before the manifest is built).  The paper names no function.  Reading:
 * the block's L bytes, zero-padded to a multiple of 16, are vectors q = 0, 1, ... of two
 * little-endian 64-bit words (lo_q, hi_q); with k_q = SplitMix64(q), a_q = k_q | 1 and
 * b_q = rotl(k_q, 32) | 1,
 *     H = sum_q (lo_q * a_q + hi_q * b_q)  mod 2^64,      hash = SplitMix64(H xor L).
 * q counts from the block's start, so equal blocks hash equal wherever they sit.  A
 * multilinear sum with odd keys: any change of a single word changes H (odd keys are units
 * mod 2^64), and the sum can be formed in any order.  It detects changed or corrupted
 * blocks; it is not a cryptographic hash.
 * Pins: every single-word change is detected (including a change by 2^63); swapping two
 * different vectors or the two words of a vector changes the hash; H is additive over
 * blocks with disjoint support; the length is part of the hash; the GPU catalog matches.
 * ------------------------------------------------------------------------------------- */
static uint64_t rd_le64(const uint8_t* p) {
  uint64_t v = 0;
  for (int k = 7; k >= 0; --k) v = (v << 8) | p[k];
  return v;
}

uint64_t orc_block_hash_sum(const void* bytes, uint64_t len) {
  const uint8_t* src = (const uint8_t*)bytes;
  uint64_t H = 0;
  for (uint64_t q = 0; q * 16 < len; ++q) {
    uint8_t v[16] = {0};
    const uint64_t m = len - q * 16 < 16 ? len - q * 16 : 16;
    memcpy(v, src + q * 16, (size_t)m);
    const uint64_t k = orc_splitmix64(q);
    const uint64_t a = k | 1u, b = ((k << 32) | (k >> 32)) | 1u;
    H += rd_le64(v) * a + rd_le64(v + 8) * b;
  }
  return H;
}

uint64_t orc_block_hash(const void* bytes, uint64_t len) { return orc_splitmix64(orc_block_hash_sum(bytes, len) ^ len); }

/* the catalog's hashes of a family: base_hash[b], expert_hash[i * n_blocks + b] */
int orc_index_hashes(const orc_family* f, uint64_t* base_hash, uint64_t* expert_hash) {
  if (!f || !base_hash || !expert_hash) return ORC_EINVAL;
  const uint64_t es = f->dtype == ORC_BF16 ? 2u : 4u;
  for (uint64_t b = 0; b < f->n_blocks; ++b) {
    const uint64_t len = (uint64_t)f->blk_len[b] * es;
    base_hash[b] = orc_block_hash(elem_ptr(f->dtype, f->base, f->blk_off[b]), len);
    for (uint32_t i = 0; i < f->K; ++i)
      expert_hash[(uint64_t)i * f->n_blocks + b] = orc_block_hash(elem_ptr(f->dtype, f->experts[i], f->blk_off[b]), len);
  }
  return ORC_OK;
}

/* ---------------------------------------------------------------------------------------
 * Alg. 1 PlanGen (Sec. 3), cost model Eq. 3 and App. A.1.
 *  - Candidates Q: units (i, b) whose delta can change the output.  Reading: a unit
 *    with nnz = 0 contributes exactly nothing to any operator, and under TIES a unit
 *    whose largest key is below tau is trimmed entirely; both are left out (exact).
 *  - Score s(i,t,b) = |coef_i| * ||Delta_{i,t,b}||_2 in fp32 (the utility u of Prop. 2);
 *    coef_i = alpha_i (AVG, TA, DARE, renormalised AVG) or lambda (TIES, DARE-TIES).  In the
 *    score-per-byte mode (the
 *    second heuristic Sec. 3 names for the objective of Eq. 6) s is divided by the unit's
 *    byte cost c, one fp32 division.
 *  - Sort by decreasing score; ties by ascending unit id = b*K + i (block order is
 *    tensor/block order, then expert).  The key is unique, so the order is total.
 *  - Greedy fill: take a candidate if C_hat + c <= B, otherwise skip it and go on.
 *    c_{i,t,b} = elements(b) * bytes per element (App. A.1: stored byte length).
 *  - Record: mask (bit i of word b = A_{i,t,b}), C_hat, number selected, the selected-
 *    block digest and the traversal order.  Reading of the digest: FNV-1a 64 over the
 *     little-endian bytes of (kind, K, alpha[0..K-1] bits, lambda bits, density bits,
 *     trim_scope, drop_p bits, seed, score_mode, B, C_hat, n_sel, set_hash), where set_hash is the
 *     wrapping sum over selected units u of splitmix64(u).
 *  - Tensor-level fallback (Sec. 3 Planner: deterministic fallback when block metadata
 *    are missing; Alg. 1's scoring step names fallback metadata).  Reading: an entry
 *    (i, b) whose nnz is ORC_NNZ_MISSING has no block statistics.  Every (expert i,
 *    tensor t) holding such an entry is planned as ONE unit at tensor granularity: it is
 *    always a candidate (nothing rules it out), its id is the unit of the tensor's first
 *    block b0(t)*K + i, its cost is the whole tensor's bytes, and its score is
 *    |coef_i| * sqrt(ss) with ss the fp32 chain ss = fma(n_b, n_b, ss) over the known
 *    blocks of t in ascending order from 0 (the norm of the part of Delta_{i,t} the
 *    catalog knows; 0 if none), divided by the tensor's bytes (converted to fp32) in the
 *    score-per-byte mode.  The tensor's other units are not candidates.  Taking it sets
 *    bit i on every block of t; it counts once in n_sel and set_hash.
 * Pins: brute force over all subsets on tiny inputs; the cardinality-knapsack optimum
 * when all costs are equal; Prop. 1 (C_hat <= B); full budget selects every candidate;
 * the order depends on |coef| only; relabelling experts or reordering blocks relabels the
 * plan; TIES candidates per trim group against keys computed from the data; for the
 * fallback, hand-worked catalogs (equal and unequal signed coefficients) and the
 * known-part norm against the deltas.
 * ------------------------------------------------------------------------------------- */
typedef struct {
  float score;
  uint32_t unit;
  uint64_t cost;
} orc_cand;

static int cand_cmp(const void* a, const void* b) {
  const orc_cand* x = (const orc_cand*)a;
  const orc_cand* y = (const orc_cand*)b;
  if (x->score > y->score) return -1;
  if (x->score < y->score) return 1;
  return x->unit < y->unit ? -1 : (x->unit > y->unit ? 1 : 0);
}

static size_t put_u32(uint8_t* p, uint32_t v) {
  for (int k = 0; k < 4; ++k) p[k] = (uint8_t)(v >> (8 * k));
  return 4;
}
static size_t put_u64(uint8_t* p, uint64_t v) {
  for (int k = 0; k < 8; ++k) p[k] = (uint8_t)(v >> (8 * k));
  return 8;
}

int orc_plan(uint32_t K, uint64_t n_blocks, const uint32_t* blk_len, const uint32_t* blk_group,
             uint32_t n_groups, uint32_t elem_size, const orc_op* op, const float* norm,
             const float* maxabs, const uint32_t* nnz, const uint32_t* tau, uint64_t budget,
             uint32_t* mask, uint64_t* chat_out, uint64_t* n_sel_out, uint64_t* n_cand_out,
             uint64_t* set_hash_out, uint64_t* digest_out, uint32_t* order, const uint32_t* blk_tensor,
             uint32_t n_tensors) {
  if (!op || K == 0 || K > 32 || op->K != K || !norm || !maxabs || !nnz || !mask) return ORC_EINVAL;
  if (op->kind == ORC_TIES && (!tau || !blk_group)) return ORC_EINVAL;
  if (op->kind != ORC_TIES && op->kind != ORC_DARE_TIES && op->kind != ORC_TIES_MASKED && !op->alpha)
    return ORC_EINVAL;
  if (n_blocks * K > 0xFFFFFFFFull) return ORC_EINVAL;
  if (blk_tensor) /* tensors in checkpoint order: the blocks of a tensor are contiguous */
    for (uint64_t b = 0; b < n_blocks; ++b)
      if (blk_tensor[b] >= n_tensors || (b > 0 && blk_tensor[b] < blk_tensor[b - 1])) return ORC_EINVAL;

  /* fallback pairs (i, t): some entry of tensor t has no statistics for expert i */
  uint8_t* fb = NULL;
  if (blk_tensor) {
    fb = (uint8_t*)calloc((size_t)K * n_tensors + 1, 1);
    if (!fb) return ORC_EOOM;
  }
  for (uint32_t i = 0; i < K; ++i)
    for (uint64_t b = 0; b < n_blocks; ++b)
      if (nnz[(uint64_t)i * n_blocks + b] == ORC_NNZ_MISSING) {
        if (!fb) return ORC_EINVAL; /* missing statistics need the tensor map */
        fb[(size_t)i * n_tensors + blk_tensor[b]] = 1;
      }

  orc_cand* q = (orc_cand*)malloc(sizeof(orc_cand) * (size_t)(n_blocks * K + 1));
  if (!q) {
    free(fb);
    return ORC_EOOM;
  }
  uint64_t nq = 0;
  for (uint64_t b = 0; b < n_blocks; ++b) {
    for (uint32_t i = 0; i < K; ++i) {
      uint64_t s = (uint64_t)i * n_blocks + b;
      float coef = (op->kind == ORC_TIES || op->kind == ORC_DARE_TIES || op->kind == ORC_TIES_MASKED) ? op->lambda
                                                                                                    : op->alpha[i];
      if (fb && fb[(size_t)i * n_tensors + blk_tensor[b]]) {
        const uint32_t t = blk_tensor[b];
        if (b > 0 && blk_tensor[b - 1] == t) continue; /* only the tensor's first block */
        float ss = 0.0f;
        uint64_t cost = 0;
        for (uint64_t b2 = b; b2 < n_blocks && blk_tensor[b2] == t; ++b2) {
          const uint64_t s2 = (uint64_t)i * n_blocks + b2;
          cost += (uint64_t)blk_len[b2] * elem_size;
          if (nnz[s2] != ORC_NNZ_MISSING) ss = fmaf(norm[s2], norm[s2], ss);
        }
        q[nq].score = fabsf(coef) * sqrtf(ss);
        q[nq].unit = (uint32_t)(b * K + i);
        q[nq].cost = cost;
        if (op->score_mode) q[nq].score = q[nq].score / (float)cost;
        ++nq;
        continue;
      }
      if (nnz[s] == 0) continue;
      if (op->kind == ORC_TIES && orc_ties_key(maxabs[s]) < tau[(size_t)i * n_groups + blk_group[b]])
        continue;
      q[nq].score = fabsf(coef) * norm[s];
      q[nq].unit = (uint32_t)(b * K + i);
      q[nq].cost = (uint64_t)blk_len[b] * elem_size;
      if (op->score_mode) q[nq].score = q[nq].score / (float)q[nq].cost;
      ++nq;
    }
  }
  qsort(q, (size_t)nq, sizeof(orc_cand), cand_cmp);

  memset(mask, 0, sizeof(uint32_t) * (size_t)n_blocks);
  uint64_t chat = 0, nsel = 0, set_hash = 0;
  for (uint64_t r = 0; r < nq; ++r) {
    if (chat + q[r].cost <= budget) {
      const uint64_t b = q[r].unit / K;
      const uint32_t i = q[r].unit % K;
      chat += q[r].cost;
      if (fb && fb[(size_t)i * n_tensors + blk_tensor[b]]) {
        for (uint64_t b2 = b; b2 < n_blocks && blk_tensor[b2] == blk_tensor[b]; ++b2) mask[b2] |= 1u << i;
      } else {
        mask[b] |= 1u << i;
      }
      set_hash += orc_splitmix64(q[r].unit);
      ++nsel;
    }
    if (order) order[r] = q[r].unit;
  }
  free(q);
  free(fb);

  uint8_t hdr[4 + 4 + 4 * 32 + 4 + 4 + 4 + 8 + 8 + 4 + 8 + 8 + 8 + 8];
  size_t o = 0;
  o += put_u32(hdr + o, (uint32_t)op->kind);
  o += put_u32(hdr + o, K);
  for (uint32_t i = 0; i < K; ++i) o += put_u32(hdr + o, op->alpha ? f2u(op->alpha[i]) : 0u);
  o += put_u32(hdr + o, f2u(op->lambda));
  o += put_u32(hdr + o, f2u(op->density));
  o += put_u32(hdr + o, op->trim_scope);
  uint64_t pbits;
  memcpy(&pbits, &op->drop_p, 8);
  o += put_u64(hdr + o, pbits);
  o += put_u64(hdr + o, op->seed);
  o += put_u32(hdr + o, op->score_mode);
  o += put_u64(hdr + o, budget);
  o += put_u64(hdr + o, chat);
  o += put_u64(hdr + o, nsel);
  o += put_u64(hdr + o, set_hash);

  if (chat_out) *chat_out = chat;
  if (n_sel_out) *n_sel_out = nsel;
  if (n_cand_out) *n_cand_out = nq;
  if (set_hash_out) *set_hash_out = set_hash;
  if (digest_out) *digest_out = orc_fnv1a64(hdr, o);
  return ORC_OK;
}

/* ---------------------------------------------------------------------------------------
 * Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel random numbers: as easy as 1, 2,
 * 3", SC 2011): ten rounds of two 32x32->64 multiplies with multipliers 0xD2511F53 and
 * 0xCD9E8D57, the key bumped by the Weyl constants 0x9E3779B9 and 0xBB67AE85 between
 * rounds.  Pins: cuRAND's Philox4_32_10 (an independent implementation), its host
 * generator on the CPU and its device generator on the GPU.
 * ------------------------------------------------------------------------------------- */
void orc_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]) {
  uint32_t c0 = ctr[0], c1 = ctr[1], c2 = ctr[2], c3 = ctr[3];
  uint32_t k0 = key[0], k1 = key[1];
  for (int r = 0; r < 10; ++r) {
    if (r > 0) {
      k0 += 0x9E3779B9u;
      k1 += 0xBB67AE85u;
    }
    uint64_t p0 = (uint64_t)0xD2511F53u * c0;
    uint64_t p1 = (uint64_t)0xCD9E8D57u * c2;
    uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
    uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
    uint32_t n0 = hi1 ^ c1 ^ k0;
    uint32_t n2 = hi0 ^ c3 ^ k1;
    c0 = n0;
    c1 = lo1;
    c2 = n2;
    c3 = lo0;
  }
  out[0] = c0;
  out[1] = c1;
  out[2] = c2;
  out[3] = c3;
}

/* DARE keep decision for expert i, flat element j (App. A.1: random drop and rescale with a
   fixed seed omega).  Reading: one Philox call per 8 consecutive elements, counter
   (j/8 low, j/8 high, i, 0x44415245), key (seed low, seed high); element j takes the
   16-bit word number j mod 8 of the output (word e is bits 16*(e%2).. of output e/2);
   keep iff that word >= T = floor(p * 65536). */
static uint32_t dare_threshold(double p) {
  double t = floor(p * 65536.0);
  if (!(t > 0.0)) return 0u;
  if (t > 65536.0) return 65536u;
  return (uint32_t)t;
}

int orc_dare_keep(uint64_t seed, uint32_t expert, uint64_t j, double p) {
  uint64_t g = j >> 3;
  uint32_t ctr[4] = {(uint32_t)g, (uint32_t)(g >> 32), expert, 0x44415245u};
  uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
  uint32_t w[4];
  orc_philox4x32_10(ctr, key, w);
  uint32_t e = (uint32_t)(j & 7u);
  uint32_t r = (w[e >> 1] >> (16u * (e & 1u))) & 0xFFFFu;
  return r >= dare_threshold(p);
}

/* ---------------------------------------------------------------------------------------
 * Budgeted operator Psi_op on one block (Eq. 4, App. A.1), with the mask's omitted
 * experts contributing exactly zero and never read (non-anticipatory, Sec. 2).  Order of
 * fp32 operations (reading; the paper fixes none): experts in ascending index.
 *  AVG / TA (zero-completed tuple):  acc = sum_i fma(alpha_i, A_i delta_i, acc);
 *                                    out = round(M_0 + acc)
 *  DARE: v_i = delta_i * sigma for a kept entry, sigma = fp32(1/(1-p)); a dropped entry is
 *        omitted from the sum, as an unselected one is (its zero is never added);
 *        acc = sum over the kept selected i of fma(alpha_i, v_i, acc); out = round(M_0 + acc)
 *  TIES: d^_i = A_i delta_i if key(delta_i) >= tau_i else 0;  P = sum of the d^_i > 0,
 *        N = sum of the d^_i < 0 (each an ascending fp32 chain from +0), c+ and c- their
 *        counts;  gamma = sign(P + N), taken exactly as P > -N, P < -N or P = -N (the
 *        rounded sum fl(P + N) has the sign of P + N);  m = P / c+ if gamma > 0, N / c- if
 *        gamma < 0, else 0;  out = round(fma(lambda, m, M_0))
 *  AVG, renormalised over the selected experts (App. A.1, the selected-only variant with
 *        coefficients beta_i(A) = 0 when A_i = 0): s = sum of alpha_j over the experts j that
 *        are selected or whose delta block is exactly zero (ascending fp32 adds from +0);
 *        beta_i = alpha_i / s;
 *        acc = sum_i fma(beta_i, A_i delta_i, acc); out = round(M_0 + acc)
 *  TIES after masking: as TIES, with tau the threshold of the masked deltas
 *        (orc_ties_masked_thresholds)
 *  DARE-TIES: DARE's drop and rescale with the same mask omega, then TIES's election and
 *        disjoint mean without magnitude trimming: d^_i = A_i (keep_i ? delta_i * sigma : 0),
 *        then P, N, gamma, m and out as TIES
 * round = bf16 round-to-nearest-even, or none for fp32 checkpoints.
 * Pins: hand-computed TIES, AVG and renormalised-AVG examples (an omitted expert counts as
 * zero whatever its data); Eq. 5 against an fp64 restatement of the unmasked operator
 * (within one bf16 ulp); per-tensor TIES trims are separable; Prop. 2 bound and the
 * coefficient-drift bound of App. A.1; the renormalised AVG through the full-budget plan
 * equals AVG; DARE at p = 0 equals AVG (also over 2^21 entries), drops are independent
 * across blocks and the DARE mean over seeds tends to AVG; DARE-TIES at p = 0 equals TIES
 * at density 1.
 * ------------------------------------------------------------------------------------- */
int orc_merge_block(int dtype, uint64_t n, uint64_t j0, const void* base, const void* const* experts,
                    uint32_t mask, uint32_t known_zero, const orc_op* op, const uint32_t* tau_k, void* out) {
  if (!op || op->K == 0 || op->K > 32 || (n > 0 && (!base || !out))) return ORC_EINVAL;
  const uint32_t K = op->K;
  for (uint32_t i = 0; i < K; ++i)
    if (((mask >> i) & 1u) && !experts[i]) return ORC_EINVAL;
  const int ties_like = op->kind == ORC_TIES || op->kind == ORC_DARE_TIES || op->kind == ORC_TIES_MASKED;
  const int trims = op->kind == ORC_TIES || op->kind == ORC_TIES_MASKED;
  if (trims && !tau_k) return ORC_EINVAL;
  if (!ties_like && !op->alpha) return ORC_EINVAL;
  float sigma = op->drop_p < 1.0 ? (float)(1.0 / (1.0 - op->drop_p)) : 0.0f;
  /* renormalised AVG: the sum, ascending, of the coefficients of the experts that take part:
     the selected ones and those whose delta block is exactly zero (known from the catalog
     without a read; counting them is what makes the full budget equal the full-read
     average, Eq. 5) */
  float s_sel = 0.0f;
  if (op->kind == ORC_AVG_RENORM) {
    for (uint32_t i = 0; i < K; ++i)
      if (((mask | known_zero) >> i) & 1u) {
        if (!(op->alpha[i] > 0.0f)) return ORC_EINVAL;
        s_sel = s_sel + op->alpha[i];
      }
  }

  for (uint64_t k = 0; k < n; ++k) {
    float x0 = load_elem(dtype, base, k);
    float res;
    if (ties_like) {
      float P = 0.0f, Nn = 0.0f;
      uint32_t cp = 0, cn = 0;
      for (uint32_t i = 0; i < K; ++i) {
        float dh = 0.0f;
        if ((mask >> i) & 1u) {
          float d = load_elem(dtype, experts[i], k) - x0;
          if (trims) {
            if (orc_ties_key(d) >= tau_k[i]) dh = d;
          } else if (orc_dare_keep(op->seed, i, j0 + k, op->drop_p)) {
            dh = d * sigma;
          }
        }
        if (dh > 0.0f) {
          P = P + dh;
          ++cp;
        } else if (dh < 0.0f) {
          Nn = Nn + dh;
          ++cn;
        }
      }
      float m = 0.0f;
      if (P > -Nn) m = P / (float)cp;
      else if (P < -Nn) m = Nn / (float)cn;
      res = fmaf(op->lambda, m, x0);
    } else {
      float acc = 0.0f;
      for (uint32_t i = 0; i < K; ++i) {
        if (!((mask >> i) & 1u)) continue; /* omitted: zero entry, never read */
        float d = load_elem(dtype, experts[i], k) - x0;
        if (op->kind == ORC_DARE) {
          if (!orc_dare_keep(op->seed, i, j0 + k, op->drop_p)) continue; /* dropped: omitted */
          d = d * sigma;
        }
        const float coef = op->kind == ORC_AVG_RENORM ? op->alpha[i] / s_sel : op->alpha[i];
        acc = fmaf(coef, d, acc);
      }
      res = x0 + acc;
    }
    store_elem(dtype, out, k, res);
  }
  return ORC_OK;
}

/* Alg. 2 ExecuteMerge: tensors in order, blocks in order, every block materialised
   (untouched blocks are copies of the base; the paper's comparisons use full logical
   checkpoint materialisation).  mask may be NULL for the full read A = 1 (Eq. 1).
   nnz: the catalog's nonzero counts [K][n_blocks], which tell the renormalised AVG which
   deltas are known to be zero; NULL derives them from the data (the full catalog).  An
   entry of ORC_NNZ_MISSING is not known to be zero. */
int orc_merge(const orc_family* f, const orc_op* op, const uint32_t* tau, const uint32_t* mask,
              void* out, const uint32_t* nnz) {
  if (!f || !op || !out || op->K != f->K || f->K == 0 || f->K > 32) return ORC_EINVAL;
  const uint32_t all = f->K == 32 ? 0xFFFFFFFFu : ((1u << f->K) - 1u);
  uint32_t tau_k[32];
  const void* ex[32];
  for (uint64_t b = 0; b < f->n_blocks; ++b) {
    uint64_t off = f->blk_off[b];
    for (uint32_t i = 0; i < f->K; ++i) {
      ex[i] = elem_ptr(f->dtype, f->experts[i], off);
      if (op->kind == ORC_TIES || op->kind == ORC_TIES_MASKED) tau_k[i] = tau[(size_t)i * f->n_groups + f->blk_group[b]];
    }
    uint32_t known_zero = 0;
    if (op->kind == ORC_AVG_RENORM && nnz) {
      for (uint32_t i = 0; i < f->K; ++i)
        if (nnz[(size_t)i * f->n_blocks + b] == 0) known_zero |= 1u << i;
    } else if (op->kind == ORC_AVG_RENORM) {
      const void* b0 = elem_ptr(f->dtype, f->base, off);
      for (uint32_t i = 0; i < f->K; ++i) {
        uint64_t k = 0;
        while (k < f->blk_len[b] && load_elem(f->dtype, ex[i], k) - load_elem(f->dtype, b0, k) == 0.0f) ++k;
        if (k == f->blk_len[b]) known_zero |= 1u << i;
      }
    }
    int rc = orc_merge_block(f->dtype, f->blk_len[b], off, elem_ptr(f->dtype, f->base, off), ex,
                             mask ? mask[b] : all, known_zero, op, tau_k,
                             (char*)out + off * (f->dtype == ORC_BF16 ? 2u : 4u));
    if (rc != ORC_OK) return rc;
  }
  return ORC_OK;
}
