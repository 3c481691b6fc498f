/*
 * CPU oracle for the budgeted, mask-aware merge (MergePipe, "Access Sets
 * Matter: Budgeting Expert Reads for Scalable Weight-Space Model Merging").
 *
 * TEST INFRASTRUCTURE ONLY.  This is a plain, slow, single-threaded C
 * restatement of what the method computes, used to check the CUDA path.
 * Only the test suite, the package's smoke check and the benchmark's CPU
 * baseline may load it; the product path never calls it.  It shares no code,
 * header or table with the CUDA path.
 *
 * Every function cites the passage of the paper it follows.  Where the paper
 * leaves a choice open (block layout, rounding order, TIES trim population,
 * DARE generator, tie-breaks, digest), the reading used is stated beside the
 * function and is the same one the CUDA path implements.
 */
#ifndef MP_ORACLE_H
#define MP_ORACLE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum { ORC_BF16 = 0, ORC_F32 = 1 };
enum { ORC_AVG = 0, ORC_TA = 1, ORC_TIES = 2, ORC_DARE = 3, ORC_AVG_RENORM = 4, ORC_DARE_TIES = 5, ORC_TIES_MASKED = 6 };
enum { ORC_OK = 0, ORC_EINVAL = -1, ORC_EOOM = -3, ORC_ENONFINITE = -4 };
#define ORC_TAU_NONE 0x8000u /* TIES threshold when k = 0: no 15-bit key reaches it */
#define ORC_NNZ_MISSING 0xFFFFFFFFu /* catalog entry without block statistics (tensor-level fallback) */

/* merge operator and its parameters theta (Alg. 1 records op and theta) */
typedef struct {
  int kind;            /* ORC_AVG / ORC_TA / ORC_TIES / ORC_DARE / ORC_AVG_RENORM / ORC_DARE_TIES / ORC_TIES_MASKED */
  uint32_t K;          /* number of experts */
  const float* alpha;  /* K coefficients (AVG, TA, DARE); may be NULL for TIES */
  float lambda;        /* TIES: scale of the merged task vector */
  float density;       /* TIES: fraction rho of each trim population kept */
  uint32_t trim_scope; /* TIES: 0 = per (expert, tensor), 1 = per expert */
  double drop_p;       /* DARE: drop probability p */
  uint64_t seed;       /* DARE: seed of the fixed random mask omega */
  uint32_t score_mode; /* planning score: 0 = |coef_i| * norm; 1 = that per byte of the block */
} orc_op;

/* block geometry plus data: blocks are disjoint spans of the flat checkpoints (Sec. 2) */
typedef struct {
  int dtype;                  /* ORC_BF16 (uint16 bit patterns) or ORC_F32 */
  uint32_t K;
  uint64_t n_blocks;
  const uint64_t* blk_off;    /* element offset of each block */
  const uint32_t* blk_len;    /* elements in each block */
  const uint32_t* blk_group;  /* TIES trim group of each block */
  uint32_t n_groups;
  const void* base;           /* M_0, flat */
  const void* const* experts; /* M_1..M_K, flat */
} orc_family;

/* element conversion (bf16 round to nearest even, written from the IEEE definition) */
float orc_bf16_to_f32(uint16_t h);
uint16_t orc_f32_to_bf16(float f);
uint32_t orc_ties_key(float delta);

/* statistics of one expert block: norm (canonical fp32 order), max |delta|, nonzero count,
   and the fp64 sum of squares for checks */
int orc_block_stats(int dtype, uint64_t n, const void* base, const void* expert, float* norm,
                    float* maxabs, uint32_t* nnz, double* ss_f64);
int orc_index(const orc_family* f, float* norm, float* maxabs, uint32_t* nnz);

/* TIES trim thresholds */
int orc_key_hist(int dtype, uint64_t n, const void* base, const void* expert, uint64_t* hist32768);
uint32_t orc_tau_from_hist(const uint64_t* hist32768, uint64_t numel, float density);
int orc_ties_thresholds(const orc_family* f, float density, uint32_t* tau);
/* thresholds of the zero-completed masked deltas (TIES after masking) */
int orc_ties_masked_thresholds(const orc_family* f, float density, const uint32_t* mask, uint32_t* tau);

/* Alg. 1 PlanGen */
int orc_plan(uint32_t K, uint64_t n_blocks, const uint32_t* blk_len, const uint32_t* blk_group,
             uint32_t n_groups, uint32_t elem_size, const orc_op* op, const float* norm,
             const float* maxabs, const uint32_t* nnz, const uint32_t* tau, uint64_t budget,
             uint32_t* mask, uint64_t* chat, uint64_t* n_sel, uint64_t* n_cand, uint64_t* set_hash,
             uint64_t* digest, uint32_t* order, const uint32_t* blk_tensor, uint32_t n_tensors);

/* Eq. 4 budgeted merge of one block, and of a whole family (Alg. 2).  known_zero (used by
   the renormalised AVG only): bit i set when expert i's delta block is exactly zero, which
   the catalog records (nnz = 0) so that no read is needed to count that expert. */
int orc_merge_block(int dtype, uint64_t n, uint64_t j0, const void* base, const void* const* experts,
                    uint32_t mask, uint32_t known_zero, const orc_op* op, const uint32_t* tau_k, void* out);
int orc_merge(const orc_family* f, const orc_op* op, const uint32_t* tau, const uint32_t* mask,
              void* out, const uint32_t* nnz);

/* generators and hashes */
void orc_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]);
int orc_dare_keep(uint64_t seed, uint32_t expert, uint64_t j, double p);
uint64_t orc_fnv1a64(const uint8_t* data, size_t n);
uint64_t orc_splitmix64(uint64_t state);

/* block content hash (catalog hashes; Alg. 2 validation): the multilinear sum H and the hash */
uint64_t orc_block_hash_sum(const void* bytes, uint64_t len);
uint64_t orc_block_hash(const void* bytes, uint64_t len);
int orc_index_hashes(const orc_family* f, uint64_t* base_hash, uint64_t* expert_hash);

#ifdef __cplusplus
}
#endif
#endif
