/*
 * mergepipe.h — C ABI of the GB300 budgeted, mask-aware merge.
 *
 * The method (MergePipe, "Access Sets Matter: Budgeting Expert Reads for
 * Scalable Weight-Space Model Merging") merges a base checkpoint M_0 with K
 * experts M_1..M_K that share its weight coordinates.  It runs in three calls:
 *
 *   mp_index_blocks  per-block statistics of every expert delta (the catalog
 *                    of Sec. 3; the Analyze reads of Sec. 2), plus the TIES
 *                    trim thresholds when the operator is TIES;
 *   mp_plan          a deterministic access plan under an expert-read budget
 *                    B (Alg. 1 PlanGen; Eq. 2, 3 and 6);
 *   mp_merge         the induced budgeted operator over only the planned
 *                    blocks (Eq. 4; Alg. 2 ExecuteMerge) and its manifest;
 *                    mp_merge_touched writes only the touched blocks and leaves
 *                    the rest as references to the base (WriteBlockOrReference).
 *
 * Conventions
 *  - Data pointers are device pointers unless stated (experts may also live in
 *    pinned host memory, see mp_family.experts_location).  The caller owns
 *    every data buffer; the library owns the opaque handles (release them with
 *    mp_free).  No torch or CUDA types appear in this header: a stream is the
 *    CUDA runtime's cudaStream_t passed as mp_stream (NULL = legacy default).
 *  - Every call enqueues its GPU work on the given stream and returns without
 *    waiting for it, except the accessors (mp_*_info, mp_index_stats), which
 *    wait for the handle's work to finish.  mp_index_blocks, mp_plan, mp_merge and
 *    mp_merge_touched enqueue kernels only (their small tables and results move
 *    through pinned memory that kernels read and write), so bulk transfers the
 *    caller runs on other streams do not hold them up; the exceptions use
 *    cudaMemcpyAsync: a block table above 8 MiB, the thresholds of TIES after
 *    masking, and the arrays that mp_index_import copies in.
 *  - CUDA graphs: for a family whose experts are in device memory, a step made of
 *    mp_index_blocks, mp_plan and mp_merge / mp_merge_touched calls can be captured
 *    on a stream (stream capture) and the graph replayed; each replay recomputes the
 *    catalog, the plans and the merges from the buffers' current contents into the
 *    handles made during the capture.  The accessors of those handles then wait for
 *    the whole device (a captured event cannot be waited for from the host).  Free
 *    such handles before the graph is destroyed.  Host-resident pools, TIES after
 *    masking and mp_index_import are not capturable.  Errors found by a kernel (a
 *    non-finite delta, a timed-out wait) are reported by the next accessor on
 *    that handle or on a handle derived from it.
 *  - Checked build: libmergepipe_checked.so exports the same entry points from the same
 *    sources compiled with MP_CHECKED.  Before a kernel streams a range of a checkpoint
 *    (a block of the catalog pass or of the host-pool gather, a chunk of the merge, a
 *    block of the hash pass) it checks the range against the block table, the call's block
 *    range, the buffers' extents, the 16-byte alignment of bulk copies and the number of
 *    experts, and the planner checks every compaction slot and unit id it writes; a
 *    range that fails is not touched, and the accessors of the call's handle
 *    return MP_ERR_CUDA with "a bounds check of the checked build failed".  mp_version()
 *    names the build.  Meant for debugging; its checks cost little (within 1 % of the
 *    default build on a Qwen2.5-0.5B-shaped task-arithmetic step).
 *  - On an error return no handle is produced and *out is set to NULL; the
 *    contents of a merge output buffer are then unspecified.
 *  - mp_last_error() returns a thread-local message for the last failure.
 */
#ifndef MERGEPIPE_H
#define MERGEPIPE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int32_t mp_status;
#define MP_OK 0
#define MP_ERR_INVALID_ARG (-1) /* a bad argument; nothing was enqueued */
#define MP_ERR_CUDA (-2)        /* a CUDA runtime call failed */
#define MP_ERR_OOM (-3)         /* device or host allocation failed */
#define MP_ERR_NONFINITE (-4)   /* a delta was NaN or infinite (reported by accessors) */
#define MP_ERR_BUDGET (-5)      /* realized reads exceeded the plan (Prop. 1 violated) */
#define MP_ERR_TIMEOUT (-6)     /* a bounded device wait gave up (reported by accessors) */
#define MP_ERR_UNSUPPORTED (-7) /* a valid request the library does not handle */
#define MP_ERR_MISMATCH (-8)    /* handles that do not belong together */

typedef struct CUstream_st* mp_stream;

/* nnz of a catalog entry that has no block statistics (mp_index_import); no block holds
   2^32 - 1 elements, so no count takes this value */
#define MP_NNZ_MISSING 0xFFFFFFFFu

typedef enum { MP_BF16 = 0, MP_F32 = 1 } mp_dtype;

/* Merge operators (Sec. 1, App. A.1).  AVG and TA are the fixed-coefficient additive
   operator sum_i alpha_i A_i Delta_i (Prop. 2); they differ only in how the caller
   chose alpha (AVG: sum alpha = 1; TA: alpha_i = lambda).  AVG_RENORM is App. A.1's
   selected-only average: per block, beta_i = alpha_i / (sum of alpha over the selected
   experts), 0 for an omitted expert (the coefficient-drift bound of App. A.1 applies, not
   Prop. 2); every alpha_i must be > 0.  DARE_TIES drops and rescales like DARE (same
   mask omega), then elects signs and takes the disjoint mean like TIES, without the
   magnitude trim (lambda, drop_p and seed are used; no tau).  TIES_MASKED is TIES applied
   after masking (App. A.1): its trim threshold is that of the zero-completed masked
   deltas A_i Delta_i (the k-th largest key, k = floor(density * numel) of the group, an
   omitted entry counting as a zero), so it depends on the plan; lambda, density and
   trim_scope are used.  With every block selected it is TIES. */
typedef enum {
  MP_OP_AVG = 0,
  MP_OP_TA = 1,
  MP_OP_TIES = 2,
  MP_OP_DARE = 3,
  MP_OP_AVG_RENORM = 4,
  MP_OP_DARE_TIES = 5,
  MP_OP_TIES_MASKED = 6
} mp_op_kind;

/* One tensor of the tensor set T (Sec. 2), as a span of the flat checkpoint buffers. */
typedef struct {
  uint64_t offset_elems; /* start, in elements, in every flat buffer; offset*elem_size % 16 == 0 */
  uint64_t numel;        /* elements; any value >= 1 */
} mp_tensor;

/* A checkpoint family: base, K experts and the block partition (Sec. 2: tensor set T,
   deterministic blocks B_t).  Tensor t is cut into ceil(numel_t / block_elems)
   contiguous blocks; the last may be partial; blocks never cross tensors.  Blocks are
   numbered globally in tensor order (b = 0, 1, ...); unit (i, b) is expert i's block b.
   Tensors must be given in ascending, non-overlapping offset order.  Elements that lie
   in no tensor are never read and never written. */
typedef struct {
  mp_dtype dtype;
  uint32_t n_tensors;
  const mp_tensor* tensors;       /* host array of n_tensors, in checkpoint order */
  uint32_t block_elems;           /* elements per block; multiple of 8, in [256, 2^24] */
  const void* base;               /* device pointer: M_0 */
  uint32_t K;                     /* number of experts, 1..32 */
  const void* const* experts;     /* host array of K pointers: M_1..M_K */
  uint32_t experts_location;      /* 0 = device memory, 1 = pinned host memory */
  const uint64_t* lineage_ids;    /* optional host array of K + 1 caller ids of M_0..M_K,
                                     recorded in the manifest (Sec. 3 "Executor"); NULL = none */
} mp_family;

/* Operator and its parameters theta (Alg. 1 records op and theta with the plan). */
typedef struct {
  mp_op_kind kind;
  const float* alpha;  /* host array of K coefficients; required for AVG, TA, DARE, AVG_RENORM */
  float lambda;        /* TIES, DARE_TIES: scale of the merged task vector (1 = standard) */
  float density;       /* TIES: fraction rho of each trim population kept, in [0, 1] */
  uint32_t trim_scope; /* TIES: 0 = trim per (expert, tensor), 1 = per expert */
  double drop_p;       /* DARE, DARE_TIES: drop probability p in [0, 1] */
  uint64_t seed;       /* DARE, DARE_TIES: seed of the fixed random mask omega */
  uint32_t score_mode; /* planning score (Sec. 3, Eq. 6 and the heuristics that follow it):
                          0 = u = |coef_i| * ||Delta||_2 (Prop. 2's utility);
                          1 = score per byte, u / c in fp32 (c = the block's bytes) */
} mp_op;

typedef struct mp_index_s mp_index;
typedef struct mp_plan_s mp_plan_t;
typedef struct mp_manifest_s mp_manifest;

/*
 * mp_index_blocks — the catalog pass (Sec. 3 "Catalog"; Sec. 2: Analyze reads that build
 * norms are amortised catalog construction).  For every unit (i, b) with
 * delta = fp32(M_i) - fp32(M_0) it computes nnz = #{delta != 0}, maxabs = max |delta|
 * and norm = ||Delta_{i,t,b}||_2 (fp32, one fixed summation order: 256 lanes over
 * 16-byte vectors, a per-lane fma chain, then a butterfly over lanes).  If op->kind is
 * MP_OP_TIES it also computes the trim threshold tau of each (expert, trim group): the
 * k-th largest 15-bit key bits(bf16(|delta|)) & 0x7FFF with k = floor(density * numel)
 * (k = 0 gives tau = 0x8000, nothing kept).  For MP_OP_TIES_MASKED it computes the same
 * and also keeps every (expert, block)'s 256-bin histogram of the upper 8 key bits (zero
 * deltas in bin 0; 1 KB per unit), from which each merge finds its plan's threshold.  op
 * may be NULL for non-TIES use.
 * The family's buffers must stay valid and unchanged until the stream reaches this work.
 * Errors: MP_ERR_INVALID_ARG (bad family or op), MP_ERR_OOM, MP_ERR_CUDA; a non-finite
 * delta makes mp_index_stats (and plans built on this index) report MP_ERR_NONFINITE.
 */
mp_status mp_index_blocks(const mp_family* family, const mp_op* op, mp_stream stream, mp_index** out);

/*
 * mp_index_import — a catalog from statistics computed earlier, without reading the
 * experts (Sec. 3 "Catalog": the metadata are reusable, so planning needs no new scan).
 * norm, maxabs, nnz: host arrays [K][n_blocks], expert-major, in the layout and meaning
 * mp_index_stats returns for this family's geometry; tau: host [K][n_groups] TIES
 * thresholds (required iff op is TIES; n_groups as for mp_index_blocks), else NULL.
 * An entry whose nnz is MP_NNZ_MISSING has no block metadata (its norm and maxabs are
 * ignored): mp_plan then plans every (expert, tensor) pair holding such an entry at tensor
 * granularity (Sec. 3 "Planner", the deterministic tensor-level fallback; see mp_plan).
 * Every other entry must be a block statistic: nnz <= the block's elements, norm and
 * maxabs finite and >= 0; tau entries in [0, 0x8000].  base_hash [n_blocks] and
 * expert_hash [K][n_blocks] (host, optional, both or neither) are the catalog's block
 * hashes as mp_index_hash_values returns them.  The arrays are copied before the call
 * returns; the family's buffers are not read here (only its geometry), but must be the
 * ones the statistics describe when the index is used to merge.  The renormalised AVG
 * treats a delta as known to be zero only where nnz = 0.
 * Errors: MP_ERR_INVALID_ARG (bad family, op or entry), MP_ERR_OOM, MP_ERR_CUDA.
 */
mp_status mp_index_import(const mp_family* family, const mp_op* op, const float* norm, const float* maxabs,
                          const uint32_t* nnz, const uint32_t* tau, const uint64_t* base_hash,
                          const uint64_t* expert_hash, mp_stream stream, mp_index** out);

/*
 * mp_index_hashes — the catalog's block content hashes (Sec. 3 "Catalog" stores hashes of
 * every block; Alg. 2 validates them).  For the base and every expert, each block's bytes
 * (L of them, zero-padded to 16-byte vectors q of two little-endian 64-bit words lo_q,
 * hi_q) hash to SplitMix64(H xor L), H = sum_q lo_q * (k_q | 1) + hi_q * (rotl(k_q, 32) | 1)
 * mod 2^64 with k_q = SplitMix64(q) counted from the block's start: equal blocks hash
 * equal, and any change of one 64-bit word changes the hash (not a cryptographic hash).
 * One pass over (K + 1) N s bytes, enqueued on stream after the index's own work; the
 * hashes are stored in the index.  family must be the index's family (same geometry).
 * Errors: MP_ERR_INVALID_ARG, MP_ERR_MISMATCH, MP_ERR_OOM, MP_ERR_CUDA.
 */
mp_status mp_index_hashes(const mp_family* family, mp_index* index, mp_stream stream);

/* Host copies of the catalog's block hashes: base_hash [n_blocks], expert_hash [K][n_blocks]
   (either may be NULL).  Waits for the index work.  MP_ERR_INVALID_ARG if the index holds
   no hashes. */
mp_status mp_index_hash_values(const mp_index* index, uint64_t* base_hash, uint64_t* expert_hash);

/*
 * mp_plan — Alg. 1 PlanGen under budget B (bytes of expert reads, Eq. 3; cost of unit
 * (i,b) = elements(b) * element size, App. A.1).
 *  candidates: units with nnz > 0 (for TIES also bf16 key of maxabs >= tau; TIES_MASKED's
 *              threshold depends on the plan, so it prunes nothing more); the others
 *              contribute exactly nothing and are never read;
 *  score:      |alpha_i| * norm (TIES: |lambda| * norm), fp32 (Prop. 2's utility);
 *  order:      decreasing score, ties by ascending unit id b*K + i;
 *  select:     greedy with skip — a candidate is taken iff C_hat + c <= B.
 *  fallback:   (imported catalogs with MP_NNZ_MISSING entries; Sec. 3 "Planner") each
 *              (expert i, tensor t) holding such an entry is ONE candidate with unit id
 *              b0(t)*K + i (b0 = the tensor's first block), cost = the whole tensor's bytes
 *              and score |coef_i| * sqrt(ss), ss = the fp32 chain fma(norm, norm, ss) over
 *              t's known blocks in block order (0 if none); per byte in score mode 1 (the
 *              cost converted to fp32).  t's other units of expert i are not candidates;
 *              taking it sets bit i on every block of t.  It counts once in the number
 *              selected and in the set hash.
 * The plan records the access mask (bit i of word b = A_{i,t,b}), C_hat, the number of
 * selected units, the traversal order and a digest (FNV-1a 64 over op, theta, B, C_hat,
 * count and the sum of splitmix64(unit) over the selected units).  Budget soundness
 * (Prop. 1) holds by construction: C_hat <= B.  op must have the same kind and, for
 * TIES, the same density and trim scope as the op given to mp_index_blocks.  The traversal
 * order does not depend on B: the index keeps the order of the first operator planned on
 * it, and later plans with the same operator start from it (same result, less work).
 * Errors: MP_ERR_INVALID_ARG, MP_ERR_MISMATCH (op differs from the index's), MP_ERR_OOM,
 * MP_ERR_CUDA.
 */
mp_status mp_plan(const mp_index* index, const mp_op* op, uint64_t budget_bytes, mp_stream stream,
                  mp_plan_t** out);

/*
 * mp_merge — Alg. 2 ExecuteMerge: M_A = M_0 + Psi_op(A, Delta; omega) (Eq. 4) written in
 * full to out (a device buffer laid out like the base; every tensor element is written,
 * untouched blocks as copies of the base).  Only planned expert blocks are read;
 * omitted entries enter as zeros (non-anticipatory, Sec. 2).  Per element, fp32:
 *  AVG/TA: acc = fma(alpha_i, delta_i, acc) over selected i ascending; out = M_0 + acc
 *  DARE:   delta_i kept iff a Philox4x32-10 word >= floor(p*65536), then scaled by
 *          fp32(1/(1-p)); combined as AVG
 *  TIES:   trimmed by tau, sign elected from the sum, disjoint mean m; out = fma(lambda, m, M_0)
 * then bf16 round-to-nearest-even for bf16 families.  At B >= the full candidate cost
 * the result equals the full-read merge (Eq. 5, Prop. 1).  out must not overlap the base
 * or an expert.  The family must be the one the index was built from (same geometry).
 * *man receives the manifest: per-expert realized read bytes counted by the kernels,
 * touched blocks and the plan digest (Sec. 3 "Executor").
 * Errors: MP_ERR_INVALID_ARG, MP_ERR_MISMATCH, MP_ERR_OOM, MP_ERR_CUDA; MP_ERR_TIMEOUT
 * from mp_manifest_info if a bounded device wait gave up.
 */
mp_status mp_merge(const mp_family* family, const mp_index* index, const mp_plan_t* plan, void* out,
                   mp_stream stream, mp_manifest** man);
/* (TIES_MASKED, in mp_merge and mp_merge_touched: before the merge the threshold of the
   masked deltas is found from the catalog's per-block coarse key histograms of the selected
   blocks and one pass over the selected expert blocks that can hold keys in its coarse bin;
   those expert bytes are reported by mp_manifest_threshold_reads, apart from the planned
   reads the budget bounds.) */

/*
 * mp_merge_touched — Alg. 2 with WriteBlockOrReference: only the touched blocks (at least
 * one selected expert) are materialised; every other block of the merged checkpoint is a
 * reference to the base block and is neither read nor written.  For a touched block, out
 * receives exactly what mp_merge writes there; out keeps its previous contents everywhere
 * else.  out may therefore be the base itself (an in-place merge: each chunk is read before
 * its output is written and chunks are disjoint) or any buffer the caller has filled, e.g.
 * a copy of the base; it must not overlap an expert, nor overlap the base without being the
 * base.  The bytes moved drop from 2 N s + C_hat to 2 (touched elements) s + C_hat.  Untouched
 * blocks keep the base's bits exactly, where mp_merge writes M_0 + 0 (which turns a -0
 * into +0).  Other arguments, the manifest and errors as mp_merge.
 */
mp_status mp_merge_touched(const mp_family* family, const mp_index* index, const mp_plan_t* plan, void* out,
                           mp_stream stream, mp_manifest** man);

/*
 * mp_plan_noalloc — the same access plan as mp_plan, for callers that cannot allocate.
 * The paper has no counterpart: this is a deployment variant.  Some callers may not call
 * cudaMalloc or any allocator — code whose device memory must all come from another
 * framework's arena, latency-critical loops that cannot afford an allocation or the
 * synchronisation of a free, code running where CUDA allocation calls are not allowed.
 * This call allocates nothing: every input and output is a caller buffer, and the
 * planner's scratch is one file-scope device array of 16 MiB that every GPU loading the
 * library holds until the process exits.
 *  inputs (device): blk_len[n_blocks], blk_group[n_blocks] (TIES trim group of each
 *    block; may be NULL unless TIES), norm/maxabs/nnz [K][n_blocks] expert-major as
 *    mp_index_stats returns them, tau[K][n_groups] (TIES only, else NULL), index_err (one
 *    uint32 error word of whatever produced the statistics; 0 = fine);
 *  outputs (device): mask[n_blocks], order[K*n_blocks] (first n_candidates valid),
 *    summary[8] uint64 = {planned bytes, selected, candidates, selected-unit set hash,
 *    digest, touched blocks, error word, 0}.  The results equal mp_plan's bit for bit.
 *    This call has no tensor map, so it does not plan the tensor-level fallback: an nnz
 *    of MP_NNZ_MISSING sets the bit of value 8 in the error word, and that entry is never
 *    read.  Every buffer is aligned to its element size (summary to 8 bytes); a misaligned
 *    one returns MP_ERR_INVALID_ARG before any CUDA call.  Whether a buffer is device
 *    memory is not checked (no pointer query is made, so the call can be captured).
 * Limit: K * n_blocks <= 524288 units; larger requests return MP_ERR_INVALID_ARG and
 * launch nothing.  The first call on a device looks up the array's device address
 * (cudaGetSymbolAddress, with that device current); make that first call before any
 * stream capture.  Every call shares the one array and leaves its contents behind (the
 * planner clears what must start at zero), so calls whose GPU work overlaps — on
 * different streams, or from different threads — race and must be serialised by the
 * caller.  Errors are reported without allocating (mp_last_error returns a literal).
 */
mp_status mp_plan_noalloc(uint32_t K, uint64_t n_blocks, uint32_t n_groups, mp_dtype dtype,
                          const uint32_t* blk_len, const uint32_t* blk_group, const float* norm,
                          const float* maxabs, const uint32_t* nnz, const uint32_t* tau,
                          const uint32_t* index_err, const mp_op* op, uint64_t budget_bytes,
                          uint32_t* mask, uint32_t* order, uint64_t* summary, mp_stream stream);

/* Release an mp_index, mp_plan_t or mp_manifest (waits for its pending work).  NULL is a
   no-op.  Passing anything else is undefined. */
void mp_free(void* handle);

/* Host copies of the index statistics, expert-major [K][n_blocks]; tau is [K][n_groups]
   (n_groups = n_tensors for trim_scope 0, 1 for trim_scope 1).  Any pointer may be NULL.
   Waits for the index work.  Errors: MP_ERR_INVALID_ARG (not an index), MP_ERR_NONFINITE
   (a delta was not finite), MP_ERR_TIMEOUT (a bounded device wait in the index kernels gave
   up), MP_ERR_CUDA (a copy failed).  The arrays are filled before the error word is read. */
mp_status mp_index_stats(const mp_index* index, float* norm, float* maxabs, uint32_t* nnz, uint32_t* tau);

/* Geometry of an index: number of blocks, units (K * n_blocks) and TIES trim groups. */
mp_status mp_index_shape(const mp_index* index, uint64_t* n_blocks, uint64_t* n_units, uint32_t* n_groups);

/* Plan summary (waits for the plan work).  mask: n_blocks words; order: the traversal
   order (unit ids of the n_candidates candidates, decreasing score).  Any pointer may be
   NULL.  Errors: MP_ERR_INVALID_ARG (not a plan), MP_ERR_NONFINITE (the index saw a
   non-finite delta), MP_ERR_UNSUPPORTED (a catalog entry without statistics met a plan with
   no tensor map), MP_ERR_TIMEOUT (a bounded device wait gave up), MP_ERR_BUDGET (planned
   bytes above the budget: never expected, Prop. 1), MP_ERR_CUDA. */
mp_status mp_plan_info(const mp_plan_t* plan, uint64_t* planned_bytes, uint64_t* n_selected,
                       uint64_t* n_candidates, uint64_t* digest, uint32_t* mask, uint32_t* order);

/* Manifest (waits for the merge): realized expert-read bytes per expert (K words),
   their total, touched blocks (#{b : mask_b != 0}) and the plan digest.  Errors:
   MP_ERR_INVALID_ARG (not a manifest), MP_ERR_TIMEOUT (a bounded device wait in the merge
   gave up), MP_ERR_CUDA (the merge kernels reported another error), MP_ERR_BUDGET (realized
   reads above the planned bytes: never expected). */
mp_status mp_manifest_info(const mp_manifest* man, uint64_t* realized_bytes_per_expert,
                           uint64_t* realized_total, uint64_t* touched_blocks, uint64_t* digest);

/*
 * mp_manifest_validate — Alg. 2's hash validation before the manifest is final: after the
 * merge recorded in man (stream-ordered after it), hash every base block, every expert
 * block the plan selected (exactly the blocks the merge read) and every block of out (the
 * buffer the merge wrote), with the function of mp_index_hashes.  The inputs are compared
 * with the catalog's hashes, which detects a base or expert buffer changed since the index
 * was built; the output's hashes are recorded in the manifest (a merged checkpoint can be
 * checked against them later).  Reads N s + C_hat + N s bytes.  index must hold hashes.
 * Errors: MP_ERR_UNSUPPORTED (no catalog hashes), MP_ERR_MISMATCH (handles or geometry do
 * not belong together), MP_ERR_INVALID_ARG, MP_ERR_OOM, MP_ERR_CUDA.  Mismatches are
 * reported by mp_manifest_validation.
 */
mp_status mp_manifest_validate(const mp_family* family, const mp_index* index, const mp_plan_t* plan, const void* out,
                               mp_stream stream, mp_manifest* man);

/* Results of mp_manifest_validate (waits for it): blocks checked against the catalog,
   mismatches, and out_hash [n_blocks] the merged output's block hashes (any pointer may be
   NULL).  Returns MP_ERR_MISMATCH when a block read by the merge differs from the catalog
   (the message names the first one), MP_ERR_INVALID_ARG if the manifest was not
   validated. */
mp_status mp_manifest_validation(const mp_manifest* man, uint64_t* checked, uint64_t* mismatched, uint64_t* out_hash);

/* Expert bytes read to find the TIES_MASKED threshold (0 for every other operator): a
   subset of the selected blocks read a second time, reported apart from the realized reads
   that the budget bounds.  Waits for the merge. */
mp_status mp_manifest_threshold_reads(const mp_manifest* man, uint64_t* bytes);

/* The manifest's lineage (Sec. 3: the manifest records lineage): the K + 1 caller ids of
   M_0..M_K given in mp_family.lineage_ids at merge time, copied into ids[0..K] (all zero
   when the family gave none).  Host only; no device wait. */
mp_status mp_manifest_lineage(const mp_manifest* man, uint64_t* ids);

/* B = floor(f * C_full) with C_full = K * sum_t numel_t * element size (the full expert
   read); f in [0, 1] (clamped).  Returns 0 for an invalid family. */
uint64_t mp_budget_from_fraction(const mp_family* family, double f);

/* Thread-local text of the last error ("" if none). */
const char* mp_last_error(void);

/* Library version string (it ends in ", checked)" in the checked build). */
const char* mp_version(void);

/* Number of CUDA kernels this library has launched in this process (all devices,
   all threads).  A diagnostic for counting launches per step; never resets. */
uint64_t mp_kernel_launch_count(void);

/* Device-time trace of the calls (tracing for the phase timings of Tab. 4 and the
 * gather/merge overlap of a host-resident pool, Sec. 3 "Executor").
 *
 * mp_trace_start(capacity): from now on every call records the device time of its work
 * as ranges of two CUDA events, on the stream that runs it, until capacity ranges are
 * held: one range per mp_index_blocks (MP_TRACE_INDEX), mp_plan (MP_TRACE_PLAN) and
 * mp_merge / mp_merge_touched (MP_TRACE_MERGE) on the caller's stream, and, for experts in
 * pinned host memory, one range per segment for its gather on the side stream
 * (MP_TRACE_GATHER) and for its kernels on the caller's stream (MP_TRACE_SEGMENT).  A
 * start while a trace is held discards it.  Returns MP_ERR_INVALID_ARG for capacity 0 or
 * above 2^20, MP_ERR_CUDA if the events cannot be created.
 * mp_trace_stop(n_ranges): stops recording, waits for the recorded events and returns the
 * number of ranges held (ranges beyond the capacity are dropped, not recorded).
 * mp_trace_read(out, n): copies the first n ranges (n <= the count mp_trace_stop gave) in
 * the order they were enqueued; times are in ms from the earliest start among them.
 * Process-wide; the host-side NVTX ranges of the calls (one per entry point, named after
 * it) are always emitted and cost nothing without a tool attached.
 */
#define MP_TRACE_INDEX 1
#define MP_TRACE_PLAN 2
#define MP_TRACE_MERGE 3
#define MP_TRACE_GATHER 4
#define MP_TRACE_SEGMENT 5
typedef struct mp_trace_range {
  uint32_t kind;     /* MP_TRACE_* */
  uint32_t segment;  /* host-pool segment (GATHER, SEGMENT), else 0 */
  uint32_t stream;   /* 0: the caller's stream; 1: the host-pool gather stream */
  uint32_t reserved;
  double t0_ms;      /* start of the range's device work */
  double t1_ms;      /* end of the range's device work */
} mp_trace_range;
mp_status mp_trace_start(uint32_t capacity);
mp_status mp_trace_stop(uint64_t* n_ranges);
mp_status mp_trace_read(mp_trace_range* out, uint64_t n);

/*
 * Test hooks for the failure paths.  The paper has no counterpart: they exist so that the
 * error returns of this library (a run either produces its handle or leaves none, Alg. 2)
 * can be exercised without provoking a real GPU fault.  Both settings are process-wide and
 * are meant for tests only.
 *
 * mp_debug_inject_fault(kind, n): the n-th event of the kind from now on fails (n >= 1;
 * n = 0 disarms), once, on the host, before anything is enqueued for it:
 *   MP_FAULT_ALLOC   a device allocation of the library (handle memory, planner scratch,
 *                    host-pool staging) fails as if the device were out of memory: the call
 *                    returns MP_ERR_OOM and no handle;
 *   MP_FAULT_GATHER  a host-pool gather launch (mp_index_blocks / mp_merge with experts in
 *                    pinned host memory) is not made: the call returns MP_ERR_CUDA and no
 *                    handle, after the work already enqueued has been joined.
 * mp_last_error() then names the injected fault.  Returns MP_ERR_INVALID_ARG for an unknown
 * kind.
 *
 * mp_debug_stall_pipeline(rounds): the index and merge kernels launched from now on never arm
 * the first slot of each CTA's shared-memory ring (its bulk copy is not issued), so the
 * consumers' wait for it cannot complete, and every pipeline wait (producer or consumer
 * mbarrier) gives up after `rounds` polling rounds instead of the default 2^21.  The wait
 * that runs out sets the handle's error word; the accessors of that handle and of the
 * handles built from it return MP_ERR_TIMEOUT.  The waits that drain a CTA's own bulk
 * copies before it exits keep the full limit, so no copy is in flight when a kernel
 * returns.  rounds = 0 turns the stall off.
 */
#define MP_FAULT_ALLOC 1
#define MP_FAULT_GATHER 2
mp_status mp_debug_inject_fault(int32_t kind, uint64_t n);
void mp_debug_stall_pipeline(uint32_t rounds);

#ifdef __cplusplus
}
#endif
#endif /* MERGEPIPE_H */
