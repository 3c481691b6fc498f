// Internal declarations of the merge library: handle layouts, kernel parameter blocks
// and the launch functions each translation unit provides to api.cu.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <string>
#include <mutex>
#include <utility>
#include <vector>

#include "checked.cuh"
#include "mergepipe.h"

namespace mp {

constexpr uint32_t kMagicIndex = 0x58495043u;  // handle tags
constexpr uint32_t kMagicPlan = 0x4C505043u;
constexpr uint32_t kMagicManifest = 0x464D5043u;

constexpr uint32_t kTauNone = 0x8000u;  // TIES threshold meaning "keep nothing"
constexpr int kLanes = 256;             // lanes of the canonical norm order (one CTA)
constexpr int kMaxK = 32;
constexpr int kCounterSlots = 64;  // realized-byte counters are spread over slots

// device error word bits
// (kErrBounds: a range failed a check of the checked build and was skipped)
enum : uint32_t { kErrNonfinite = 1u, kErrTimeout = 2u, kErrInternal = 4u, kErrMissing = 8u, kErrBounds = 16u };
// nnz of a catalog entry without block statistics (no block holds 2^32 - 1 elements)
constexpr uint32_t kNnzMissing = 0xFFFFFFFFu;

struct ExpertPtrs {
  const void* p[kMaxK];
};

// geometry shared by every handle built from one family
struct Geometry {
  mp_dtype dtype = MP_BF16;
  uint32_t elem_size = 2;
  uint32_t K = 0;
  uint32_t block_elems = 0;
  uint32_t n_tensors = 0;
  uint64_t n_blocks = 0;
  uint64_t n_params = 0;      // sum of numel
  uint64_t span_elems = 0;    // max(offset + numel)
  uint32_t max_blk_len = 0;
  std::vector<uint64_t> t_off, t_numel, t_first_block;
  bool same_as(const Geometry& o) const {
    return dtype == o.dtype && K == o.K && block_elems == o.block_elems && t_off == o.t_off &&
           t_numel == o.t_numel;
  }
};

struct Alloc {
  void* ptr = nullptr;
  size_t bytes = 0;
  cudaStream_t stream = nullptr;
};

}  // namespace mp

struct mp_index_s {
  uint32_t magic;
  uint64_t id;
  int device;
  mp::Geometry g;
  int op_kind;
  float density;
  uint32_t trim_scope;
  uint32_t n_groups;
  mp::Alloc mem;
  uint64_t* d_blk_off;     // [n_blocks] element offset of each block
  uint32_t* d_blk_len;     // [n_blocks] elements of each block
  uint32_t* d_blk_group;   // [n_blocks] TIES trim group of each block
  uint32_t* d_blk_tensor;  // [n_blocks] tensor of each block
  uint32_t* d_t_blk0;      // [n_tensors + 1] first block of each tensor, then n_blocks
  bool has_missing;        // some entry has nnz == kNnzMissing (imported catalogs only)
  uint32_t* d_unit_hist;   // [K][n_blocks][256] coarse key histograms (TIES_MASKED only)
  // the traversal order of the first operator planned on this index, kept for later plans
  // with the same operator (written once, then only read; guarded by order_mu on the host)
  mp::Alloc order_mem;
  uint32_t* d_order_cache;           // [K * n_blocks]
  unsigned long long* d_order_q;     // candidates
  std::vector<uint8_t> order_key;    // the operator's digest header without the budget
  bool order_captured;               // the cached order was written under stream capture
  cudaEvent_t order_ready;
  std::mutex* order_mu;
  mp::Alloc hash_mem;      // the catalog's block hashes, once computed or imported
  unsigned long long* d_base_hash;    // [n_blocks]
  unsigned long long* d_expert_hash;  // [K][n_blocks]
  float* d_norm;           // [K][n_blocks]
  float* d_maxabs;         // [K][n_blocks]
  uint32_t* d_nnz;         // [K][n_blocks]
  uint32_t* d_tau;         // [K][n_groups] (TIES only)
  uint32_t* d_err;         // error word
  cudaEvent_t done;
  bool captured;           // built under stream capture: waits go through the device
  std::vector<std::pair<void*, size_t>> pinned;  // pinned staging of the uploads (released by mp_free)
  std::vector<uint64_t> h_blk_off;  // host copy of the block table (segments of a host pool)
  std::vector<uint32_t> h_blk_len;
};

struct mp_plan_s {
  uint32_t magic;
  uint64_t id;
  uint64_t index_id;
  int device;
  mp::Geometry g;
  int op_kind;
  float alpha[mp::kMaxK];
  float lambda, density;
  uint32_t trim_scope;
  double drop_p;
  uint64_t seed;
  uint64_t budget;
  uint32_t n_groups;
  mp::Alloc mem;
  uint32_t* d_mask;        // [n_blocks] access mask
  uint32_t* d_order;       // [K*n_blocks] traversal order (first n_cand valid)
  uint64_t* d_summary;     // [8] chat, n_sel, n_cand, set_hash, digest, touched, err, pad
  uint64_t* h_summary;     // pinned host copy of d_summary
  cudaEvent_t done;
  bool captured;           // built under stream capture: waits go through the device
};

struct mp_manifest_s {
  uint32_t magic;
  uint64_t plan_id;
  int device;
  uint32_t K;
  mp::Alloc mem;
  unsigned long long* d_realized;  // [kCounterSlots][K]
  uint32_t* d_err;
  unsigned long long* h_realized;  // pinned host copy (slots summed on host)
  uint32_t* h_err;
  uint64_t planned, touched, digest;
  uint64_t lineage[mp::kMaxK + 1];  // caller ids of M_0..M_K (zeros when none were given)
  cudaEvent_t done;
  bool captured;                    // built under stream capture: waits go through the device
  // hash validation (mp_manifest_validate): checked / mismatched / first bad item, and
  // the output's block hashes
  mp::Alloc valid_mem;
  unsigned long long* d_vresult;   // [3]
  unsigned long long* d_out_hash;  // [n_blocks]
  uint64_t n_blocks;
  cudaEvent_t valid_done;
};

namespace mp {

// ---- launch accounting (api.cu) ------------------------------------------------------------
void count_launches(uint64_t n);

// ---- error reporting (api.cu) -----------------------------------------------------------
void set_error(const std::string& msg);
// records a string literal as the last error without allocating
void set_static_error(const char* msg);
mp_status cuda_fail(cudaError_t e, const char* what);

// CUDA graphs: a call made while its stream is being captured records its work (and its
// handle's completion event) into the graph.  Such an event cannot be waited for from the
// host, so the waits of a handle built under capture go through the whole device, which
// covers every replay of the graph enqueued so far.
bool capturing(cudaStream_t st);
cudaError_t wait_handle(cudaEvent_t done, bool captured);
cudaError_t stream_wait(cudaStream_t cs, cudaEvent_t ev, bool ev_captured, bool now_captured);

// device-time ranges of the calls (trace.cu): trace_begin records the start of a range on
// st and returns its ticket, or -1 while no trace is recording (or it is full); trace_end
// records the end on the stream that ran the range's work
int trace_begin(uint32_t kind, uint32_t segment, uint32_t stream_kind, cudaStream_t st);
void trace_end(int ticket, cudaStream_t st);
struct TraceScope {
  int ticket;
  cudaStream_t st;
  TraceScope(uint32_t kind, cudaStream_t s) : ticket(trace_begin(kind, 0, 0, s)), st(s) {}
  ~TraceScope() { trace_end(ticket, st); }
};
// host-side NVTX range of an entry point, for the lifetime of the object
struct NvtxScope {
  explicit NvtxScope(const char* name);
  ~NvtxScope();
};

// ---- index (index.cu) -------------------------------------------------------------------
struct IndexLaunch {
  mp_dtype dtype;
  uint32_t K;
  uint64_t n_blocks;
  uint32_t n_groups;
  const void* base;
  ExpertPtrs experts;
  const uint64_t* blk_off;
  const uint32_t* blk_len;
  const uint32_t* blk_group;
  float* norm;
  float* maxabs;
  uint32_t* nnz;
  uint32_t* err;
  // TIES (null when not TIES)
  unsigned long long* coarse;  // [K][n_groups][256]
  unsigned long long* fine;    // [K][n_groups][128]
  const unsigned long long* kth;  // [n_groups] k = floor(density * numel_g)
  uint32_t* estar;             // [K][n_groups] coarse bin of tau (or 0xFFFFFFFF)
  unsigned long long* rank;    // [K][n_groups] rank of tau inside that bin
  uint32_t* tau;               // [K][n_groups]
  // TIES after masking: the catalog keeps each unit's coarse key histogram (256 bins, zero
  // deltas in bin 0); the fine pass then reads only the blocks the plan selected and counts
  // the expert bytes it reads
  uint32_t* unit_hist;         // [K][n_blocks][256] or null
  // TIES with a predicted window (device-resident experts, not after masking; null
  // otherwise): a sample of each trim group predicts the coarse bin of its threshold, the
  // catalog pass counts the 384 keys of a window around it at full resolution, and the
  // two-level select runs only for the (expert, group) pairs whose threshold left the window
  float density;                  // rho
  const uint32_t* grp_blk0;       // [n_groups + 1] first block of each trim group, then n_blocks
  const uint2* samp_span;         // [n_samp_spans] {group, first block} of each sampling CTA
  uint32_t n_samp_spans;
  unsigned long long* shist;      // [K][n_groups][256] coarse bins of the sampled deltas
  unsigned long long* scnt;       // [n_groups] sampled elements
  uint32_t* wlo;                  // [K][n_groups] first key L of the window
  unsigned long long* wfine;      // [K][n_groups][384] counts of the keys L .. L + 383
  unsigned long long* wabove;     // [K][n_groups] keys above the window
  uint32_t* gmiss;                // [K][n_groups] 1: the pair needs the two-level select
  uint32_t* miss;                 // [1] nonzero when some pair does
  const uint32_t* mask;        // the access mask for the fine pass, or null (every block)
  unsigned long long* thr_reads;  // expert bytes read by the fine pass, or null
  unsigned long long* work;    // item counter of the dynamic scheduler (zeroed per launch)
  // the launch covers blocks [b_begin, b_end); expert pointers address element
  // expert_origin of the flat layout (0 for resident experts, a segment start when they
  // point into a staging buffer)
  uint64_t b_begin, b_end, expert_origin;
  Extents ext;            // buffer extents, for the checks of the checked build
  int defer_ties_select;  // 1: leave the TIES selection to launch_ties_finish
  uint32_t wait_limit;    // try_wait rounds of the pipeline waits (0: the default)
  uint32_t stall;         // test hook: every CTA's first ring fill is never armed
};
cudaError_t launch_index(const IndexLaunch& p, cudaStream_t st);
cudaError_t launch_ties_finish(const IndexLaunch& p, cudaStream_t st);
// the windowed TIES catalog in stages, for a host-resident pool walked in segments: the
// sample and window select over the whole family (experts read in place over the host
// mapping); one pass over blocks [b_begin, b_end) of staged experts with window bins, or with
// coarse bins for the pairs the window finish marked (a launch that returns at once when
// none is); the window finish
cudaError_t launch_ties_window_begin(const IndexLaunch& p, cudaStream_t st);
cudaError_t launch_index_pass(const IndexLaunch& p, bool window, cudaStream_t st);
cudaError_t launch_ties_window_end(const IndexLaunch& p, cudaStream_t st);
// the TIES_MASKED threshold of a plan: coarse bins summed from the per-unit histograms of
// the selected blocks (zero entries for the others), then the select, fine pass and select
// of launch_ties_finish restricted to the selected blocks (p.mask)
cudaError_t launch_ties_masked(const IndexLaunch& p, cudaStream_t st);

// ---- plan (plan.cu) ---------------------------------------------------------------------
struct PlanLaunch {
  uint32_t K;
  uint64_t n_blocks;
  uint32_t n_groups;
  uint32_t elem_size;
  int op_kind;
  uint32_t score_mode;  // 0: |coef_i| * norm; 1: that per byte of the block
  float coef[kMaxK];   // |alpha_i| or |lambda|
  const uint32_t* blk_len;
  const uint32_t* blk_group;
  const float* norm;
  const float* maxabs;
  const uint32_t* nnz;
  const uint32_t* tau;
  const uint32_t* index_err;
  // tensor-level fallback: with fallback = 1, an (expert, tensor) pair holding an entry
  // with nnz == kNnzMissing is planned as one unit (blk_tensor, t_blk0 as in mp_index_s);
  // with fallback = 0 such an entry is reported (kErrMissing) and never read
  uint32_t fallback;
  uint32_t n_tensors;
  const uint32_t* blk_tensor;
  const uint32_t* t_blk0;
  // the candidates' traversal order does not depend on the budget: a plan may take it
  // from an earlier plan of the same index and operator (cache_*_in), or leave it for
  // later ones (cache_*_out); all null for a plan on its own
  const uint32_t* cache_order_in;
  const unsigned long long* cache_q_in;
  uint32_t* cache_order_out;
  unsigned long long* cache_q_out;
  uint64_t budget;
  uint32_t* mask;
  uint32_t* order;
  uint64_t* summary;
  // digest header fields (host-built, hashed on the device after C_hat is known)
  uint8_t hdr_prefix[256];
  uint32_t hdr_prefix_len;
};
// scratch bytes the planner needs for n_units units and n_pairs (expert, tensor) pairs
// (n_pairs = 0 without the tensor-level fallback)
size_t plan_scratch_bytes(uint64_t n_units, uint64_t n_pairs);
cudaError_t launch_plan(const PlanLaunch& p, void* scratch, cudaStream_t st);

// ---- merge (merge.cu) -------------------------------------------------------------------
struct MergeLaunch {
  mp_dtype dtype;
  int op_kind;
  uint32_t K;
  uint64_t n_blocks;
  uint32_t block_elems;
  uint32_t n_groups;
  const void* base;
  ExpertPtrs experts;
  void* out;
  const uint64_t* blk_off;
  const uint32_t* blk_len;
  const uint32_t* blk_group;
  const uint32_t* mask;
  const uint32_t* tau;  // TIES
  const uint32_t* nnz;  // renormalised AVG: catalog nonzero counts [K][n_blocks]
  float alpha[kMaxK];
  float lambda;
  float sigma;          // DARE rescale
  uint32_t dare_T;      // DARE keep threshold on 16-bit words
  uint32_t dare_T16;    // min(dare_T, 65535) << 16: the same test on a word in the upper half
                        // (p = 1 has sigma = 0, so a word kept by the clamp adds exactly +-0)
  uint32_t dare_rk[10][2];  // DARE: Philox round keys of the seed (precomputed on the host)
  uint64_t seed;
  unsigned long long* realized;  // [kCounterSlots][K]
  unsigned long long* work;      // chunk counter of the dynamic scheduler (zeroed per launch)
  uint32_t* err;
  uint64_t b_begin, b_end, expert_origin;  // as in IndexLaunch
  Extents ext;                             // as in IndexLaunch
  uint32_t touched_only;  // 1: blocks with an empty mask are neither read nor written
  uint32_t wait_limit;    // try_wait rounds of the pipeline waits (0: the default)
  uint32_t stall;         // test hook: every CTA's first ring fill is never armed
};
cudaError_t launch_merge(const MergeLaunch& p, cudaStream_t st);

// ---- host-pool gather (gather.cu) ---------------------------------------------------------
// copies the planned (block, expert) pairs of blocks [b_begin, b_end) from the experts'
// pinned host memory into staging buffers laid out like the flat checkpoint from element
// `origin` on
struct GatherLaunch {
  uint32_t K;
  uint32_t elem_size;
  uint64_t b_begin, b_end, origin;
  const uint64_t* blk_off;
  const uint32_t* blk_len;
  const uint32_t* mask;   // the access mask of the plan; NULL copies every expert block
  ExpertPtrs src;         // device views of the host experts
  ExpertPtrs dst;         // staging buffers
  unsigned long long* gathered;  // bytes copied, accumulated (may be NULL)
  const uint32_t* gate;          // when set, the launch copies nothing unless *gate != 0
  Extents ext;                   // span: the host experts; x_span: the staging from origin
  uint32_t* err;                 // the call's error word (checked build)
};
cudaError_t launch_gather(const GatherLaunch& g, cudaStream_t st);
// copies and fills by kernel on st (no copy engine); host buffers must be pinned memory
cudaError_t launch_copy(void* dst, const void* src, size_t bytes, cudaStream_t st);
cudaError_t launch_fill(void* dst, uint32_t byte_value, size_t bytes, cudaStream_t st);

// ---- block content hashes (hash.cu) --------------------------------------------------------
// catalog mode (validate = 0): hash every block of the base and of each expert into
// base_hash / expert_hash.  Validation: hash the base, the expert blocks selected by mask
// and every block of out; compare the first two with the catalog (result[0] += blocks
// checked, result[1] += mismatches, result[2] = min mismatching item), write out_hash.
struct HashLaunch {
  uint32_t K;
  uint32_t elem_size;
  uint64_t n_blocks;
  const uint64_t* blk_off;
  const uint32_t* blk_len;
  const void* base;
  ExpertPtrs experts;
  const void* out;
  const uint32_t* mask;
  uint32_t validate;
  unsigned long long* base_hash;    // [n_blocks]
  unsigned long long* expert_hash;  // [K][n_blocks]
  unsigned long long* out_hash;     // [n_blocks]
  unsigned long long* result;       // [3]
  Extents ext;                      // every buffer spans the family (x_span = span)
  uint32_t* err;                    // the call's error word (checked build)
};
cudaError_t launch_hash(const HashLaunch& p, cudaStream_t st);

}  // namespace mp
