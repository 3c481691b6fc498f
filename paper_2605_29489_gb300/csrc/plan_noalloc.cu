// mp_plan_noalloc: the access plan of mp_plan for callers that must not allocate.
//
// Some callers cannot call cudaMalloc (or any allocator): code whose every device byte
// must come from another framework's memory arena, latency-critical loops that cannot
// pay for an allocation or the implicit synchronisation of a free, and code running
// where CUDA allocation calls are not permitted.  This entry point runs exactly the same
// planner kernels as mp_plan, but takes every input and output as a caller buffer and
// draws the planner's scratch from one file-scope device array of fixed size instead of
// allocating it.  That array exists once per GPU that loads the library and is held
// until the process exits.
#include <math.h>
#include <string.h>

#include <mutex>

#include "mp_internal.cuh"

namespace {

// planner scratch for up to kNoAllocMaxUnits units (K * n_blocks): 16 MiB per GPU
constexpr uint64_t kNoAllocMaxUnits = 1ull << 19;
constexpr size_t kNoAllocScratchBytes = 16u << 20;

static __device__ __align__(256) unsigned char g_plan_scratch[kNoAllocScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_setup_mu;
void* g_scratch_dev[kMaxDevices];  // device address of g_plan_scratch, per device
bool g_scratch_ready[kMaxDevices];

// error text is a string literal stored by pointer: reporting an error allocates nothing
mp_status fail_static(mp_status st, const char* msg) {
  mp::set_static_error(msg);
  return st;
}

// the array's device address for the current device; looked up once per device
mp_status scratch_for_current_device(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    cudaGetLastError();
    return fail_static(MP_ERR_CUDA, "mp_plan_noalloc: no usable current device");
  }
  std::lock_guard<std::mutex> lk(g_setup_mu);
  if (!g_scratch_ready[dev]) {
    void* p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_plan_scratch);
    if (e != cudaSuccess || p == nullptr) {
      cudaGetLastError();
      return fail_static(MP_ERR_CUDA, "mp_plan_noalloc: cudaGetSymbolAddress of the static scratch failed");
    }
    g_scratch_dev[dev] = p;
    g_scratch_ready[dev] = true;
  }
  *out = g_scratch_dev[dev];
  return MP_OK;
}

void put_u32(uint8_t* b, uint32_t& o, uint32_t x) {
  for (int k = 0; k < 4; ++k) b[o++] = (uint8_t)(x >> (8 * k));
}
void put_u64(uint8_t* b, uint32_t& o, uint64_t x) {
  for (int k = 0; k < 8; ++k) b[o++] = (uint8_t)(x >> (8 * k));
}
uint32_t fbits(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  return u;
}

}  // namespace

extern "C" mp_status mp_plan_noalloc(uint32_t K, uint64_t n_blocks, uint32_t n_groups, mp_dtype dtype,
                                     const uint32_t* blk_len, const uint32_t* blk_group, const float* norm,
                                     const float* maxabs, const uint32_t* nnz, const uint32_t* tau,
                                     const uint32_t* index_err, const mp_op* op, uint64_t budget_bytes,
                                     uint32_t* mask, uint32_t* order, uint64_t* summary, mp_stream stream) {
  if (K < 1 || K > (uint32_t)mp::kMaxK) return fail_static(MP_ERR_INVALID_ARG, "mp_plan_noalloc: K must be in 1..32");
  if (n_blocks == 0 || n_groups == 0) return fail_static(MP_ERR_INVALID_ARG, "mp_plan_noalloc: empty geometry");
  if (dtype != MP_BF16 && dtype != MP_F32) return fail_static(MP_ERR_INVALID_ARG, "mp_plan_noalloc: bad dtype");
  const uint64_t U = (uint64_t)K * n_blocks;
  if (U > kNoAllocMaxUnits || mp::plan_scratch_bytes(U, 0) > kNoAllocScratchBytes)
    return fail_static(MP_ERR_INVALID_ARG,
                       "mp_plan_noalloc: K * n_blocks exceeds the static scratch limit of 524288 units");
  if (!op || op->kind < MP_OP_AVG || op->kind > MP_OP_TIES_MASKED)
    return fail_static(MP_ERR_INVALID_ARG, "mp_plan_noalloc: bad op");
  // the same operator checks as mp_plan, with literal messages
  const bool by_lambda = op->kind == MP_OP_TIES || op->kind == MP_OP_DARE_TIES || op->kind == MP_OP_TIES_MASKED;
  if (by_lambda) {
    if (!isfinite(op->lambda)) return fail_static(MP_ERR_INVALID_ARG, "mp_plan_noalloc: lambda must be finite");
  } else {
    if (!op->alpha)
      return fail_static(MP_ERR_INVALID_ARG, "mp_plan_noalloc: alpha is required for AVG, TA, DARE and AVG_RENORM");
    for (uint32_t i = 0; i < K; ++i)
      if (!isfinite(op->alpha[i])) return fail_static(MP_ERR_INVALID_ARG, "mp_plan_noalloc: alpha must be finite");
    if (op->kind == MP_OP_AVG_RENORM)
      for (uint32_t i = 0; i < K; ++i)
        if (!(op->alpha[i] > 0.0f))
          return fail_static(MP_ERR_INVALID_ARG, "mp_plan_noalloc: AVG_RENORM needs every alpha > 0");
  }
  if (op->kind == MP_OP_TIES || op->kind == MP_OP_TIES_MASKED) {
    if (!(op->density >= 0.0f && op->density <= 1.0f))
      return fail_static(MP_ERR_INVALID_ARG, "mp_plan_noalloc: density must be in [0, 1]");
    if (op->trim_scope > 1) return fail_static(MP_ERR_INVALID_ARG, "mp_plan_noalloc: trim_scope must be 0 or 1");
  }
  if ((op->kind == MP_OP_DARE || op->kind == MP_OP_DARE_TIES) && !(op->drop_p >= 0.0 && op->drop_p <= 1.0))
    return fail_static(MP_ERR_INVALID_ARG, "mp_plan_noalloc: drop_p must be in [0, 1]");
  if (op->score_mode > 1) return fail_static(MP_ERR_INVALID_ARG, "mp_plan_noalloc: score_mode must be 0 or 1");
  if (op->kind == MP_OP_TIES && (!tau || !blk_group))
    return fail_static(MP_ERR_INVALID_ARG, "mp_plan_noalloc: TIES needs tau and blk_group");
  if (!blk_len || !norm || !maxabs || !nnz || !index_err || !mask || !order || !summary)
    return fail_static(MP_ERR_INVALID_ARG, "mp_plan_noalloc: a required buffer is NULL");
  // the kernels load every buffer by its element type: a misaligned pointer is refused
  // here rather than met by the GPU
  const auto misaligned = [](const void* q, uintptr_t a) { return q && reinterpret_cast<uintptr_t>(q) % a != 0; };
  if (misaligned(blk_len, 4) || misaligned(blk_group, 4) || misaligned(norm, 4) || misaligned(maxabs, 4) ||
      misaligned(nnz, 4) || misaligned(tau, 4) || misaligned(index_err, 4) || misaligned(mask, 4) ||
      misaligned(order, 4) || misaligned(summary, 8))
    return fail_static(MP_ERR_INVALID_ARG, "mp_plan_noalloc: a buffer is not aligned to its element size");

  void* scratch = nullptr;
  mp_status st = scratch_for_current_device(&scratch);
  if (st != MP_OK) return st;

  mp::PlanLaunch p;
  memset(&p, 0, sizeof(p));
  p.K = K;
  p.n_blocks = n_blocks;
  p.n_groups = n_groups;
  p.elem_size = dtype == MP_BF16 ? 2u : 4u;
  p.op_kind = op->kind;
  p.score_mode = op->score_mode;
  // |coef| as mp_plan takes it: fabsf also clears the sign of -0, whose score must be +0
  for (uint32_t i = 0; i < K; ++i) p.coef[i] = fabsf(by_lambda ? op->lambda : op->alpha[i]);
  p.blk_len = blk_len;
  p.blk_group = blk_group;
  p.norm = norm;
  p.maxabs = maxabs;
  p.nnz = nnz;
  p.tau = tau;
  p.index_err = index_err;
  p.budget = budget_bytes;
  p.mask = mask;
  p.order = order;
  p.summary = summary;
  uint32_t o = 0;
  put_u32(p.hdr_prefix, o, (uint32_t)op->kind);
  put_u32(p.hdr_prefix, o, K);
  for (uint32_t i = 0; i < K; ++i) put_u32(p.hdr_prefix, o, op->alpha ? fbits(op->alpha[i]) : 0u);
  put_u32(p.hdr_prefix, o, fbits(op->lambda));
  put_u32(p.hdr_prefix, o, fbits(op->density));
  put_u32(p.hdr_prefix, o, op->trim_scope);
  uint64_t pb;
  memcpy(&pb, &op->drop_p, 8);
  put_u64(p.hdr_prefix, o, pb);
  put_u64(p.hdr_prefix, o, op->seed);
  put_u32(p.hdr_prefix, o, op->score_mode);
  put_u64(p.hdr_prefix, o, budget_bytes);
  p.hdr_prefix_len = o;

  cudaError_t e = mp::launch_plan(p, scratch, reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) {
    cudaGetLastError();
    return fail_static(MP_ERR_CUDA, "mp_plan_noalloc: launching the planner kernels failed");
  }
  return MP_OK;
}
