// Bounds checks of the checked build (compiled with -DMP_CHECKED into
// libmergepipe_checked.so; the default build compiles none of them).
//
// The kernels that stream checkpoint data address it through the block table: a work item
// or chunk is a block b and an element range [off, off + n) inside it, read from the base
// and from the experts whose bits are set in the item's expert mask (the plan's access
// mask, or a run of the catalog's experts).  In the checked build every such range is
// checked before any copy or load is issued for it: against the block table's entry, the
// launch's block range, the extents of the buffers it touches, the 16-byte alignment a
// bulk copy needs, and the number of experts.  A range that fails is not touched: the
// kernel sets kErrBounds in the call's error word, skips it, and the accessors of the
// call's handle report the failure.  No check traps.
#pragma once

#include <stdint.h>

namespace mp {

#ifdef MP_CHECKED
constexpr bool kChecked = true;
#else
constexpr bool kChecked = false;
#endif

// what a launch may touch besides its block range
struct Extents {
  uint64_t span;    // elements of the base and output buffers (and of host-resident experts)
  uint64_t x_span;  // elements each expert buffer holds from the launch's expert origin (all
                    // of them for resident experts, a segment's staging for a host pool)
};

// true when elements [off, off + n) of block b (table entry blk_off, blk_len), read from the
// base and from the experts set in `experts` (whose buffers start at element x_origin), lie
// inside the block, the block inside [b_begin, b_end), the range inside every buffer, its
// first byte at a 16-byte boundary (with no byte offset past 2^64), and every expert bit
// below K
__host__ __device__ inline bool chunk_in_bounds(uint64_t b, uint64_t b_begin, uint64_t b_end, uint64_t blk_off,
                                                uint32_t blk_len, uint64_t off, uint32_t n, uint64_t experts,
                                                uint32_t K, uint32_t elem_size, uint64_t x_origin,
                                                const Extents& x) {
  if (b < b_begin || b >= b_end) return false;
  if (off < blk_off || off - blk_off > blk_len || n > blk_len - (off - blk_off)) return false;
  if (elem_size == 0u || x.span > ~0ull / elem_size) return false;  // byte offsets must not wrap
  if (off > x.span || n > x.span - off) return false;
  if (((off * elem_size) & 15u) != 0u) return false;
  if (K > 64u || (K < 64u && (experts >> K) != 0u)) return false;
  if (experts != 0u && (off < x_origin || off - x_origin > x.x_span || n > x.x_span - (off - x_origin)))
    return false;
  return true;
}

// the expert mask of experts i0 .. i0 + kc - 1
__host__ __device__ inline uint64_t expert_run(uint32_t i0, uint32_t kc) {
  if (kc == 0u || i0 >= 64u) return kc == 0u ? 0u : ~0ull;  // i0 >= 64 is never valid: flag it
  const uint64_t run = kc >= 64u ? ~0ull : ((1ull << kc) - 1ull);
  return run << i0;
}

}  // namespace mp
