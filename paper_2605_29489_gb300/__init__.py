"""GB300 (sm_103a) budgeted, mask-aware model merge — Python binding of the C ABI.

The three steps of the method (MergePipe: index, plan, merge) run in the CUDA
library ``_build/libmergepipe.so`` behind ``include/mergepipe.h``.  This module
only marshals arguments: torch tensors provide device memory and streams, and
every call goes straight to the C entry point of the same name.  There is no
CPU fallback: if the library cannot be built or loaded, the calls raise.

    fam   = family(tensors, base, experts, block_elems=65536)
    op    = make_op(MP_OP_TA, alpha=[0.3] * K)
    idx   = mp_index_blocks(fam, op)
    plan  = mp_plan(idx, op, mp_budget_from_fraction(fam, 0.25))
    man   = mp_merge(fam, idx, plan, out)
    info  = mp_manifest_info(man)
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

__all__ = [
    "MP_OK", "MP_BF16", "MP_F32", "MP_OP_AVG", "MP_OP_TA", "MP_OP_TIES", "MP_OP_DARE", "MP_OP_AVG_RENORM", "MP_OP_DARE_TIES",
    "MP_OP_TIES_MASKED", "mp_manifest_threshold_reads", "MergePipeError",
    "family", "make_op", "mp_index_blocks", "mp_plan", "mp_merge", "mp_merge_touched", "mp_free", "mp_index_stats",
    "mp_index_shape", "mp_plan_info", "mp_manifest_info", "mp_manifest_lineage", "mp_budget_from_fraction", "mp_last_error",
    "mp_version", "mp_kernel_launch_count", "mp_plan_noalloc", "mp_index_import", "MP_NNZ_MISSING", "mp_index_hashes",
    "mp_index_hash_values", "mp_manifest_validate", "mp_manifest_validation", "lib",
    "MP_FAULT_ALLOC", "MP_FAULT_GATHER", "mp_debug_inject_fault", "mp_debug_stall_pipeline",
    "MP_TRACE_INDEX", "MP_TRACE_PLAN", "MP_TRACE_MERGE", "MP_TRACE_GATHER", "MP_TRACE_SEGMENT",
    "mp_trace_start", "mp_trace_stop", "library_path",
]

MP_OK = 0
MP_ERR = {-1: "MP_ERR_INVALID_ARG", -2: "MP_ERR_CUDA", -3: "MP_ERR_OOM", -4: "MP_ERR_NONFINITE",
          -5: "MP_ERR_BUDGET", -6: "MP_ERR_TIMEOUT", -7: "MP_ERR_UNSUPPORTED", -8: "MP_ERR_MISMATCH"}
MP_BF16, MP_F32 = 0, 1
MP_OP_AVG, MP_OP_TA, MP_OP_TIES, MP_OP_DARE, MP_OP_AVG_RENORM, MP_OP_DARE_TIES, MP_OP_TIES_MASKED = 0, 1, 2, 3, 4, 5, 6
MP_NNZ_MISSING = 0xFFFFFFFF   # catalog entry without block statistics (tensor-level fallback)
MP_FAULT_ALLOC, MP_FAULT_GATHER = 1, 2  # test hooks: kinds of injected host-side failures
# kinds of traced device-time ranges (mp_trace_start)
MP_TRACE_INDEX, MP_TRACE_PLAN, MP_TRACE_MERGE, MP_TRACE_GATHER, MP_TRACE_SEGMENT = 1, 2, 3, 4, 5


class MergePipeError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{MP_ERR.get(status, status)}: {msg}")
        self.status = status


class _Tensor(ctypes.Structure):
    _fields_ = [("offset_elems", ctypes.c_uint64), ("numel", ctypes.c_uint64)]


class _Family(ctypes.Structure):
    _fields_ = [("dtype", ctypes.c_int), ("n_tensors", ctypes.c_uint32), ("tensors", ctypes.POINTER(_Tensor)),
                ("block_elems", ctypes.c_uint32), ("base", ctypes.c_void_p), ("K", ctypes.c_uint32),
                ("experts", ctypes.POINTER(ctypes.c_void_p)), ("experts_location", ctypes.c_uint32),
                ("lineage_ids", ctypes.POINTER(ctypes.c_uint64))]


class _TraceRange(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_uint32), ("segment", ctypes.c_uint32), ("stream", ctypes.c_uint32),
                ("reserved", ctypes.c_uint32), ("t0_ms", ctypes.c_double), ("t1_ms", ctypes.c_double)]


class _Op(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int), ("alpha", ctypes.POINTER(ctypes.c_float)), ("lambda_", ctypes.c_float),
                ("density", ctypes.c_float), ("trim_scope", ctypes.c_uint32), ("drop_p", ctypes.c_double),
                ("seed", ctypes.c_uint64), ("score_mode", ctypes.c_uint32)]


_lib = None


def library_path() -> str:
    """the default library, or with MERGEPIPE_CHECKED=1 in the environment the checked build
    (every range a kernel streams is checked against the block table and the buffers first;
    a failed check is reported by the accessors as MP_ERR_CUDA)"""
    from . import build as _build
    return _build.build_mergepipe(checked=os.environ.get("MERGEPIPE_CHECKED", "0") == "1")


def lib():
    """The loaded CUDA library (built in-tree on first use)."""
    global _lib
    if _lib is None:
        L = ctypes.CDLL(library_path())
        vp, u64, st = ctypes.c_void_p, ctypes.c_uint64, ctypes.c_int32
        for name, args in [
            ("mp_index_blocks", [vp, vp, vp, vp]),
            ("mp_index_import", [vp, vp, vp, vp, vp, vp, vp, vp, vp, vp]),
            ("mp_index_hashes", [vp, vp, vp]),
            ("mp_index_hash_values", [vp, vp, vp]),
            ("mp_manifest_validate", [vp, vp, vp, vp, vp, vp]),
            ("mp_manifest_validation", [vp, vp, vp, vp]),
            ("mp_plan", [vp, vp, u64, vp, vp]),
            ("mp_merge", [vp, vp, vp, vp, vp, vp]),
            ("mp_merge_touched", [vp, vp, vp, vp, vp, vp]),
            ("mp_index_stats", [vp, vp, vp, vp, vp]),
            ("mp_index_shape", [vp, vp, vp, vp]),
            ("mp_plan_info", [vp, vp, vp, vp, vp, vp, vp]),
            ("mp_manifest_info", [vp, vp, vp, vp, vp]),
            ("mp_manifest_lineage", [vp, vp]),
            ("mp_manifest_threshold_reads", [vp, vp]),
        ]:
            f = getattr(L, name)
            f.restype, f.argtypes = st, args
        L.mp_free.restype, L.mp_free.argtypes = None, [vp]
        L.mp_budget_from_fraction.restype, L.mp_budget_from_fraction.argtypes = u64, [vp, ctypes.c_double]
        L.mp_last_error.restype, L.mp_last_error.argtypes = ctypes.c_char_p, []
        L.mp_version.restype, L.mp_version.argtypes = ctypes.c_char_p, []
        L.mp_kernel_launch_count.restype, L.mp_kernel_launch_count.argtypes = u64, []
        L.mp_debug_inject_fault.restype, L.mp_debug_inject_fault.argtypes = st, [ctypes.c_int32, u64]
        L.mp_debug_stall_pipeline.restype, L.mp_debug_stall_pipeline.argtypes = None, [ctypes.c_uint32]
        L.mp_trace_start.restype, L.mp_trace_start.argtypes = st, [ctypes.c_uint32]
        L.mp_trace_stop.restype, L.mp_trace_stop.argtypes = st, [ctypes.POINTER(u64)]
        L.mp_trace_read.restype, L.mp_trace_read.argtypes = st, [ctypes.POINTER(_TraceRange), u64]
        _lib = L
    return _lib


def _check(rc: int):
    if rc != MP_OK:
        raise MergePipeError(rc, mp_last_error())


def _stream_ptr(stream) -> int | None:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


class Family:
    """An mp_family plus the Python objects that keep its memory alive."""

    def __init__(self, tensors, base, experts, block_elems, dtype, experts_location, lineage_ids=None):
        self.tensors = [(int(o), int(n)) for o, n in tensors]
        self.base, self.experts = base, list(experts)
        self._tarr = (_Tensor * len(self.tensors))(*[_Tensor(o, n) for o, n in self.tensors])
        self._earr = (ctypes.c_void_p * len(self.experts))(*[_ptr(e) for e in self.experts])
        self._lin = None if lineage_ids is None else (ctypes.c_uint64 * (len(self.experts) + 1))(*lineage_ids)
        self.c = _Family(dtype, len(self.tensors), self._tarr, block_elems, _ptr(base), len(self.experts),
                         self._earr, experts_location, self._lin)

    @property
    def K(self):
        return self.c.K

    def ref(self):
        return ctypes.byref(self.c)


def _ptr(t) -> int:
    if hasattr(t, "data_ptr"):
        return t.data_ptr()
    if isinstance(t, np.ndarray):
        return t.ctypes.data
    return int(t)


def family(tensors, base, experts, block_elems=65536, dtype=None, experts_location=None, lineage_ids=None) -> Family:
    """tensors: [(offset_elems, numel)] in checkpoint order; base/experts: flat torch tensors;
    lineage_ids: optional K + 1 integer ids of the base and the experts, kept in the manifest"""
    if dtype is None:
        import torch
        dtype = MP_BF16 if base.dtype == torch.bfloat16 else MP_F32
    if experts_location is None:
        experts_location = 0 if getattr(experts[0], "is_cuda", True) else 1
    if lineage_ids is not None and len(lineage_ids) != len(experts) + 1:
        raise ValueError("lineage_ids needs K + 1 ids (base first)")
    return Family(tensors, base, experts, block_elems, dtype, experts_location, lineage_ids)


class Op:
    def __init__(self, kind, alpha, lam, density, trim_scope, drop_p, seed, score_mode=0):
        self.alpha = None if alpha is None else np.ascontiguousarray(np.asarray(alpha, np.float32))
        ap = None if self.alpha is None else self.alpha.ctypes.data_as(ctypes.POINTER(ctypes.c_float))
        self.c = _Op(kind, ap, lam, density, trim_scope, drop_p, seed, score_mode)
        self.kind = kind

    def ref(self):
        return ctypes.byref(self.c)


def make_op(kind, alpha=None, lam=1.0, density=0.2, trim_scope=0, drop_p=0.0, seed=0, score_mode=0) -> Op:
    return Op(kind, alpha, float(lam), float(density), int(trim_scope), float(drop_p), int(seed), int(score_mode))


class Handle:
    """Owns an opaque library handle; released by mp_free (or on garbage collection)."""

    def __init__(self, ptr: int, kind: str, keep=()):
        self.ptr, self.kind, self._keep = ptr, kind, keep

    def free(self):
        if self.ptr:
            lib().mp_free(ctypes.c_void_p(self.ptr))
            self.ptr = 0

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *a):
        self.free()


def mp_index_blocks(fam: Family, op: Op | None = None, stream=None) -> Handle:
    out = ctypes.c_void_p()
    _check(lib().mp_index_blocks(fam.ref(), None if op is None else op.ref(), ctypes.c_void_p(_stream_ptr(stream)),
                                 ctypes.byref(out)))
    return Handle(out.value, "index")


def mp_index_import(fam: Family, op: Op | None, norm, maxabs, nnz, tau=None, stream=None, base_hash=None,
                    expert_hash=None) -> Handle:
    """a catalog from saved statistics (host arrays [K, n_blocks], tau [K, n_groups] for TIES,
    optional block hashes [n_blocks] and [K, n_blocks]); entries with nnz == MP_NNZ_MISSING
    have no statistics"""
    arrs = [np.ascontiguousarray(norm, np.float32), np.ascontiguousarray(maxabs, np.float32),
            np.ascontiguousarray(nnz, np.uint32), None if tau is None else np.ascontiguousarray(tau, np.uint32),
            None if base_hash is None else np.ascontiguousarray(base_hash, np.uint64),
            None if expert_hash is None else np.ascontiguousarray(expert_hash, np.uint64)]
    out = ctypes.c_void_p()
    _check(lib().mp_index_import(fam.ref(), None if op is None else op.ref(),
                                 *[None if a is None else a.ctypes.data for a in arrs],
                                 ctypes.c_void_p(_stream_ptr(stream)), ctypes.byref(out)))
    return Handle(out.value, "index")


def mp_index_hashes(fam: Family, index: Handle, stream=None):
    """add the catalog's block content hashes to an index (one pass over every checkpoint)"""
    _check(lib().mp_index_hashes(fam.ref(), ctypes.c_void_p(index.ptr), ctypes.c_void_p(_stream_ptr(stream))))


def mp_index_hash_values(index: Handle):
    """(base_hash [n_blocks], expert_hash [K, n_blocks]) uint64"""
    nb, nu, _ = mp_index_shape(index)
    bh = np.zeros(nb, np.uint64)
    eh = np.zeros((nu // nb, nb), np.uint64)
    _check(lib().mp_index_hash_values(ctypes.c_void_p(index.ptr), bh.ctypes.data, eh.ctypes.data))
    return bh, eh


def mp_manifest_threshold_reads(man: Handle) -> int:
    """expert bytes read to find a TIES_MASKED threshold (0 for other operators)"""
    v = ctypes.c_uint64()
    _check(lib().mp_manifest_threshold_reads(ctypes.c_void_p(man.ptr), ctypes.byref(v)))
    return v.value


def mp_manifest_validate(fam: Family, index: Handle, plan: Handle, out, man: Handle, stream=None):
    """Alg. 2's hash validation of the blocks a merge read, and the output's block hashes"""
    _check(lib().mp_manifest_validate(fam.ref(), ctypes.c_void_p(index.ptr), ctypes.c_void_p(plan.ptr),
                                      ctypes.c_void_p(_ptr(out)), ctypes.c_void_p(_stream_ptr(stream)),
                                      ctypes.c_void_p(man.ptr)))


def mp_manifest_validation(man: Handle, n_blocks: int, check: bool = True):
    """dict(checked, mismatched, out_hash, status) of mp_manifest_validate"""
    c, m = ctypes.c_uint64(), ctypes.c_uint64()
    oh = np.zeros(n_blocks, np.uint64)
    rc = lib().mp_manifest_validation(ctypes.c_void_p(man.ptr), ctypes.byref(c), ctypes.byref(m), oh.ctypes.data)
    if check:
        _check(rc)
    return dict(checked=c.value, mismatched=m.value, out_hash=oh, status=rc,
                error=mp_last_error() if rc != MP_OK else "")


def mp_plan(index: Handle, op: Op, budget_bytes: int, stream=None) -> Handle:
    out = ctypes.c_void_p()
    _check(lib().mp_plan(ctypes.c_void_p(index.ptr), op.ref(), int(budget_bytes),
                         ctypes.c_void_p(_stream_ptr(stream)), ctypes.byref(out)))
    return Handle(out.value, "plan")


def mp_merge(fam: Family, index: Handle, plan: Handle, out, stream=None) -> Handle:
    man = ctypes.c_void_p()
    _check(lib().mp_merge(fam.ref(), ctypes.c_void_p(index.ptr), ctypes.c_void_p(plan.ptr), ctypes.c_void_p(_ptr(out)),
                          ctypes.c_void_p(_stream_ptr(stream)), ctypes.byref(man)))
    return Handle(man.value, "manifest")


def mp_merge_touched(fam: Family, index: Handle, plan: Handle, out, stream=None) -> Handle:
    man = ctypes.c_void_p()
    _check(lib().mp_merge_touched(fam.ref(), ctypes.c_void_p(index.ptr), ctypes.c_void_p(plan.ptr),
                                  ctypes.c_void_p(_ptr(out)), ctypes.c_void_p(_stream_ptr(stream)), ctypes.byref(man)))
    return Handle(man.value, "manifest")


def mp_free(h: Handle | None):
    if h is not None:
        h.free()


def mp_index_shape(index: Handle):
    nb, nu, ng = ctypes.c_uint64(), ctypes.c_uint64(), ctypes.c_uint32()
    _check(lib().mp_index_shape(ctypes.c_void_p(index.ptr), ctypes.byref(nb), ctypes.byref(nu), ctypes.byref(ng)))
    return nb.value, nu.value, ng.value


def mp_index_stats(index: Handle, check: bool = True):
    """(norm, maxabs, nnz, tau) as numpy arrays [K, n_blocks] / [K, n_groups]"""
    nb, nu, ng = mp_index_shape(index)
    K = nu // nb
    norm = np.zeros((K, nb), np.float32)
    maxabs = np.zeros((K, nb), np.float32)
    nnz = np.zeros((K, nb), np.uint32)
    tau = np.zeros((K, ng), np.uint32)
    rc = lib().mp_index_stats(ctypes.c_void_p(index.ptr), norm.ctypes.data, maxabs.ctypes.data, nnz.ctypes.data,
                              tau.ctypes.data)
    if check:
        _check(rc)
    return norm, maxabs, nnz, tau


def mp_plan_info(plan: Handle, index: Handle | None = None, with_arrays: bool = True, check: bool = True):
    """dict(chat, n_sel, n_cand, digest[, mask, order])"""
    v = [ctypes.c_uint64() for _ in range(4)]
    rc = lib().mp_plan_info(ctypes.c_void_p(plan.ptr), *[ctypes.byref(x) for x in v], None, None)
    if check:
        _check(rc)
    d = dict(chat=v[0].value, n_sel=v[1].value, n_cand=v[2].value, digest=v[3].value, status=rc)
    if with_arrays and index is not None:
        nb, nu, _ = mp_index_shape(index)
        mask = np.zeros(nb, np.uint32)
        order = np.zeros(max(d["n_cand"], 1), np.uint32)
        rc2 = lib().mp_plan_info(ctypes.c_void_p(plan.ptr), None, None, None, None, mask.ctypes.data, order.ctypes.data)
        if check:
            _check(rc2)
        d["mask"], d["order"] = mask, order[: d["n_cand"]]
    return d


def mp_manifest_info(man: Handle, K: int, check: bool = True):
    per = np.zeros(K, np.uint64)
    tot, touched, dig = ctypes.c_uint64(), ctypes.c_uint64(), ctypes.c_uint64()
    rc = lib().mp_manifest_info(ctypes.c_void_p(man.ptr), per.ctypes.data, ctypes.byref(tot), ctypes.byref(touched),
                                ctypes.byref(dig))
    if check:
        _check(rc)
    return dict(realized=per, realized_total=tot.value, touched=touched.value, digest=dig.value, status=rc)


def mp_manifest_lineage(man: Handle, K: int):
    """the K + 1 lineage ids recorded in the manifest (zeros when none were given)"""
    ids = np.zeros(K + 1, np.uint64)
    _check(lib().mp_manifest_lineage(ctypes.c_void_p(man.ptr), ids.ctypes.data))
    return ids


def mp_budget_from_fraction(fam: Family, f: float) -> int:
    return int(lib().mp_budget_from_fraction(fam.ref(), float(f)))


def mp_last_error() -> str:
    return lib().mp_last_error().decode()


def mp_version() -> str:
    return lib().mp_version().decode()


def mp_kernel_launch_count() -> int:
    return int(lib().mp_kernel_launch_count())


def mp_debug_inject_fault(kind: int, n: int) -> None:
    """Test hook: the n-th device allocation (MP_FAULT_ALLOC) or host-pool gather launch
    (MP_FAULT_GATHER) from now on fails once, on the host; n = 0 disarms."""
    _check(lib().mp_debug_inject_fault(int(kind), int(n)))


def mp_debug_stall_pipeline(rounds: int) -> None:
    """Test hook: index and merge kernels launched from now on never arm their first ring
    slot and give up a pipeline wait after `rounds` polling rounds (0 = off)."""
    lib().mp_debug_stall_pipeline(int(rounds))


def mp_trace_start(capacity: int = 4096) -> None:
    """Record the device time of the calls from now on (at most `capacity` ranges)."""
    _check(lib().mp_trace_start(int(capacity)))


def mp_trace_stop() -> list:
    """Stop recording; the ranges as dicts (kind, segment, stream, t0_ms, t1_ms) in the
    order they were enqueued, times in ms from the earliest start."""
    n = ctypes.c_uint64(0)
    _check(lib().mp_trace_stop(ctypes.byref(n)))
    arr = (_TraceRange * max(1, n.value))()
    _check(lib().mp_trace_read(arr, n.value))
    return [{"kind": r.kind, "segment": r.segment, "stream": r.stream, "t0_ms": r.t0_ms, "t1_ms": r.t1_ms}
            for r in arr[:n.value]]


def mp_plan_noalloc(K, n_blocks, n_groups, dtype, blk_len, blk_group, norm, maxabs, nnz, tau, index_err, op: Op,
                    budget_bytes, mask, order, summary, stream=None):
    """The plan without any allocation: every argument is a caller device buffer (torch
    tensors or raw pointers; blk_group and tau may be None).  For callers that must not
    allocate; the planner's scratch is a fixed 16 MiB device array inside the library."""
    L = lib()
    if not getattr(L, "_noalloc_typed", False):
        vp = ctypes.c_void_p
        L.mp_plan_noalloc.restype = ctypes.c_int32
        L.mp_plan_noalloc.argtypes = [ctypes.c_uint32, ctypes.c_uint64, ctypes.c_uint32, ctypes.c_int, vp, vp, vp,
                                      vp, vp, vp, vp, vp, ctypes.c_uint64, vp, vp, vp, vp]
        L._noalloc_typed = True
    opt = lambda t: None if t is None else ctypes.c_void_p(_ptr(t))  # noqa: E731
    _check(L.mp_plan_noalloc(K, n_blocks, n_groups, dtype, opt(blk_len), opt(blk_group), opt(norm), opt(maxabs),
                             opt(nnz), opt(tau), opt(index_err), op.ref(), int(budget_bytes), opt(mask), opt(order),
                             opt(summary), ctypes.c_void_p(_stream_ptr(stream))))
