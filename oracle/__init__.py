"""CPU oracle for the budgeted, mask-aware merge — TEST INFRASTRUCTURE ONLY.

A ctypes binding over ``oracle.c`` (plain single-threaded C).  Only the tests,
``__graft_entry__.smoke()`` and the benchmark's CPU-baseline leg may import this
module; the product path (``paper_2605_29489_gb300``) never does, and this module
imports nothing from it.  All arrays are numpy; bf16 data is passed as uint16 bit
patterns.  Per-unit arrays are expert-major ``[K, n_blocks]``.
"""
from __future__ import annotations

import ctypes
import os
import struct

import numpy as np

from . import build as _build

BF16, F32 = 0, 1
AVG, TA, TIES, DARE, AVG_RENORM, DARE_TIES, TIES_MASKED = 0, 1, 2, 3, 4, 5, 6
OK, EINVAL, EOOM, ENONFINITE = 0, -1, -3, -4
TAU_NONE = 0x8000
NNZ_MISSING = 0xFFFFFFFF  # catalog entry without block statistics (tensor-level fallback)

_lib = None

# The mutation check of the pins (tests/test_oracle_mutants.py) builds copies of oracle.c
# with one planted mistake each and runs the pins in a child process whose oracle is
# such a copy: the child names that library here.  Unset, the oracle is oracle.c built.
LIBRARY_UNDER_TEST_ENV = "ORACLE_LIBRARY_UNDER_TEST"


class _Op(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int), ("K", ctypes.c_uint32), ("alpha", ctypes.c_void_p),
                ("lambda_", ctypes.c_float), ("density", ctypes.c_float), ("trim_scope", ctypes.c_uint32),
                ("drop_p", ctypes.c_double), ("seed", ctypes.c_uint64), ("score_mode", ctypes.c_uint32)]


class _Family(ctypes.Structure):
    _fields_ = [("dtype", ctypes.c_int), ("K", ctypes.c_uint32), ("n_blocks", ctypes.c_uint64),
                ("blk_off", ctypes.c_void_p), ("blk_len", ctypes.c_void_p), ("blk_group", ctypes.c_void_p),
                ("n_groups", ctypes.c_uint32), ("base", ctypes.c_void_p), ("experts", ctypes.c_void_p)]


def lib():
    global _lib
    if _lib is None:
        L = ctypes.CDLL(os.environ.get(LIBRARY_UNDER_TEST_ENV) or _build.build())
        vp, u32, u64 = ctypes.c_void_p, ctypes.c_uint32, ctypes.c_uint64
        L.orc_bf16_to_f32.restype = ctypes.c_float
        L.orc_bf16_to_f32.argtypes = [ctypes.c_uint16]
        L.orc_f32_to_bf16.restype = ctypes.c_uint16
        L.orc_f32_to_bf16.argtypes = [ctypes.c_float]
        L.orc_ties_key.restype = u32
        L.orc_ties_key.argtypes = [ctypes.c_float]
        L.orc_block_stats.argtypes = [ctypes.c_int, u64, vp, vp, vp, vp, vp, vp]
        L.orc_index.argtypes = [vp, vp, vp, vp]
        L.orc_key_hist.argtypes = [ctypes.c_int, u64, vp, vp, vp]
        L.orc_tau_from_hist.restype = u32
        L.orc_tau_from_hist.argtypes = [vp, u64, ctypes.c_float]
        L.orc_ties_thresholds.argtypes = [vp, ctypes.c_float, vp]
        L.orc_ties_masked_thresholds.argtypes = [vp, ctypes.c_float, vp, vp]
        L.orc_plan.argtypes = [u32, u64, vp, vp, u32, u32, vp, vp, vp, vp, vp, u64, vp, vp, vp, vp, vp, vp, vp, vp, u32]
        L.orc_merge_block.argtypes = [ctypes.c_int, u64, u64, vp, vp, u32, u32, vp, vp, vp]
        L.orc_merge.argtypes = [vp, vp, vp, vp, vp, vp]
        L.orc_philox4x32_10.argtypes = [vp, vp, vp]
        L.orc_dare_keep.argtypes = [u64, u32, u64, ctypes.c_double]
        L.orc_fnv1a64.restype = u64
        L.orc_fnv1a64.argtypes = [vp, ctypes.c_size_t]
        L.orc_splitmix64.restype = u64
        L.orc_splitmix64.argtypes = [u64]
        for nm in ("orc_block_hash", "orc_block_hash_sum"):
            getattr(L, nm).restype = u64
            getattr(L, nm).argtypes = [vp, u64]
        L.orc_index_hashes.argtypes = [vp, vp, vp]
        _lib = L
    return _lib


def _p(a):
    return None if a is None else ctypes.c_void_p(a.ctypes.data)


def _np_dtype(dtype):
    return np.uint16 if dtype == BF16 else np.float32


def _check(rc):
    if rc != OK:
        raise OracleError(rc)


class OracleError(RuntimeError):
    def __init__(self, rc):
        super().__init__(f"oracle status {rc}")
        self.rc = rc


class Op:
    """Merge operator and parameters (mirrors the oracle's orc_op)."""

    def __init__(self, kind, K, alpha=None, lam=1.0, density=0.2, trim_scope=0, drop_p=0.0, seed=0, score_mode=0):
        self.kind, self.K = kind, K
        self.alpha = None if alpha is None else np.ascontiguousarray(np.asarray(alpha, np.float32))
        self.lam, self.density, self.trim_scope = float(lam), float(density), int(trim_scope)
        self.drop_p, self.seed, self.score_mode = float(drop_p), int(seed), int(score_mode)

    def c(self):
        return _Op(self.kind, self.K, None if self.alpha is None else self.alpha.ctypes.data,
                   self.lam, self.density, self.trim_scope, self.drop_p, self.seed, self.score_mode)


class Family:
    """Block geometry plus numpy data for a whole family (small cases)."""

    def __init__(self, dtype, blk_off, blk_len, blk_group, n_groups, base, experts):
        self.dtype = dtype
        self.blk_off = np.ascontiguousarray(blk_off, np.uint64)
        self.blk_len = np.ascontiguousarray(blk_len, np.uint32)
        self.blk_group = np.ascontiguousarray(blk_group, np.uint32)
        self.n_groups = int(n_groups)
        self.base = np.ascontiguousarray(base)
        self.experts = [np.ascontiguousarray(e) for e in experts]
        self.K = len(experts)
        self._ptrs = (ctypes.c_void_p * self.K)(*[e.ctypes.data for e in self.experts])

    @property
    def n_blocks(self):
        return int(self.blk_off.shape[0])

    def c(self):
        return _Family(self.dtype, self.K, self.n_blocks, self.blk_off.ctypes.data, self.blk_len.ctypes.data,
                       self.blk_group.ctypes.data, self.n_groups, self.base.ctypes.data,
                       ctypes.cast(self._ptrs, ctypes.c_void_p).value)


# ---- element helpers ------------------------------------------------------------------------

def bf16_bits(x: float) -> int:
    return int(lib().orc_f32_to_bf16(ctypes.c_float(x)))


def bf16_value(h: int) -> float:
    return float(lib().orc_bf16_to_f32(ctypes.c_uint16(h)))


def ties_key(d: float) -> int:
    return int(lib().orc_ties_key(ctypes.c_float(d)))


# ---- index ------------------------------------------------------------------------------------

def block_stats(dtype, base, expert):
    """(norm, maxabs, nnz, ss_f64) of one block; raises OracleError on non-finite deltas"""
    base = np.ascontiguousarray(base, _np_dtype(dtype))
    expert = np.ascontiguousarray(expert, _np_dtype(dtype))
    nrm, mx = ctypes.c_float(), ctypes.c_float()
    nz, ss = ctypes.c_uint32(), ctypes.c_double()
    _check(lib().orc_block_stats(dtype, base.shape[0], _p(base), _p(expert), ctypes.byref(nrm),
                                 ctypes.byref(mx), ctypes.byref(nz), ctypes.byref(ss)))
    return nrm.value, mx.value, nz.value, ss.value


def index(fam: Family):
    K, nb = fam.K, fam.n_blocks
    norm = np.zeros((K, nb), np.float32)
    maxabs = np.zeros((K, nb), np.float32)
    nnz = np.zeros((K, nb), np.uint32)
    c = fam.c()
    _check(lib().orc_index(ctypes.byref(c), _p(norm), _p(maxabs), _p(nnz)))
    return norm, maxabs, nnz


def key_hist(dtype, base, expert, hist=None):
    hist = np.zeros(32768, np.uint64) if hist is None else hist
    base = np.ascontiguousarray(base, _np_dtype(dtype))
    expert = np.ascontiguousarray(expert, _np_dtype(dtype))
    _check(lib().orc_key_hist(dtype, base.shape[0], _p(base), _p(expert), _p(hist)))
    return hist


def tau_from_hist(hist, numel, density):
    hist = np.ascontiguousarray(hist, np.uint64)
    return int(lib().orc_tau_from_hist(_p(hist), int(numel), ctypes.c_float(density)))


def ties_thresholds(fam: Family, density):
    tau = np.zeros((fam.K, fam.n_groups), np.uint32)
    c = fam.c()
    _check(lib().orc_ties_thresholds(ctypes.byref(c), ctypes.c_float(density), _p(tau)))
    return tau


def ties_masked_thresholds(fam: Family, density, mask):
    """TIES after masking: thresholds of the zero-completed masked deltas [K, n_groups]"""
    tau = np.zeros((fam.K, fam.n_groups), np.uint32)
    m = np.ascontiguousarray(mask, np.uint32)
    c = fam.c()
    _check(lib().orc_ties_masked_thresholds(ctypes.byref(c), ctypes.c_float(density), _p(m), _p(tau)))
    return tau


# ---- plan -------------------------------------------------------------------------------------

def plan(K, blk_len, blk_group, n_groups, elem_size, op: Op, norm, maxabs, nnz, tau, budget, blk_tensor=None):
    """Alg. 1; blk_tensor (tensor id of each block) enables the tensor-level fallback for
    entries whose nnz is NNZ_MISSING"""
    blk_len = np.ascontiguousarray(blk_len, np.uint32)
    blk_group = np.ascontiguousarray(blk_group, np.uint32)
    nb = blk_len.shape[0]
    norm = np.ascontiguousarray(norm, np.float32)
    maxabs = np.ascontiguousarray(maxabs, np.float32)
    nnz = np.ascontiguousarray(nnz, np.uint32)
    tau = None if tau is None else np.ascontiguousarray(tau, np.uint32)
    mask = np.zeros(nb, np.uint32)
    order = np.zeros(nb * K, np.uint32)
    out = [ctypes.c_uint64() for _ in range(5)]
    oc = op.c()
    bt = None if blk_tensor is None else np.ascontiguousarray(blk_tensor, np.uint32)
    n_t = 0 if bt is None else (int(bt.max()) + 1 if bt.size else 0)
    _check(lib().orc_plan(K, nb, _p(blk_len), _p(blk_group), n_groups, elem_size, ctypes.byref(oc),
                          _p(norm), _p(maxabs), _p(nnz), _p(tau), int(budget), _p(mask),
                          *[ctypes.byref(o) for o in out], _p(order), _p(bt), n_t))
    chat, nsel, ncand, set_hash, digest = [o.value for o in out]
    return dict(mask=mask, chat=chat, n_sel=nsel, n_cand=ncand, set_hash=set_hash, digest=digest,
                order=order[:ncand].copy())


# ---- merge ------------------------------------------------------------------------------------

def merge_block(dtype, j0, base, experts, mask, op: Op, tau_k=None, known_zero=0):
    """Psi_op on one block: experts is a list of K arrays (entries for unselected experts may be None);
    known_zero: bits of the experts whose delta block is exactly zero (renormalised AVG only)"""
    npd = _np_dtype(dtype)
    base = np.ascontiguousarray(base, npd)
    keep = [None if e is None else np.ascontiguousarray(e, npd) for e in experts]
    ptrs = (ctypes.c_void_p * op.K)(*[None if e is None else e.ctypes.data for e in keep])
    out = np.empty_like(base)
    tk = None if tau_k is None else np.ascontiguousarray(tau_k, np.uint32)
    oc = op.c()
    _check(lib().orc_merge_block(dtype, base.shape[0], int(j0), _p(base), ptrs, int(mask), int(known_zero),
                                 ctypes.byref(oc),
                                 _p(tk), _p(out)))
    return out


def merge(fam: Family, op: Op, tau=None, mask=None, out=None, nnz=None):
    """Alg. 2; nnz: the catalog's nonzero counts [K][n_blocks] (known-zero deltas for the
    renormalised AVG), None to derive them from the data"""
    out = np.zeros_like(fam.base) if out is None else out
    tau = None if tau is None else np.ascontiguousarray(tau, np.uint32)
    mask = None if mask is None else np.ascontiguousarray(mask, np.uint32)
    nz = None if nnz is None else np.ascontiguousarray(nnz, np.uint32)
    c, oc = fam.c(), op.c()
    _check(lib().orc_merge(ctypes.byref(c), ctypes.byref(oc), _p(tau), _p(mask), _p(out), _p(nz)))
    return out


# ---- generators and hashes --------------------------------------------------------------------

def philox4x32_10(ctr, key):
    c = np.ascontiguousarray(ctr, np.uint32)
    k = np.ascontiguousarray(key, np.uint32)
    o = np.zeros(4, np.uint32)
    lib().orc_philox4x32_10(_p(c), _p(k), _p(o))
    return o


def dare_keep(seed, expert, j, p):
    return bool(lib().orc_dare_keep(int(seed), int(expert), int(j), float(p)))


def fnv1a64(data: bytes) -> int:
    buf = ctypes.create_string_buffer(data, len(data))
    return int(lib().orc_fnv1a64(ctypes.cast(buf, ctypes.c_void_p), len(data)))


def splitmix64(state: int) -> int:
    return int(lib().orc_splitmix64(state & 0xFFFFFFFFFFFFFFFF))


def block_hash(data: bytes) -> int:
    """the catalog's content hash of one block's bytes"""
    buf = ctypes.create_string_buffer(bytes(data), max(1, len(data)))
    return int(lib().orc_block_hash(ctypes.cast(buf, ctypes.c_void_p), len(data)))


def block_hash_sum(data: bytes) -> int:
    """the multilinear sum H of the block hash (before the final mix)"""
    buf = ctypes.create_string_buffer(bytes(data), max(1, len(data)))
    return int(lib().orc_block_hash_sum(ctypes.cast(buf, ctypes.c_void_p), len(data)))


def index_hashes(fam: Family):
    """(base_hash [n_blocks], expert_hash [K, n_blocks]) uint64"""
    bh = np.zeros(fam.n_blocks, np.uint64)
    eh = np.zeros((fam.K, fam.n_blocks), np.uint64)
    c = fam.c()
    _check(lib().orc_index_hashes(ctypes.byref(c), _p(bh), _p(eh)))
    return bh, eh


def f32_bits(x: float) -> int:
    return struct.unpack("<I", struct.pack("<f", x))[0]
