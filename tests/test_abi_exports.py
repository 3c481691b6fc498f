"""The C-ABI library builds, loads without a GPU and exports every entry point that
include/*.h declares (no compute calls: those need a GPU)."""
import ctypes
import glob
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        src = open(h).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        for m in re.finditer(r"^\s*(?:mp_status|void|uint64_t|const char\s*\*)\s*\**\s*(mp_\w+)\s*\(", src, re.M):
            names.add(m.group(1))
    return sorted(names)


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ["mp_index_blocks", "mp_plan", "mp_merge", "mp_free"]:
        assert required in names
    assert len(names) >= 10


def test_library_exports_every_declared_symbol():
    import paper_2605_29489_gb300 as mp

    L = ctypes.CDLL(mp.library_path())
    missing = [n for n in declared_functions() if not hasattr(L, n)]
    assert not missing, missing


def test_binding_names_match_the_abi():
    import paper_2605_29489_gb300 as mp

    for n in ["mp_index_blocks", "mp_plan", "mp_merge", "mp_free", "mp_index_stats", "mp_plan_info",
              "mp_manifest_info", "mp_budget_from_fraction", "mp_last_error"]:
        assert callable(getattr(mp, n))


def test_version_and_error_without_gpu():
    import paper_2605_29489_gb300 as mp

    assert "sm_103a" in mp.mp_version()
    assert isinstance(mp.mp_last_error(), str)


def test_budget_from_fraction_host_only():
    """C_full = K * params * element size; B = floor(f * C_full) (host arithmetic only)"""
    import numpy as np
    import paper_2605_29489_gb300 as mp

    base = np.zeros(4096 + 300, np.uint16)
    experts = [np.zeros_like(base) for _ in range(3)]
    fam = mp.family([(0, 4096), (4096, 300)], base, experts, block_elems=1024, dtype=mp.MP_BF16, experts_location=0)
    full = 3 * (4096 + 300) * 2
    assert mp.mp_budget_from_fraction(fam, 1.0) == full
    assert mp.mp_budget_from_fraction(fam, 0.5) == full // 2
    assert mp.mp_budget_from_fraction(fam, 0.1) == int(np.floor(0.1 * full))
    assert mp.mp_budget_from_fraction(fam, 0.0) == 0
    assert mp.mp_budget_from_fraction(fam, 2.0) == full


def test_index_import_refuses_bad_entries_before_any_device_work():
    """mp_index_import checks every entry on the host: an nnz above the block's length, a
    negative norm, or a TIES catalog without tau is refused before any CUDA call"""
    import numpy as np
    import paper_2605_29489_gb300 as mp

    base = np.zeros(4096 + 300, np.uint16)
    experts = [np.zeros_like(base) for _ in range(2)]
    fam = mp.family([(0, 4096), (4096, 300)], base, experts, block_elems=1024, dtype=mp.MP_BF16, experts_location=0)
    K, nb = 2, 5
    norm = np.ones((K, nb), np.float32)
    maxabs = np.ones((K, nb), np.float32)
    nnz = np.full((K, nb), 3, np.uint32)
    op = mp.make_op(mp.MP_OP_TA, alpha=[0.5, 0.5])
    bad = nnz.copy()
    bad[1, 4] = 301                      # the last block holds 300 elements
    with pytest.raises(mp.MergePipeError) as e:
        mp.mp_index_import(fam, op, norm, maxabs, bad, stream=0)
    assert e.value.status == -1
    neg = norm.copy()
    neg[0, 1] = -0.5
    with pytest.raises(mp.MergePipeError) as e:
        mp.mp_index_import(fam, op, neg, maxabs, nnz, stream=0)
    assert e.value.status == -1
    with pytest.raises(mp.MergePipeError) as e:
        mp.mp_index_import(fam, mp.make_op(mp.MP_OP_TIES, lam=1.0, density=0.2), norm, maxabs, nnz, None, stream=0)
    assert e.value.status == -1
    # a TIES-after-masking catalog carries per-block key histograms, which are not imported
    with pytest.raises(mp.MergePipeError) as e:
        mp.mp_index_import(fam, mp.make_op(mp.MP_OP_TIES_MASKED, lam=1.0, density=0.2), norm, maxabs, nnz, stream=0)
    assert e.value.status == -7


def test_plan_noalloc_refuses_bad_arguments_before_any_device_work():
    """mp_plan_noalloc checks its arguments on the host before any CUDA call: a NULL or
    misaligned buffer, too many units or a TIES plan without thresholds is refused (the
    addresses here are never dereferenced)"""
    import paper_2605_29489_gb300 as mp

    A = 0x100000  # an aligned address, never touched
    op = mp.make_op(mp.MP_OP_TA, alpha=[0.5, 0.5])

    def call(K=2, n_blocks=8, op=op, tau=None, blk_group=None, **bufs):
        b = dict(blk_len=A, norm=A, maxabs=A, nnz=A, index_err=A, mask=A, order=A, summary=A)
        b.update(bufs)
        with pytest.raises(mp.MergePipeError) as e:
            mp.mp_plan_noalloc(K, n_blocks, 1, mp.MP_BF16, b["blk_len"], blk_group, b["norm"], b["maxabs"],
                               b["nnz"], tau, b["index_err"], op, 1 << 20, b["mask"], b["order"], b["summary"],
                               stream=0)
        assert e.value.status == -1
        return str(e.value)

    assert "aligned" in call(norm=A + 2)
    assert "aligned" in call(order=A + 1)
    assert "aligned" in call(summary=A + 4)  # 8-byte words
    assert "aligned" in call(blk_group=A + 2)
    assert "NULL" in call(mask=None)
    assert "524288" in call(K=2, n_blocks=(1 << 18) + 1)
    assert "tau" in call(op=mp.make_op(mp.MP_OP_TIES, lam=1.0, density=0.2), blk_group=A)
    # the operator checks of mp_plan, with the same refusals
    nan = float("nan")
    assert "alpha must be finite" in call(op=mp.make_op(mp.MP_OP_TA, alpha=[0.5, nan]))
    assert "lambda must be finite" in call(op=mp.make_op(mp.MP_OP_TIES, lam=float("inf"), density=0.2), tau=A,
                                           blk_group=A)
    assert "alpha > 0" in call(op=mp.make_op(mp.MP_OP_AVG_RENORM, alpha=[0.5, 0.0]))
    assert "alpha > 0" in call(op=mp.make_op(mp.MP_OP_AVG_RENORM, alpha=[-0.5, 0.5]))
    assert "density" in call(op=mp.make_op(mp.MP_OP_TIES, lam=1.0, density=1.5), tau=A, blk_group=A)
    assert "trim_scope" in call(op=mp.make_op(mp.MP_OP_TIES, lam=1.0, density=0.2, trim_scope=2), tau=A, blk_group=A)
    assert "drop_p" in call(op=mp.make_op(mp.MP_OP_DARE, alpha=[0.5, 0.5], drop_p=1.5))
    assert "drop_p" in call(op=mp.make_op(mp.MP_OP_DARE_TIES, lam=1.0, drop_p=-0.1))


def test_fault_injection_hook_arms_and_refuses_unknown_kinds_without_gpu():
    """the host-side fault hook is plain host state: arming and disarming the two kinds
    succeeds, an unknown kind is refused (no CUDA call is made)"""
    import paper_2605_29489_gb300 as mp

    for kind in (mp.MP_FAULT_ALLOC, mp.MP_FAULT_GATHER):
        mp.mp_debug_inject_fault(kind, 3)
        mp.mp_debug_inject_fault(kind, 0)
    with pytest.raises(mp.MergePipeError) as e:
        mp.mp_debug_inject_fault(0, 1)
    assert e.value.status == -1
    mp.mp_debug_stall_pipeline(0)


def test_trace_refuses_bad_arguments_and_stops_empty_without_gpu():
    """the trace API checks its arguments on the host: capacity 0 or above 2^20 is refused,
    and a stop without a start holds no ranges (neither makes a CUDA call)"""
    import paper_2605_29489_gb300 as mp

    for cap in (0, (1 << 20) + 1):
        with pytest.raises(mp.MergePipeError) as e:
            mp.mp_trace_start(cap)
        assert e.value.status == -1
    assert mp.mp_trace_stop() == []
    with pytest.raises(mp.MergePipeError) as e:
        mp._check(mp.lib().mp_trace_read(None, 1))
    assert e.value.status == -1
