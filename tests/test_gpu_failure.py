"""Failure paths, exercised without a GPU fault.

* A bounded device wait that runs out: with the test hook mp_debug_stall_pipeline the index
  and merge kernels never arm the first slot of their shared-memory rings and give up a
  pipeline wait after a few thousand polling rounds, so their consumers' wait for that slot
  runs out.  The kernels record the timeout and return (the waits that drain their own
  copies keep the full limit); the accessors report MP_ERR_TIMEOUT for the index, for a
  plan built on it and for the manifest of a merge.
* Failures made on the host (mp_debug_inject_fault): the n-th device allocation or the
  n-th host-pool gather launch fails; the call returns its error and produces no handle
  (Alg. 2: a run either publishes or leaves no visible state), and the next calls work.
After each case the same work without the hook gives the oracle's results again.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
from conftest import oracle_family
from test_gpu_parity import host, upload

pytestmark = pytest.mark.gpu

import paper_2605_29489_gb300 as mp  # noqa: E402
from paper_2605_29489_gb300 import synth  # noqa: E402

TIMEOUT, OOM, CUDA = -6, -3, -2
STALL_ROUNDS = 4096  # polling rounds before a stalled wait gives up


def _family(K=3):
    return synth.custom([70001, 4096, 300, 20000, 131072], dtype=synth.BF16, block_elems=4096, K=K,
                        active_frac=0.5, name="failure")


def _oracle_merge(fam, base, experts, oop, f):
    of = oracle_family(fam, base, experts)
    norm, maxabs, nnz = oracle.index(of)
    tau = oracle.ties_thresholds(of, oop.density) if oop.kind == oracle.TIES else None
    _, bl, bt = fam.block_table()
    full = fam.K * int(bl.sum()) * fam.elem_size
    pl = oracle.plan(fam.K, bl, bt, len(fam.tensors), fam.elem_size, oop, norm, maxabs, nnz, tau,
                     int(np.floor(f * full)))
    return oracle.merge(of, oop, tau=tau, mask=pl["mask"]), pl


def _covered(fam):
    offs, nums, _ = fam.layout()
    c = np.zeros(fam.total_elems, bool)
    for o, n in zip(offs.tolist(), nums.tolist()):
        c[o:o + n] = True
    return c


def _raw_call(fn, *args):
    """call a C entry point whose last argument is a handle out-pointer; returns (status, handle)"""
    out = ctypes.c_void_p(12345)
    rc = fn(*args, ctypes.byref(out))
    return rc, out.value


@pytest.fixture
def restore_hooks():
    yield
    mp.mp_debug_stall_pipeline(0)
    mp.mp_debug_inject_fault(mp.MP_FAULT_ALLOC, 0)
    mp.mp_debug_inject_fault(mp.MP_FAULT_GATHER, 0)


@pytest.mark.parametrize("kind", ["ta", "ties"])
def test_wait_that_runs_out_is_reported_as_timeout(kind, restore_hooks):
    fam = _family()
    base, experts = fam.host_arrays()
    mf, b, ex = upload(fam, base, experts)
    K = fam.K
    if kind == "ta":
        gop, oop = mp.make_op(mp.MP_OP_TA, alpha=[0.3] * K), oracle.Op(oracle.TA, K, alpha=[0.3] * K)
    else:
        gop, oop = mp.make_op(mp.MP_OP_TIES, density=0.2), oracle.Op(oracle.TIES, K, density=0.2)
    B = mp.mp_budget_from_fraction(mf, 0.5)
    want, opl = _oracle_merge(fam, base, experts, oop, 0.5)
    cov = _covered(fam)

    # the index kernel gives up: its statistics and every plan built on it report the timeout
    mp.mp_debug_stall_pipeline(STALL_ROUNDS)
    idx_bad = mp.mp_index_blocks(mf, gop)
    mp.mp_debug_stall_pipeline(0)
    with pytest.raises(mp.MergePipeError) as e:
        mp.mp_index_stats(idx_bad)
    assert e.value.status == TIMEOUT
    plan_bad = mp.mp_plan(idx_bad, gop, B)
    with pytest.raises(mp.MergePipeError) as e:
        mp.mp_plan_info(plan_bad, idx_bad)
    assert e.value.status == TIMEOUT
    plan_bad.free()
    idx_bad.free()

    # a merge whose waits give up: its manifest reports the timeout, and nothing else
    idx = mp.mp_index_blocks(mf, gop)
    plan = mp.mp_plan(idx, gop, B)
    out = torch.empty_like(b)
    mp.mp_debug_stall_pipeline(STALL_ROUNDS)
    man_bad = mp.mp_merge(mf, idx, plan, out)
    mp.mp_debug_stall_pipeline(0)
    with pytest.raises(mp.MergePipeError) as e:
        mp.mp_manifest_info(man_bad, K)
    assert e.value.status == TIMEOUT
    man_bad.free()

    # the context is intact: the same merge without the hook is the oracle's
    man = mp.mp_merge(mf, idx, plan, out)
    mi = mp.mp_manifest_info(man, K)
    pi = mp.mp_plan_info(plan, idx)
    assert pi["digest"] == opl["digest"] and mi["realized_total"] == pi["chat"] == opl["chat"]
    assert np.array_equal(host(fam, out)[cov], want[cov])
    for h in (man, plan, idx):
        h.free()


def test_injected_allocation_failures_leave_no_handle(restore_hooks):
    fam = _family()
    base, experts = fam.host_arrays()
    mf, b, ex = upload(fam, base, experts)
    K = fam.K
    gop = mp.make_op(mp.MP_OP_TA, alpha=[0.3] * K)
    L = mp.lib()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)

    # the index handle's allocation
    mp.mp_debug_inject_fault(mp.MP_FAULT_ALLOC, 1)
    rc, h = _raw_call(L.mp_index_blocks, mf.ref(), gop.ref(), stream)
    assert (rc, h) == (OOM, None)
    assert "injected" in mp.mp_last_error()
    idx = mp.mp_index_blocks(mf, gop)

    # the plan allocates its handle, then its scratch: fail the second
    B = mp.mp_budget_from_fraction(mf, 0.5)
    mp.mp_debug_inject_fault(mp.MP_FAULT_ALLOC, 2)
    rc, h = _raw_call(L.mp_plan, ctypes.c_void_p(idx.ptr), gop.ref(), ctypes.c_uint64(B), stream)
    assert (rc, h) == (OOM, None)
    plan = mp.mp_plan(idx, gop, B)

    # the manifest's allocation
    out = torch.zeros_like(b)
    mp.mp_debug_inject_fault(mp.MP_FAULT_ALLOC, 1)
    rc, h = _raw_call(L.mp_merge, mf.ref(), ctypes.c_void_p(idx.ptr), ctypes.c_void_p(plan.ptr),
                      ctypes.c_void_p(out.data_ptr()), stream)
    assert (rc, h) == (OOM, None)
    man = mp.mp_merge(mf, idx, plan, out)
    assert mp.mp_manifest_info(man, K)["realized_total"] == mp.mp_plan_info(plan, idx)["chat"]
    for x in (man, plan, idx):
        x.free()
    with pytest.raises(mp.MergePipeError) as e:
        mp.mp_debug_inject_fault(7, 1)
    assert e.value.status == -1


def test_injected_gather_failure_in_host_pool(restore_hooks):
    """experts in pinned host memory: the n-th gather launch of the index or of the merge is
    not made; the call returns MP_ERR_CUDA and no handle, and a retry gives the oracle's merge"""
    fam = synth.custom([300000, 4096, 777, 200000], dtype=synth.BF16, block_elems=4096, K=3, active_frac=0.5,
                       name="failure-pool")
    base, experts = fam.host_arrays()
    mf, b, ex = upload(fam, base, experts, host_experts=True)
    K = fam.K
    gop, oop = mp.make_op(mp.MP_OP_TA, alpha=[0.3] * K), oracle.Op(oracle.TA, K, alpha=[0.3] * K)
    L = mp.lib()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)

    mp.mp_debug_inject_fault(mp.MP_FAULT_GATHER, 1)
    rc, h = _raw_call(L.mp_index_blocks, mf.ref(), gop.ref(), stream)
    assert (rc, h) == (CUDA, None)
    assert "injected" in mp.mp_last_error()
    idx = mp.mp_index_blocks(mf, gop)
    B = mp.mp_budget_from_fraction(mf, 0.5)
    plan = mp.mp_plan(idx, gop, B)
    out = torch.zeros_like(b)
    mp.mp_debug_inject_fault(mp.MP_FAULT_GATHER, 1)
    rc, h = _raw_call(L.mp_merge, mf.ref(), ctypes.c_void_p(idx.ptr), ctypes.c_void_p(plan.ptr),
                      ctypes.c_void_p(out.data_ptr()), stream)
    assert (rc, h) == (CUDA, None)
    man = mp.mp_merge(mf, idx, plan, out)
    mi = mp.mp_manifest_info(man, K)
    want, opl = _oracle_merge(fam, base, experts, oop, 0.5)
    assert mi["realized_total"] == opl["chat"]
    cov = _covered(fam)
    assert np.array_equal(host(fam, out)[cov], want[cov])
    for x in (man, plan, idx):
        x.free()
