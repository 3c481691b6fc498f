"""The touched-only merge (mp_merge_touched; Alg. 2 with WriteBlockOrReference): a block
with at least one selected expert receives exactly the oracle's merged block; every other
block, and every element between tensors, keeps what the output held before the call.
Checked with a sentinel-filled output, in place (the output is the base itself), at a
zero budget (nothing is written) and with a host-resident expert pool."""
import numpy as np
import pytest
import torch

import oracle
from conftest import oracle_family
from test_gpu_parity import (assert_merge_close, fam_k9, fam_k32, fam_ragged_bf16, fam_ragged_f32, host, ops_for,
                             upload)

pytestmark = pytest.mark.gpu

import paper_2605_29489_gb300 as mp  # noqa: E402
from paper_2605_29489_gb300 import synth  # noqa: E402

SENTINEL = 0x5A


def touched_elements(fam, mask):
    """bool mask of the elements of blocks whose access mask is nonzero"""
    bo, bl, _ = fam.block_table()
    _, _, total = fam.layout()
    t = np.zeros(total, bool)
    for b in np.nonzero(mask)[0].tolist():
        t[int(bo[b]):int(bo[b] + bl[b])] = True
    return t


def sentinel_like(t):
    out = torch.empty_like(t)
    out.view(torch.uint8).fill_(SENTINEL)
    return out


def check_family(fam, kinds, fracs, host_experts=False):
    base, experts = fam.host_arrays()
    mf, b, ex = upload(fam, base, experts, host_experts)
    bo, bl, _ = fam.block_table()
    for name, gop, oop in ops_for(fam.K, kinds):
        masked = oop.kind == oracle.TIES_MASKED
        scope = oop.trim_scope if oop.kind in (oracle.TIES, oracle.TIES_MASKED) else 0
        of = oracle_family(fam, base, experts, trim_scope=scope)
        o_norm, o_max, o_nnz = oracle.index(of)
        tau = oracle.ties_thresholds(of, oop.density) if oop.kind == oracle.TIES else None
        idx = mp.mp_index_blocks(mf, gop)
        for f in fracs:
            B = mp.mp_budget_from_fraction(mf, f)
            plan = mp.mp_plan(idx, gop, B)
            pi = mp.mp_plan_info(plan, idx)
            what = f"{fam.name}/{name}/f={f}"
            opl = oracle.plan(fam.K, bl, of.blk_group, of.n_groups, fam.elem_size, oop, o_norm, o_max, o_nnz, tau, B)
            assert pi["digest"] == opl["digest"] and np.array_equal(pi["mask"], opl["mask"]), what
            touched = touched_elements(fam, opl["mask"])
            m_tau = oracle.ties_masked_thresholds(of, oop.density, opl["mask"]) if masked else tau
            want = oracle.merge(of, oop, tau=m_tau, mask=opl["mask"])

            out = sentinel_like(b)
            before = host(fam, out).copy()
            man = mp.mp_merge_touched(mf, idx, plan, out)
            mi = mp.mp_manifest_info(man, fam.K)
            assert mi["realized_total"] == opl["chat"] <= B, what
            assert mi["touched"] == int((opl["mask"] != 0).sum()), what
            got = host(fam, out)
            assert_merge_close(fam, got[touched], want[touched], what)
            assert np.array_equal(got[~touched].view(np.uint8), before[~touched].view(np.uint8)), what
            man.free()

            # in place: the output is the base buffer of a family over a copy of the base
            b2 = dev_copy(b)
            mf2 = mp.family(list(zip(*[x.tolist() for x in fam.layout()[:2]])), b2, ex, fam.block_elems, fam.dtype,
                            1 if host_experts else 0)
            man2 = mp.mp_merge_touched(mf2, idx, plan, b2)
            got2 = host(fam, b2)
            assert_merge_close(fam, got2[touched], want[touched], what + " in place")
            assert np.array_equal(got2[~touched].view(np.uint8), base[~touched].view(np.uint8)), what + " in place"
            man2.free()
            plan.free()
        idx.free()


def dev_copy(t):
    c = torch.empty_like(t)
    c.copy_(t)
    return c


@pytest.mark.parametrize("make", [fam_ragged_bf16, fam_ragged_f32, fam_k9, fam_k32], ids=lambda f: f.__name__)
def test_touched_only_matches_oracle_on_touched_blocks(make):
    check_family(make(), ("avg", "ta", "ties", "dare", "avg_renorm", "dare_ties", "ties_masked"), [0.1, 0.5, 1.0])


def test_touched_only_zero_budget_writes_nothing():
    fam = fam_ragged_bf16()
    base, experts = fam.host_arrays()
    mf, b, ex = upload(fam, base, experts)
    gop = mp.make_op(mp.MP_OP_AVG, alpha=[1.0 / fam.K] * fam.K)
    idx = mp.mp_index_blocks(mf, gop)
    plan = mp.mp_plan(idx, gop, 0)
    out = sentinel_like(b)
    man = mp.mp_merge_touched(mf, idx, plan, out)
    assert mp.mp_manifest_info(man, fam.K)["touched"] == 0
    assert bool((out.view(torch.uint8) == SENTINEL).all())
    for h in (man, plan, idx):
        h.free()


def test_touched_only_host_pool():
    check_family(fam_k9(), ("avg", "ties"), [0.25, 1.0], host_experts=True)


def test_touched_only_rejects_partial_overlap_with_base():
    fam = fam_ragged_bf16()
    base, experts = fam.host_arrays()
    mf, b, ex = upload(fam, base, experts)
    gop = mp.make_op(mp.MP_OP_AVG, alpha=[1.0 / fam.K] * fam.K)
    idx = mp.mp_index_blocks(mf, gop)
    plan = mp.mp_plan(idx, gop, mp.mp_budget_from_fraction(mf, 1.0))
    big = torch.empty(b.numel() + 64, dtype=b.dtype, device="cuda")
    big[8:8 + b.numel()].copy_(b)
    offs, nums, _ = fam.layout()
    mf_big = mp.family(list(zip(offs.tolist(), nums.tolist())), big[8:8 + b.numel()], ex, fam.block_elems,
                       fam.dtype, 0)
    with pytest.raises(mp.MergePipeError):
        mp.mp_merge_touched(mf_big, idx, plan, big[16:16 + b.numel()])
    for h in (plan, idx):
        h.free()
