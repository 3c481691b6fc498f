"""Catalog block hashes and Alg. 2's hash validation on the GPU, through the C ABI,
against the oracle's hash (bit for bit).

* mp_index_hashes: every base and expert block hash equals the oracle's, for bf16 and fp32
  families with ragged tails, K = 9 and an expert pool in pinned host memory.
* mp_manifest_validate after a merge: every block read is checked (the base and exactly
  the selected expert blocks) with no mismatch, and the output's block hashes equal the
  oracle's hashes of the oracle's merged checkpoint.
* A selected expert block changed after indexing is reported (the first mismatch named);
  a change to a block the plan did not select is not read, so it is not seen.
* Hashes survive export and import; an index without hashes cannot validate.
"""
import numpy as np
import pytest
import torch

import oracle
from conftest import oracle_family
from test_gpu_parity import fam_k9, fam_ragged_bf16, fam_ragged_f32, host, ops_for, upload

pytestmark = pytest.mark.gpu

import paper_2605_29489_gb300 as mp  # noqa: E402
from paper_2605_29489_gb300 import synth  # noqa: E402


def catalog(fam, base, experts, host_experts=False):
    mf, b, ex = upload(fam, base, experts, host_experts)
    gop = mp.make_op(mp.MP_OP_TA, alpha=[0.3] * fam.K)
    idx = mp.mp_index_blocks(mf, gop)
    mp.mp_index_hashes(mf, idx)
    return mf, b, ex, gop, idx


@pytest.mark.parametrize("make,host_experts", [(fam_ragged_bf16, False), (fam_ragged_f32, False), (fam_k9, False),
                                                (fam_k9, True)], ids=["ragged-bf16", "ragged-f32", "k9", "k9-host"])
def test_catalog_hashes_match_oracle(make, host_experts):
    fam = make()
    base, experts = fam.host_arrays()
    mf, b, ex, gop, idx = catalog(fam, base, experts, host_experts)
    bh, eh = mp.mp_index_hash_values(idx)
    obh, oeh = oracle.index_hashes(oracle_family(fam, base, experts))
    assert np.array_equal(bh, obh)
    assert np.array_equal(eh, oeh)
    idx.free()


def test_validate_after_merge_checks_what_was_read_and_hashes_the_output():
    fam = fam_ragged_bf16()
    base, experts = fam.host_arrays()
    mf, b, ex, _, idx = catalog(fam, base, experts)
    of = oracle_family(fam, base, experts)
    o_norm, o_max, o_nnz = oracle.index(of)
    bo, bl, bt = fam.block_table()
    for name, gop, oop in ops_for(fam.K, ("ta", "ties", "dare")):
        if oop.kind == oracle.TIES:
            idx_t = mp.mp_index_blocks(mf, gop)
            mp.mp_index_hashes(mf, idx_t)
            use, tau = idx_t, oracle.ties_thresholds(of, oop.density)
        else:
            use, tau = idx, None
        for f in (0.3, 1.0):
            B = mp.mp_budget_from_fraction(mf, f)
            plan = mp.mp_plan(use, gop, B)
            pi = mp.mp_plan_info(plan, use)
            opl = oracle.plan(fam.K, bl, of.blk_group, of.n_groups, fam.elem_size, oop, o_norm, o_max, o_nnz, tau, B)
            assert pi["digest"] == opl["digest"] and np.array_equal(pi["mask"], opl["mask"]), (name, f)
            out = torch.empty_like(b)
            man = mp.mp_merge(mf, use, plan, out)
            mp.mp_manifest_validate(mf, use, plan, out, man)
            v = mp.mp_manifest_validation(man, fam.n_blocks)
            n_sel_blocks = int(sum(bin(int(m)).count("1") for m in opl["mask"]))
            assert v["mismatched"] == 0
            assert v["checked"] == fam.n_blocks + n_sel_blocks, (name, f)
            want = oracle.merge(of, oop, tau=tau, mask=opl["mask"])
            for blk in range(fam.n_blocks):
                s = slice(int(bo[blk]), int(bo[blk] + bl[blk]))
                assert int(v["out_hash"][blk]) == oracle.block_hash(want[s].tobytes()), (name, f, blk)
            man.free()
            plan.free()
        if use is not idx:
            use.free()
    idx.free()


def test_validate_reports_a_changed_selected_block_only():
    fam = fam_ragged_bf16()
    base, experts = fam.host_arrays()
    mf, b, ex, gop, idx = catalog(fam, base, experts)
    plan = mp.mp_plan(idx, gop, mp.mp_budget_from_fraction(mf, 0.3))
    mask = mp.mp_plan_info(plan, idx)["mask"]
    bo, bl, _ = fam.block_table()
    sel = [(blk, i) for blk in range(fam.n_blocks) for i in range(fam.K) if (int(mask[blk]) >> i) & 1]
    uns = [(blk, i) for blk in range(fam.n_blocks) for i in range(fam.K) if not (int(mask[blk]) >> i) & 1]
    assert sel and uns
    # a block the plan did not select changes: the merge never reads it, nothing is seen
    blk, i = uns[0]
    ex[i].view(torch.int16)[int(bo[blk]) + 1] += 1
    out = torch.empty_like(b)
    man = mp.mp_merge(mf, idx, plan, out)
    mp.mp_manifest_validate(mf, idx, plan, out, man)
    assert mp.mp_manifest_validation(man, fam.n_blocks)["mismatched"] == 0
    man.free()
    # a selected block changes: reported, with the first mismatching block named
    blk, i = sel[len(sel) // 2]
    ex[i].view(torch.int16)[int(bo[blk] + bl[blk]) - 1] ^= 1
    man = mp.mp_merge(mf, idx, plan, out)
    mp.mp_manifest_validate(mf, idx, plan, out, man)
    v = mp.mp_manifest_validation(man, fam.n_blocks, check=False)
    assert v["mismatched"] == 1 and v["status"] == -8
    assert f"expert {i} block {blk}" in v["error"]
    with pytest.raises(mp.MergePipeError):
        mp.mp_manifest_validation(man, fam.n_blocks)
    for h in (man, plan, idx):
        h.free()


def test_hashes_survive_export_and_import_and_are_required():
    fam = fam_k9()
    base, experts = fam.host_arrays()
    mf, b, ex, gop, idx = catalog(fam, base, experts)
    norm, maxabs, nnz, _ = mp.mp_index_stats(idx)
    bh, eh = mp.mp_index_hash_values(idx)
    imp = mp.mp_index_import(mf, gop, norm, maxabs, nnz, base_hash=bh, expert_hash=eh)
    plan = mp.mp_plan(imp, gop, mp.mp_budget_from_fraction(mf, 0.5))
    out = torch.empty_like(b)
    man = mp.mp_merge(mf, imp, plan, out)
    mp.mp_manifest_validate(mf, imp, plan, out, man)
    assert mp.mp_manifest_validation(man, fam.n_blocks)["mismatched"] == 0
    bare = mp.mp_index_import(mf, gop, norm, maxabs, nnz)
    p2 = mp.mp_plan(bare, gop, mp.mp_budget_from_fraction(mf, 0.5))
    m2 = mp.mp_merge(mf, bare, p2, out)
    with pytest.raises(mp.MergePipeError):
        mp.mp_manifest_validate(mf, bare, p2, out, m2)
    for h in (m2, p2, bare, man, plan, imp, idx):
        h.free()
