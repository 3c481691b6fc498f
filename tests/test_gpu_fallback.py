"""Imported catalogs and the tensor-level fallback plan (Sec. 3 "Catalog" and "Planner")
on the GPU, through the C ABI, against the oracle.

* The oracle's catalog imported with mp_index_import plans and merges exactly like the
  GPU's own index of the same family (which equals it bit for bit).
* Entries marked MP_NNZ_MISSING: the plan (mask, order, C_hat, counts, digest) equals the
  oracle's tensor-level fallback plan bit for bit, and the merge with that plan equals the
  oracle's merge with the same mask and the same catalog nnz.  Seeded missing patterns:
  sparse, dense, one whole tensor, every entry; tensors of one block and of more than 32
  blocks (several warp chunks of the ordered norm chain).
* mp_plan_noalloc, which has no tensor map, reports such entries and never reads them.
"""
import numpy as np
import pytest
import torch

import oracle
from conftest import oracle_family
from test_gpu_parity import assert_merge_close, fam_k9, fam_k32, fam_ragged_bf16, fam_ragged_f32, host, ops_for, \
    tensor_mask, upload

pytestmark = pytest.mark.gpu

import paper_2605_29489_gb300 as mp  # noqa: E402
from paper_2605_29489_gb300 import synth  # noqa: E402

MISS = mp.MP_NNZ_MISSING
KINDS = ("avg", "ta", "ties", "ties1", "dare", "ta_pb", "ties_pb", "avg_renorm", "dare_ties")
FRACS = [0.0, 0.05, 0.3, 0.7, 1.0]


def fam_many_blocks():
    # 256-element blocks: the first tensor has 157 blocks, the last 34
    return synth.custom([40000, 3000, 256 * 33 + 7, 100], dtype=synth.BF16, block_elems=256, K=4, active_frac=0.5,
                        per_expert_active=True, name="many-blocks")


def missing_patterns(fam, K, rng):
    _, _, bt = fam.block_table()
    nb = bt.size
    pats = {"none": np.zeros((K, nb), bool),
            "sparse": rng.random((K, nb)) < 0.05,
            "dense": rng.random((K, nb)) < 0.5,
            "all": np.ones((K, nb), bool)}
    whole = np.zeros((K, nb), bool)
    whole[:, bt == int(np.argmax(np.bincount(bt)))] = True       # the tensor with most blocks, every expert
    whole[K - 1, bt == bt[-1]] = True                             # and the last tensor of the last expert
    pats["whole-tensor"] = whole
    return pats


def run_fallback(fam, kinds=KINDS, fracs=FRACS, seed=0):
    base, experts = fam.host_arrays()
    mf, b, ex = upload(fam, base, experts)
    covered = tensor_mask(fam)
    bo, bl, bt = fam.block_table()
    es = fam.elem_size
    rng = np.random.default_rng(seed)
    pats = missing_patterns(fam, fam.K, rng)
    for name, gop, oop in ops_for(fam.K, kinds):
        scope = oop.trim_scope if oop.kind == oracle.TIES else 0
        of = oracle_family(fam, base, experts, trim_scope=scope)
        idx = mp.mp_index_blocks(mf, gop)
        norm, maxabs, nnz = oracle.index(of)       # the oracle's catalog, imported into the GPU
        o_tau = oracle.ties_thresholds(of, oop.density) if oop.kind == oracle.TIES else None
        for pname, miss in pats.items():
            nz = nnz.copy()
            nz[miss] = MISS
            nm = norm.copy()
            nm[miss] = np.float32(np.nan)      # ignored for missing entries
            imp = mp.mp_index_import(mf, gop, nm, maxabs, nz, o_tau)
            for f in fracs:
                B = mp.mp_budget_from_fraction(mf, f)
                what = f"{fam.name}/{name}/{pname}/f={f}"
                plan = mp.mp_plan(imp, gop, B)
                pi = mp.mp_plan_info(plan, imp)
                opl = oracle.plan(fam.K, bl, of.blk_group, of.n_groups, es, oop, nm, maxabs, nz, o_tau, B,
                                  blk_tensor=bt)
                assert pi["chat"] == opl["chat"] <= B, what
                assert pi["n_sel"] == opl["n_sel"], what
                assert pi["n_cand"] == opl["n_cand"], what
                assert np.array_equal(pi["mask"], opl["mask"]), what
                assert np.array_equal(pi["order"], opl["order"]), what
                assert pi["digest"] == opl["digest"], what
                if pname == "none":   # the imported catalog plans like the index it came from
                    p0 = mp.mp_plan(idx, gop, B)
                    assert mp.mp_plan_info(p0, idx)["digest"] == pi["digest"], what
                    p0.free()
                out = torch.full_like(b, float("nan"))
                man = mp.mp_merge(mf, imp, plan, out)
                mi = mp.mp_manifest_info(man, fam.K)
                assert mi["realized_total"] == opl["chat"], what
                assert mi["touched"] == int((opl["mask"] != 0).sum()), what
                want = oracle.merge(of, oop, tau=o_tau, mask=opl["mask"], nnz=nz)
                assert_merge_close(fam, host(fam, out)[covered], want[covered], what)
                man.free()
                plan.free()
            imp.free()
        idx.free()


@pytest.mark.parametrize("make", [fam_ragged_bf16, fam_ragged_f32, fam_k9, fam_k32, fam_many_blocks],
                         ids=lambda f: f.__name__)
def test_fallback_plan_and_merge_match_oracle(make):
    run_fallback(make())


def test_fallback_full_budget_reproduces_the_full_read():
    """Eq. 5 with missing entries: at B = C_full the merge equals the unmasked operator"""
    fam = fam_many_blocks()
    base, experts = fam.host_arrays()
    mf, b, ex = upload(fam, base, experts)
    covered = tensor_mask(fam)
    rng = np.random.default_rng(5)
    for name, gop, oop in ops_for(fam.K, ("ta", "ties", "avg_renorm")):
        of = oracle_family(fam, base, experts)
        idx = mp.mp_index_blocks(mf, gop)
        norm, maxabs, nnz = oracle.index(of)
        nz = nnz.copy()
        nz[rng.random(nz.shape) < 0.3] = MISS
        o_tau = oracle.ties_thresholds(of, oop.density) if oop.kind == oracle.TIES else None
        imp = mp.mp_index_import(mf, gop, norm, maxabs, nz, o_tau)
        plan = mp.mp_plan(imp, gop, mp.mp_budget_from_fraction(mf, 1.0))
        out = torch.empty_like(b)
        man = mp.mp_merge(mf, imp, plan, out)
        mp.mp_manifest_info(man, fam.K)
        phi = oracle.merge(of, oop, tau=o_tau)
        assert_merge_close(fam, host(fam, out)[covered], phi[covered], name)
        for h in (man, plan, imp, idx):
            h.free()


def test_noalloc_reports_missing_entries_and_skips_them():
    fam = fam_ragged_bf16()
    base, experts = fam.host_arrays()
    mf, b, ex = upload(fam, base, experts)
    _, bl, bt = fam.block_table()
    gop = mp.make_op(mp.MP_OP_TA, alpha=[0.3] * fam.K)
    oop = oracle.Op(oracle.TA, fam.K, alpha=[0.3] * fam.K)
    idx = mp.mp_index_blocks(mf, gop)
    norm, maxabs, nnz = oracle.index(oracle_family(fam, base, experts))
    nz = nnz.copy()
    nz[np.random.default_rng(3).random(nz.shape) < 0.2] = MISS
    K, nb = fam.K, bl.size
    d = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()  # noqa: E731
    mask = torch.zeros(nb, dtype=torch.int32, device="cuda")
    order = torch.zeros(K * nb, dtype=torch.int32, device="cuda")
    summary = torch.zeros(8, dtype=torch.int64, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    B = mp.mp_budget_from_fraction(mf, 0.4)
    mp.mp_plan_noalloc(K, nb, 1, fam.dtype, d(bl.astype(np.int32)), None, d(norm), d(maxabs),
                       d(nz.view(np.int32)), None, err, gop, B, mask, order, summary)
    torch.cuda.synchronize()
    s = summary.cpu().numpy().view(np.uint64)
    assert int(s[6]) & 8
    skipped = nz.copy()
    skipped[skipped == MISS] = 0       # never read: as if it held nothing
    opl = oracle.plan(K, bl, np.zeros(nb, np.uint32), 1, fam.elem_size, oop, norm, maxabs, skipped, None, B)
    assert np.array_equal(mask.cpu().numpy().view(np.uint32), opl["mask"])
    assert int(s[0]) == opl["chat"] and int(s[4]) == opl["digest"]
    idx.free()


def test_import_refuses_entries_that_are_not_statistics():
    fam = fam_ragged_bf16()
    base, experts = fam.host_arrays()
    mf, b, ex = upload(fam, base, experts)
    gop = mp.make_op(mp.MP_OP_TA, alpha=[0.3] * fam.K)
    idx = mp.mp_index_blocks(mf, gop)
    norm, maxabs, nnz, _ = mp.mp_index_stats(idx)
    _, bl, _ = fam.block_table()
    bad = nnz.copy()
    bad[1, 2] = bl[2] + 1
    with pytest.raises(mp.MergePipeError):
        mp.mp_index_import(mf, gop, norm, maxabs, bad)
    neg = norm.copy()
    neg[0, 0] = -1.0
    with pytest.raises(mp.MergePipeError):
        mp.mp_index_import(mf, gop, neg, maxabs, nnz)
    ties = mp.make_op(mp.MP_OP_TIES, lam=1.0, density=0.2)
    with pytest.raises(mp.MergePipeError):
        mp.mp_index_import(mf, ties, norm, maxabs, nnz, None)
    idx.free()


def test_fallback_with_a_host_resident_pool():
    """an imported catalog with missing entries plans and merges the same when the experts
    live in pinned host memory (the segment pipeline gathers the planned blocks)"""
    fam = fam_k9()
    base, experts = fam.host_arrays()
    mf_d, b_d, _ = upload(fam, base, experts)
    mf_h, b_h, _ = upload(fam, base, experts, host_experts=True)
    covered = tensor_mask(fam)
    _, bl, bt = fam.block_table()
    of = oracle_family(fam, base, experts)
    for name, gop, oop in ops_for(fam.K, ("ta", "avg_renorm")):
        idx = mp.mp_index_blocks(mf_d, gop)
        norm, maxabs, nnz = oracle.index(of)
        nz = nnz.copy()
        nz[missing_patterns(fam, fam.K, np.random.default_rng(9))["dense"]] = MISS
        imp_h = mp.mp_index_import(mf_h, gop, norm, maxabs, nz)
        for f in (0.3, 1.0):
            B = mp.mp_budget_from_fraction(mf_h, f)
            plan = mp.mp_plan(imp_h, gop, B)
            pi = mp.mp_plan_info(plan, imp_h)
            opl = oracle.plan(fam.K, bl, of.blk_group, of.n_groups, fam.elem_size, oop, norm, maxabs, nz, None, B,
                              blk_tensor=bt)
            assert pi["digest"] == opl["digest"] and np.array_equal(pi["mask"], opl["mask"]), (name, f)
            out = torch.full_like(b_h, float("nan"))
            man = mp.mp_merge(mf_h, imp_h, plan, out)
            assert mp.mp_manifest_info(man, fam.K)["realized_total"] == opl["chat"]
            want = oracle.merge(of, oop, mask=opl["mask"], nnz=nz)
            assert_merge_close(fam, host(fam, out)[covered], want[covered], f"{name}/host/f={f}")
            man.free()
            plan.free()
        imp_h.free()
        idx.free()


def test_fallback_plan_with_touched_only_merge():
    """a fallback plan merged with mp_merge_touched: touched blocks (whole fallback tensors
    among them) equal the oracle's merge, every other byte keeps the sentinel"""
    fam = fam_many_blocks()
    base, experts = fam.host_arrays()
    mf, b, ex = upload(fam, base, experts)
    bo, bl, bt = fam.block_table()
    of = oracle_family(fam, base, experts)
    norm, maxabs, nnz = oracle.index(of)
    nz = nnz.copy()
    nz[missing_patterns(fam, fam.K, np.random.default_rng(11))["whole-tensor"]] = MISS
    gop = mp.make_op(mp.MP_OP_TA, alpha=[0.3] * fam.K)
    oop = oracle.Op(oracle.TA, fam.K, alpha=[0.3] * fam.K)
    imp = mp.mp_index_import(mf, gop, norm, maxabs, nz)
    for f in (0.2, 0.6):
        B = mp.mp_budget_from_fraction(mf, f)
        plan = mp.mp_plan(imp, gop, B)
        opl = oracle.plan(fam.K, bl, of.blk_group, of.n_groups, fam.elem_size, oop, norm, maxabs, nz, None, B,
                          blk_tensor=bt)
        assert np.array_equal(mp.mp_plan_info(plan, imp)["mask"], opl["mask"]), f
        out = torch.empty_like(b)
        out.view(torch.uint8).fill_(0x5A)
        man = mp.mp_merge_touched(mf, imp, plan, out)
        assert mp.mp_manifest_info(man, fam.K)["touched"] == int((opl["mask"] != 0).sum())
        got = host(fam, out)
        want = oracle.merge(of, oop, mask=opl["mask"])
        touched = np.zeros(got.size, bool)
        for blk in np.nonzero(opl["mask"])[0].tolist():
            touched[int(bo[blk]):int(bo[blk] + bl[blk])] = True
        assert_merge_close(fam, got[touched], want[touched], f"touched/f={f}")
        assert bool((got[~touched].view(np.uint8) == 0x5A).all())
        man.free()
        plan.free()
    imp.free()
