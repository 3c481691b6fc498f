"""Parity at the full workload sizes, in the configuration bench.py times.

For each full-size family the GPU runs index -> plan -> merge exactly as the
benchmark does.  The oracle recomputes, from blocks regenerated on the host by
the seeded generator (never from GPU data):
  * the statistics of every unit (bit-exact: nnz, maxabs bits, norm bits),
  * every TIES threshold (bit-exact),
  * the whole plan at every budget from its own statistics (mask, traversal
    order, C_hat, counts and digest bit-exact),
and the merged output of a sample of blocks (first and last blocks, partial
tensor tails, small tensors and random blocks) under its own mask, which must
match the GPU output bit for bit (the bar is one bf16 ulp).  Properties that
hold at any size are checked on the whole output: realized reads = planned
bytes <= B (Prop. 1), untouched blocks are copies of the base.
The oracle runs in a spawned process pool, one task per block range or tensor.
"""
import concurrent.futures as cf
import math
import multiprocessing as mpr
import os

import numpy as np
import pytest
import torch

import oracle
import oracle_workers as ow

pytestmark = pytest.mark.gpu

import paper_2605_29489_gb300 as mp  # noqa: E402
from paper_2605_29489_gb300 import synth  # noqa: E402

NPROC = min(16, os.cpu_count() or 4)


@pytest.fixture(scope="module")
def pool():
    ex = cf.ProcessPoolExecutor(max_workers=NPROC, mp_context=mpr.get_context("spawn"), initializer=ow.init_worker)
    yield ex
    ex.shutdown(cancel_futures=True)


_CATALOGS = {}  # the oracle's statistics of a family, kept for the later tests of this module


def oracle_catalog(pool, spec, fam, ties_density=None):
    """oracle statistics [K, n_blocks] (and tau [K, n_tensors] for TIES) of the whole family"""
    if (spec, ties_density) in _CATALOGS:
        return _CATALOGS[(spec, ties_density)]
    if ties_density is None:   # the statistics do not depend on the operator
        for (sp, _), cat in _CATALOGS.items():
            if sp == spec:
                return cat[:3] + (None,)
    _CATALOGS[(spec, ties_density)] = cat = _oracle_catalog(pool, spec, fam, ties_density)
    return cat


def _oracle_catalog(pool, spec, fam, ties_density=None):
    K, nb = fam.K, fam.n_blocks
    norm = np.zeros((K, nb), np.float32)
    maxabs = np.zeros((K, nb), np.float32)
    nnz = np.zeros((K, nb), np.uint32)
    tau = None
    if ties_density is None:
        chunks = np.array_split(np.arange(nb), max(1, nb // 256))
        futs = [pool.submit(ow.block_stats, spec, c) for c in chunks]
        for f in cf.as_completed(futs):
            blocks, n, m, z = f.result()
            norm[:, blocks], maxabs[:, blocks], nnz[:, blocks] = n, m, z
    else:
        _, bl, bt = fam.block_table()
        tau = np.zeros((K, len(fam.tensors)), np.uint32)
        order = np.argsort([-int(bl[bt == t].sum()) for t in range(len(fam.tensors))])
        futs = [pool.submit(ow.tensor_stats_and_tau, spec, int(t), ties_density) for t in order]
        for f in cf.as_completed(futs):
            t, blocks, n, m, z, tt = f.result()
            norm[:, blocks], maxabs[:, blocks], nnz[:, blocks] = n, m, z
            tau[:, t] = tt
    return norm, maxabs, nnz, tau


def sample_blocks(fam, n_random=12, seed=1):
    bo, bl, bt = fam.block_table()
    nb = fam.n_blocks
    tails = [int(np.nonzero(bt == t)[0][-1]) for t in range(len(fam.tensors))]
    partial = [b for b in tails if bl[b] < fam.block_elems]
    small = [b for b in tails if bl[b] < 4096]
    rng = np.random.default_rng(seed)
    picks = {0, nb - 1, nb // 2}
    picks.update(partial[:6])
    picks.update(small[:4])
    picks.update(int(x) for x in rng.choice(nb, n_random, replace=False))
    return sorted(picks)


def run_family(pool, spec, gop, oop, fracs, ties_density=None):
    fam = ow.family(spec)
    es = fam.elem_size
    # --- GPU, as the benchmark runs it ---
    base, experts = fam.device_arrays()
    offs, nums, _ = fam.layout()
    mf = mp.family(list(zip(offs.tolist(), nums.tolist())), base, experts, fam.block_elems, fam.dtype, 0)
    idx = mp.mp_index_blocks(mf, gop)
    g_norm, g_max, g_nnz, g_tau = mp.mp_index_stats(idx)
    # --- oracle catalog of the whole family ---
    o_norm, o_max, o_nnz, o_tau = oracle_catalog(pool, spec, fam, ties_density)
    assert np.array_equal(g_nnz, o_nnz)
    assert np.array_equal(g_max.view(np.uint32), o_max.view(np.uint32))
    assert np.array_equal(g_norm.view(np.uint32), o_norm.view(np.uint32))
    if ties_density is not None:
        assert np.array_equal(g_tau, o_tau)
    bo, bl, bt = fam.block_table()
    samples = sample_blocks(fam)
    C_full = fam.K * fam.n_params * es
    out = torch.empty_like(base)
    for f in fracs:
        B = mp.mp_budget_from_fraction(mf, f)
        assert B == math.floor(f * C_full)
        plan = mp.mp_plan(idx, gop, B)
        pi = mp.mp_plan_info(plan, idx)
        opl = oracle.plan(fam.K, bl, bt, len(fam.tensors), es, oop, o_norm, o_max, o_nnz, o_tau, B)
        assert (pi["chat"], pi["n_sel"], pi["n_cand"], pi["digest"]) == (opl["chat"], opl["n_sel"], opl["n_cand"],
                                                                         opl["digest"]), f
        assert np.array_equal(pi["mask"], opl["mask"]), f
        assert np.array_equal(pi["order"], opl["order"]), f
        man = mp.mp_merge(mf, idx, plan, out)
        mi = mp.mp_manifest_info(man, fam.K)
        assert mi["realized_total"] == opl["chat"] <= B                       # Prop. 1
        assert mi["touched"] == int((opl["mask"] != 0).sum())
        # untouched blocks are copies of the base (whole output, on the GPU)
        untouched = np.nonzero(opl["mask"] == 0)[0]
        if untouched.size:
            sel = torch.zeros(fam.total_elems, dtype=torch.bool)
            for b in untouched[:: max(1, untouched.size // 2000)]:
                sel[int(bo[b]):int(bo[b] + bl[b])] = True
            sel = sel.cuda()
            assert torch.equal(out.view(torch.int16)[sel], base.view(torch.int16)[sel]), f
        # sampled blocks against the oracle's merge under its own mask
        for b in samples:
            hb, hex_ = fam.block_host(b)
            s = slice(int(bo[b]), int(bo[b] + bl[b]))
            tau_k = None if o_tau is None else o_tau[:, bt[b]]
            m = int(opl["mask"][b])
            want = oracle.merge_block(fam.dtype, int(bo[b]), hb, hex_, m, oop, tau_k)
            got = out[s].view(torch.int16).cpu().numpy().view(np.uint16)
            assert np.array_equal(got, want), (f, b)
        man.free()
        plan.free()
    idx.free()
    del base, experts, out
    torch.cuda.empty_cache()


def test_fullsize_qwen05b_task_arithmetic(pool):
    """Qwen2.5-0.5B-shaped family, K=8, task arithmetic lambda=0.3, budgets 1.0/0.5/0.25/0.1"""
    K = 8
    run_family(pool, ("qwen25_05b", ()), mp.make_op(mp.MP_OP_TA, alpha=[0.3] * K),
               oracle.Op(oracle.TA, K, alpha=[0.3] * K), [1.0, 0.5, 0.25, 0.1])


def test_fullsize_qwen15b_dare(pool):
    """Qwen2.5-1.5B-shaped family, K=16 with per-expert active sets, DARE p=0.9 then AVG, budget 0.25"""
    K = 16
    a = [1.0 / K] * K
    run_family(pool, ("qwen25_15b", ()), mp.make_op(mp.MP_OP_DARE, alpha=a, drop_p=0.9, seed=20260),
               oracle.Op(oracle.DARE, K, alpha=a, drop_p=0.9, seed=20260), [0.25])


def test_fullsize_llama3_8b_ties(pool):
    """Llama-3-8B-shaped family, K=4, TIES density 0.2, budgets 1.0/0.5/0.25/0.1"""
    K = 4
    if torch.cuda.get_device_properties(0).total_memory < 120 * 2 ** 30:
        pytest.skip("needs about 100 GB of device memory")
    run_family(pool, ("llama3_8b", ()), mp.make_op(mp.MP_OP_TIES, lam=1.0, density=0.2),
               oracle.Op(oracle.TIES, K, lam=1.0, density=0.2), [1.0, 0.5, 0.25, 0.1], ties_density=0.2)


def test_fullsize_llama3_8b_fallback_plan(pool):
    """Llama-3-8B-shaped family, K=4, TA lambda=0.3, planned from the oracle's own catalog
    imported with the bench's missing entries (tensor-level fallback), budgets 1.0 / 0.5 /
    0.25 / 0.1: plan bit-exact against the oracle's fallback plan; realized = planned; the
    merge of sampled blocks (the fallback tensors' first and last blocks among them) equal
    to the oracle's under the same mask"""
    K = 4
    if torch.cuda.get_device_properties(0).total_memory < 120 * 2 ** 30:
        pytest.skip("needs about 100 GB of device memory")
    spec = ("llama3_8b", ())
    fam = ow.family(spec)
    es = fam.elem_size
    o_norm, o_max, o_nnz, _ = oracle_catalog(pool, spec, fam)
    miss = synth.missing_entries(fam, K)
    nz = o_nnz.copy()
    nz[miss] = mp.MP_NNZ_MISSING
    gop = mp.make_op(mp.MP_OP_TA, alpha=[0.3] * K)
    oop = oracle.Op(oracle.TA, K, alpha=[0.3] * K)
    base, experts = fam.device_arrays()
    offs, nums, _ = fam.layout()
    mf = mp.family(list(zip(offs.tolist(), nums.tolist())), base, experts, fam.block_elems, fam.dtype, 0)
    imp = mp.mp_index_import(mf, gop, o_norm, o_max, nz)
    bo, bl, bt = fam.block_table()
    big = int(np.argmax(np.bincount(bt)))
    big_blocks = np.nonzero(bt == big)[0]
    samples = sorted(set(sample_blocks(fam)) | {int(big_blocks[0]), int(big_blocks[-1])})
    out = torch.empty_like(base)
    for f in (1.0, 0.5, 0.25, 0.1):
        B = mp.mp_budget_from_fraction(mf, f)
        plan = mp.mp_plan(imp, gop, B)
        pi = mp.mp_plan_info(plan, imp)
        opl = oracle.plan(K, bl, bt, len(fam.tensors), es, oop, o_norm, o_max, nz, None, B, blk_tensor=bt)
        assert (pi["chat"], pi["n_sel"], pi["n_cand"], pi["digest"]) == (opl["chat"], opl["n_sel"], opl["n_cand"],
                                                                         opl["digest"]), f
        assert np.array_equal(pi["mask"], opl["mask"]), f
        assert np.array_equal(pi["order"], opl["order"]), f
        man = mp.mp_merge(mf, imp, plan, out)
        mi = mp.mp_manifest_info(man, K)
        assert mi["realized_total"] == opl["chat"] <= B
        for b in samples:
            hb, hex_ = fam.block_host(b)
            s = slice(int(bo[b]), int(bo[b] + bl[b]))
            want = oracle.merge_block(fam.dtype, int(bo[b]), hb, hex_, int(opl["mask"][b]), oop)
            got = out[s].view(torch.int16).cpu().numpy().view(np.uint16)
            assert np.array_equal(got, want), (f, b)
        man.free()
        plan.free()
    imp.free()
    del base, experts, out
    torch.cuda.empty_cache()
