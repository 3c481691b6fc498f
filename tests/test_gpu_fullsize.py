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


def oracle_merged_hashes(pool, spec, fam, cases):
    """the oracle's merge of every block under every budget's mask of every case, hashed:
    [uint64 [n_budgets, n_blocks] per case]; cases = [(op_args, masks, tau)]"""
    nb = fam.n_blocks
    outs = [np.zeros((m.shape[0], nb), np.uint64) for _, m, _ in cases]
    chunks = np.array_split(np.arange(nb), max(1, nb // 128))
    futs = [pool.submit(ow.merged_hashes, spec, c, [(a, m[:, c], t) for a, m, t in cases]) for c in chunks]
    for f in cf.as_completed(futs):
        blocks, hs = f.result()
        for out, h in zip(outs, hs):
            out[:, blocks] = h
    return outs


def run_family(pool, spec, cases, host_pool=False):
    """For each case (gop, op_args, fracs, ties_density): index -> plan -> merge at every
    budget as the benchmark runs them; statistics, thresholds and plans bit-exact against the
    oracle; every merged block's hash equal to the hash of the oracle's merge of that block
    (a mismatching block is then compared element by element); sampled blocks element by
    element; realized = planned <= B.  host_pool: the experts live in pinned host memory."""
    fam = ow.family(spec)
    es = fam.elem_size
    # --- GPU data, as the benchmark holds it ---
    base, experts = fam.device_arrays()
    if host_pool:   # the experts in pinned host memory, one at a time through the device
        hexp = []
        for k in range(len(experts)):
            h = torch.empty(experts[k].shape, dtype=experts[k].dtype, pin_memory=True)
            h.copy_(experts[k])
            hexp.append(h)
            experts[k] = None
            torch.cuda.empty_cache()
        experts = hexp
    offs, nums, _ = fam.layout()
    mf = mp.family(list(zip(offs.tolist(), nums.tolist())), base, experts, fam.block_elems, fam.dtype,
                   1 if host_pool else 0)
    bo, bl, bt = fam.block_table()
    samples = sample_blocks(fam)
    C_full = fam.K * fam.n_params * es
    n_budgets = sum(len(c[2]) for c in cases)
    free_b, _ = torch.cuda.mem_get_info()
    n_out = n_budgets if free_b > (n_budgets + 1) * base.numel() * base.element_size() else 1
    outs = [torch.empty_like(base) for _ in range(n_out)]
    pending = []   # (case, k, f, slot): the GPU output's block hashes wait for the oracle's
    hash_cases = []
    slot = 0
    for gop, op_args, fracs, ties_density in cases:
        oop = oracle.Op(op_args[0], op_args[1], **dict(op_args[2]))
        idx = mp.mp_index_blocks(mf, gop)
        g_norm, g_max, g_nnz, g_tau = mp.mp_index_stats(idx)
        o_norm, o_max, o_nnz, o_tau = oracle_catalog(pool, spec, fam, ties_density)
        assert np.array_equal(g_nnz, o_nnz)
        assert np.array_equal(g_max.view(np.uint32), o_max.view(np.uint32))
        assert np.array_equal(g_norm.view(np.uint32), o_norm.view(np.uint32))
        if ties_density is not None:
            assert np.array_equal(g_tau, o_tau)
        mp.mp_index_hashes(mf, idx)
        masks = np.zeros((len(fracs), fam.n_blocks), np.uint32)
        g_hash = np.zeros((len(fracs), fam.n_blocks), np.uint64)
        for k, f in enumerate(fracs):
            out = outs[slot % n_out]
            B = mp.mp_budget_from_fraction(mf, f)
            assert B == math.floor(f * C_full)
            plan = mp.mp_plan(idx, gop, B)
            pi = mp.mp_plan_info(plan, idx)
            opl = oracle.plan(fam.K, bl, bt, len(fam.tensors), es, oop, o_norm, o_max, o_nnz, o_tau, B)
            assert (pi["chat"], pi["n_sel"], pi["n_cand"], pi["digest"]) == \
                (opl["chat"], opl["n_sel"], opl["n_cand"], opl["digest"]), f
            assert np.array_equal(pi["mask"], opl["mask"]), f
            assert np.array_equal(pi["order"], opl["order"]), f
            masks[k] = opl["mask"]
            man = mp.mp_merge(mf, idx, plan, out)
            mi = mp.mp_manifest_info(man, fam.K)
            assert mi["realized_total"] == opl["chat"] <= B                       # Prop. 1
            assert mi["touched"] == int((opl["mask"] != 0).sum())
            # Alg. 2's validation: every block the merge read matches the catalog; the
            # output's block hashes come back with it
            mp.mp_manifest_validate(mf, idx, plan, out, man)
            v = mp.mp_manifest_validation(man, fam.n_blocks)
            assert v["mismatched"] == 0
            g_hash[k] = v["out_hash"]
            for b in samples:   # sampled blocks element by element
                hb, hex_ = fam.block_host(b)
                s = slice(int(bo[b]), int(bo[b] + bl[b]))
                tau_k = None if o_tau is None else o_tau[:, bt[b]]
                want = oracle.merge_block(fam.dtype, int(bo[b]), hb, hex_, int(opl["mask"][b]), oop, tau_k)
                got = out[s].view(torch.int16).cpu().numpy().view(np.uint16)
                assert np.array_equal(got, want), (f, b)
            pending.append((len(hash_cases), k, f, slot))
            slot += 1
            man.free()
            plan.free()
        idx.free()
        hash_cases.append((op_args, masks, o_tau, g_hash))
    # --- every block of every budget: the output's block hashes against the oracle's merge ---
    o_hashes = oracle_merged_hashes(pool, spec, fam, [(a, m, t) for a, m, t, _ in hash_cases])
    for c, k, f, sl in pending:
        op_args, masks, o_tau, g_hash = hash_cases[c]
        bad = np.nonzero(g_hash[k] != o_hashes[c][k])[0]
        if bad.size and n_out == n_budgets:   # the differing blocks element by element
            oop = oracle.Op(op_args[0], op_args[1], **dict(op_args[2]))
            for b in bad[:8]:
                hb, hex_ = fam.block_host(int(b))
                tau_k = None if o_tau is None else o_tau[:, bt[b]]
                want = oracle.merge_block(fam.dtype, int(bo[b]), hb, hex_, int(masks[k, b]), oop, tau_k)
                got = outs[sl][int(bo[b]):int(bo[b] + bl[b])].view(torch.int16).cpu().numpy().view(np.uint16)
                d = np.nonzero(got != want)[0]
                print(f"op {op_args[0]} f={f} block {b}: {d.size} elements differ, first at {d[:5]}")
        assert bad.size == 0, (op_args[0], f, bad[:20])
    del base, experts, outs
    torch.cuda.empty_cache()


def _op_args(kind, K, **kw):
    return (kind, K, tuple(sorted(kw.items())))


def test_fullsize_qwen05b_task_arithmetic(pool):
    """Qwen2.5-0.5B-shaped family, K=8, task arithmetic lambda=0.3, budgets 1.0/0.5/0.25/0.1"""
    K = 8
    run_family(pool, ("qwen25_05b", ()), [(mp.make_op(mp.MP_OP_TA, alpha=[0.3] * K),
                                          _op_args(oracle.TA, K, alpha=(0.3,) * K), [1.0, 0.5, 0.25, 0.1], None)])


def test_fullsize_qwen15b_dare(pool):
    """Qwen2.5-1.5B-shaped family, K=16 with per-expert active sets, DARE p=0.9 then AVG, budget 0.25"""
    K = 16
    a = [1.0 / K] * K
    run_family(pool, ("qwen25_15b", ()), [(mp.make_op(mp.MP_OP_DARE, alpha=a, drop_p=0.9, seed=20260),
                                          _op_args(oracle.DARE, K, alpha=tuple(a), drop_p=0.9, seed=20260), [0.25],
                                          None)])


def test_fullsize_llama3_8b_ties(pool):
    """Llama-3-8B-shaped family, K=4, TIES density 0.2, budgets 1.0/0.5/0.25/0.1"""
    K = 4
    if torch.cuda.get_device_properties(0).total_memory < 120 * 2 ** 30:
        pytest.skip("needs about 100 GB of device memory")
    run_family(pool, ("llama3_8b", ()), [(mp.make_op(mp.MP_OP_TIES, lam=1.0, density=0.2),
                                         _op_args(oracle.TIES, K, lam=1.0, density=0.2), [1.0, 0.5, 0.25, 0.1], 0.2)])


def test_fullsize_llama3_8b_host_pool(pool):
    """Llama-3-8B-shaped base in HBM with K=8 experts (128 GB) in pinned host memory: AVG and
    TIES density 0.2 at budgets 1.0 / 0.25 / 0.1, every merged block checked"""
    K = 8
    if torch.cuda.get_device_properties(0).total_memory < 120 * 2 ** 30:
        pytest.skip("needs about 100 GB of device memory")
    if os.sysconf("SC_PHYS_PAGES") * os.sysconf("SC_PAGE_SIZE") < 160 * 2 ** 30:
        pytest.skip("needs about 160 GB of host memory (128 GB of pinned experts)")
    a = [1.0 / K] * K
    run_family(pool, ("llama3_8b", (("K", K),)),
               [(mp.make_op(mp.MP_OP_TIES, lam=1.0, density=0.2), _op_args(oracle.TIES, K, lam=1.0, density=0.2),
                 [1.0, 0.25, 0.1], 0.2),
                (mp.make_op(mp.MP_OP_AVG, alpha=a), _op_args(oracle.AVG, K, alpha=tuple(a)), [1.0, 0.25, 0.1], None)],
               host_pool=True)


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
