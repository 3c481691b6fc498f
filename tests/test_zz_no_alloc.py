"""mp_plan_noalloc: the access plan for callers that cannot allocate.

Some callers may not allocate device memory at all: their memory comes from another
framework's arena, or they run in latency-critical loops that cannot pay for an
allocation, or where CUDA allocation calls are not allowed.  mp_plan_noalloc takes
every input and output as a caller buffer and uses a fixed device array inside the
library as scratch.  This test checks, through the C ABI, that two calls in a row give
exactly the plan mp_plan gives (plans are integers: mask, traversal order, planned
bytes, counts and digest must match bit for bit), and that requests beyond the
array's limit are refused.  It sits in its own file, collected last, and passes both
alone in a fresh process and after the other tests.
"""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

import paper_2605_29489_gb300 as mp  # noqa: E402
from paper_2605_29489_gb300 import synth  # noqa: E402


def _dev(a, dtype):
    return torch.from_numpy(np.ascontiguousarray(a).view(dtype)).cuda()


def _run(fam, gop, scope, fracs):
    base, experts = fam.host_arrays()
    if fam.dtype == synth.BF16:
        b = torch.from_numpy(base.view(np.int16)).cuda().view(torch.bfloat16)
        ex = [torch.from_numpy(e.view(np.int16)).cuda().view(torch.bfloat16) for e in experts]
    else:
        b = torch.from_numpy(base).cuda()
        ex = [torch.from_numpy(e).cuda() for e in experts]
    offs, nums, _ = fam.layout()
    mf = mp.family(list(zip(offs.tolist(), nums.tolist())), b, ex, fam.block_elems, fam.dtype, 0)
    idx = mp.mp_index_blocks(mf, gop)
    norm, maxabs, nnz, tau = mp.mp_index_stats(idx)
    nb, nu, ng = mp.mp_index_shape(idx)
    _, bl, bt = fam.block_table()
    groups = bt if scope == 0 else np.zeros_like(bt)
    d_len, d_grp = _dev(bl, np.int32), _dev(groups, np.int32)
    d_norm, d_max, d_nnz = _dev(norm, np.float32), _dev(maxabs, np.float32), _dev(nnz, np.int32)
    d_tau = _dev(tau, np.int32) if gop.kind == mp.MP_OP_TIES else None
    d_err = torch.zeros(1, dtype=torch.int32, device="cuda")
    mask = torch.empty(nb, dtype=torch.int32, device="cuda")
    order = torch.empty(nu, dtype=torch.int32, device="cuda")
    summary = torch.empty(8, dtype=torch.int64, device="cuda")
    for f in fracs:
        B = mp.mp_budget_from_fraction(mf, f)
        plan = mp.mp_plan(idx, gop, B)
        ref = mp.mp_plan_info(plan, idx)
        for _ in range(2):                       # two calls in a row share the static scratch
            mask.fill_(-1)
            order.fill_(-1)
            summary.fill_(-1)
            mp.mp_plan_noalloc(fam.K, nb, ng, fam.dtype, d_len, d_grp, d_norm, d_max, d_nnz, d_tau, d_err, gop, B,
                               mask, order, summary)
            torch.cuda.synchronize()
            s = summary.cpu().numpy().view(np.uint64)
            assert (int(s[0]), int(s[1]), int(s[2]), int(s[4])) == (ref["chat"], ref["n_sel"], ref["n_cand"],
                                                                    ref["digest"]), f
            assert int(s[6]) == 0
            assert np.array_equal(mask.cpu().numpy().view(np.uint32), ref["mask"]), f
            got_order = order.cpu().numpy().view(np.uint32)[: ref["n_cand"]]
            assert np.array_equal(got_order, ref["order"]), f
        plan.free()
    idx.free()


def test_noalloc_plan_matches_mp_plan_additive_and_dare():
    fam = synth.custom([5000, 70001, 65536, 8, 131089, 300], dtype=synth.BF16, block_elems=4096, K=3,
                       active_frac=0.5)
    _run(fam, mp.make_op(mp.MP_OP_TA, alpha=[0.3] * 3), 0, [0.1, 0.5, 1.0])
    _run(fam, mp.make_op(mp.MP_OP_TA, alpha=[0.3, 0.5, 0.9], score_mode=1), 0, [0.1, 0.5])
    fam9 = synth.custom([30000, 12345, 131172], dtype=synth.BF16, block_elems=8192, K=9, active_frac=0.5,
                        per_expert_active=True)
    _run(fam9, mp.make_op(mp.MP_OP_DARE, alpha=[1 / 9] * 9, drop_p=0.9, seed=5), 0, [0.25, 0.7])


def test_noalloc_plan_matches_mp_plan_ties():
    fam = synth.custom([4096 * 3 + 5, 1000, 77, 2048], dtype=synth.F32, block_elems=1024, K=5, active_frac=0.4)
    _run(fam, mp.make_op(mp.MP_OP_TIES, lam=1.0, density=0.2, trim_scope=0), 0, [0.2, 0.6])
    _run(fam, mp.make_op(mp.MP_OP_TIES, lam=0.5, density=0.35, trim_scope=1), 1, [0.3])


def test_noalloc_plan_with_negative_zero_coefficient_matches_mp_plan():
    """an alpha of -0.0 scores its expert's units as +0 on both entry points (|coef| clears
    the sign), so a zero-weight expert ranks last, not ahead of every positive score"""
    fam = synth.custom([5000, 70001, 65536], dtype=synth.BF16, block_elems=4096, K=3, active_frac=0.5)
    _run(fam, mp.make_op(mp.MP_OP_TA, alpha=[0.3, -0.0, 0.5]), 0, [0.1, 0.5, 1.0])
    _run(fam, mp.make_op(mp.MP_OP_TA, alpha=[-0.0, 0.2, -0.4], score_mode=1), 0, [0.3])


def test_noalloc_refuses_operators_that_mp_plan_refuses():
    """a NaN alpha, an AVG_RENORM alpha <= 0 and a drop probability above 1 are refused by
    both entry points, before anything is launched"""
    fam = synth.custom([5000, 7001], dtype=synth.BF16, block_elems=4096, K=2, active_frac=0.5)
    base, experts = fam.host_arrays()
    b = torch.from_numpy(base.view(np.int16)).cuda().view(torch.bfloat16)
    ex = [torch.from_numpy(e.view(np.int16)).cuda().view(torch.bfloat16) for e in experts]
    offs, nums, _ = fam.layout()
    mf = mp.family(list(zip(offs.tolist(), nums.tolist())), b, ex, fam.block_elems, fam.dtype, 0)
    good = mp.make_op(mp.MP_OP_TA, alpha=[0.3, 0.3])
    idx = mp.mp_index_blocks(mf, good)
    nb, nu, ng = mp.mp_index_shape(idx)
    t = torch.zeros(max(nu, 16), dtype=torch.int32, device="cuda")
    summary = torch.zeros(8, dtype=torch.int64, device="cuda")
    for bad in (mp.make_op(mp.MP_OP_TA, alpha=[float("nan"), 0.3]),
                mp.make_op(mp.MP_OP_AVG_RENORM, alpha=[0.5, 0.0]),
                mp.make_op(mp.MP_OP_DARE, alpha=[0.5, 0.5], drop_p=1.5)):
        with pytest.raises(mp.MergePipeError) as e1:
            mp.mp_plan(idx, bad, 100)
        with pytest.raises(mp.MergePipeError) as e2:
            mp.mp_plan_noalloc(fam.K, nb, ng, fam.dtype, t, t, t, t, t, None, t, bad, 100, t, t, summary)
        assert e1.value.status == e2.value.status == -1
    idx.free()


def test_noalloc_plan_qwen_shaped_family():
    """Qwen2.5-0.5B tensor shapes cut to 2 layers, K=8, 64Ki-element blocks (20,400 units)"""
    _run(synth.qwen25_05b(layers=2), mp.make_op(mp.MP_OP_TA, alpha=[0.3] * 8), 0, [0.25, 1.0])


def test_noalloc_rejects_requests_beyond_the_static_limit():
    t = torch.zeros(16, dtype=torch.int32, device="cuda")
    op = mp.make_op(mp.MP_OP_AVG, alpha=[0.5, 0.5])
    with pytest.raises(mp.MergePipeError) as ei:
        mp.mp_plan_noalloc(2, 1 << 19, 1, mp.MP_BF16, t, t, t, t, t, None, t, op, 100, t, t, t)
    assert ei.value.status == -1
    assert "524288" in str(ei.value)


def test_noalloc_plan_at_the_static_limit_matches_oracle():
    """exactly K * n_blocks = 524288 units (K = 32, 16384 blocks of mixed lengths) from a
    seeded synthetic catalog: the plan equals the oracle's bit for bit"""
    import oracle

    K, nb = 32, 1 << 14
    rng = np.random.default_rng(77)
    blk_len = rng.choice([4096, 4096, 4096, 1000, 7], nb).astype(np.uint32)
    norm = rng.lognormal(size=(K, nb)).astype(np.float32)
    norm[:, ::5] = norm[:, 1::5][:, : norm[:, ::5].shape[1]]       # equal scores: the tie-break decides
    maxabs = norm.copy()
    nnz = np.minimum(rng.integers(0, 5000, (K, nb)), blk_len[None, :]).astype(np.uint32)
    nnz[rng.random((K, nb)) < 0.1] = 0
    alpha = [0.1 + 0.01 * i for i in range(K)]
    gop = mp.make_op(mp.MP_OP_TA, alpha=alpha)
    oop = oracle.Op(oracle.TA, K, alpha=alpha)
    d_len, d_norm, d_max, d_nnz = _dev(blk_len, np.int32), _dev(norm, np.float32), _dev(maxabs, np.float32), \
        _dev(nnz, np.int32)
    d_err = torch.zeros(1, dtype=torch.int32, device="cuda")
    mask = torch.empty(nb, dtype=torch.int32, device="cuda")
    order = torch.empty(K * nb, dtype=torch.int32, device="cuda")
    summary = torch.empty(8, dtype=torch.int64, device="cuda")
    full = K * int(blk_len.sum()) * 2
    for f in (0.05, 0.5):
        B = int(f * full)
        mp.mp_plan_noalloc(K, nb, 1, mp.MP_BF16, d_len, None, d_norm, d_max, d_nnz, None, d_err, gop, B, mask,
                           order, summary)
        torch.cuda.synchronize()
        opl = oracle.plan(K, blk_len, np.zeros(nb, np.uint32), 1, 2, oop, norm, maxabs, nnz, None, B)
        s = summary.cpu().numpy().view(np.uint64)
        assert (int(s[0]), int(s[1]), int(s[2]), int(s[4])) == (opl["chat"], opl["n_sel"], opl["n_cand"],
                                                                opl["digest"]), f
        assert np.array_equal(mask.cpu().numpy().view(np.uint32), opl["mask"]), f
        assert np.array_equal(order.cpu().numpy().view(np.uint32)[: opl["n_cand"]], opl["order"]), f
