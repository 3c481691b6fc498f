"""Parity of the CUDA path (through the C ABI) with the CPU oracle on seeded inputs.

Bars: bit-exact for statistics' integer fields, norm/maxabs bits, TIES thresholds,
plans (mask, C_hat, counts, traversal order, digest) and manifests; merged bf16
within one bf16 ulp (fp32 checkpoints within 1e-6 relative) — the kernels follow
the same fp32 operation order as the oracle, so the merge is also expected to be
identical and the test reports any difference.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from conftest import oracle_family

pytestmark = pytest.mark.gpu

import paper_2605_29489_gb300 as mp  # noqa: E402
from paper_2605_29489_gb300 import synth  # noqa: E402


# ---- helpers ------------------------------------------------------------------------------------

def dev(fam, a):
    if fam.dtype == synth.BF16:
        return torch.from_numpy(a.view(np.int16)).cuda().view(torch.bfloat16)
    return torch.from_numpy(a).cuda()


def host(fam, t):
    if fam.dtype == synth.BF16:
        return t.view(torch.int16).cpu().numpy().view(np.uint16)
    return t.cpu().numpy()


def pinned(fam, a):
    t = torch.from_numpy(a.view(np.int16) if fam.dtype == synth.BF16 else a).pin_memory()
    return t.view(torch.bfloat16) if fam.dtype == synth.BF16 else t


def upload(fam, base, experts, host_experts=False):
    """base on the GPU; experts on the GPU, or in pinned host memory (a host-resident pool)"""
    b = dev(fam, base)
    ex = [pinned(fam, e) if host_experts else dev(fam, e) for e in experts]
    offs, nums, _ = fam.layout()
    mf = mp.family(list(zip(offs.tolist(), nums.tolist())), b, ex, fam.block_elems, fam.dtype,
                   1 if host_experts else 0)
    return mf, b, ex


def ordered(bits):
    b = bits.astype(np.int64)
    return np.where(b & 0x8000, -(b & 0x7FFF), b)


def assert_merge_close(fam, got, want, what="", signed_zero=True):
    """within the tolerance, then identical: bit for bit (signed_zero), or equal in value
    (+0 == -0) where only the value is defined"""
    if fam.dtype == synth.BF16:
        d = np.abs(ordered(got) - ordered(want))
        assert d.max(initial=0) <= 1, f"{what}: max ulp diff {d.max()}"
        n_diff = int((got != want).sum()) if signed_zero else int((d != 0).sum())
    else:
        g, w = got.astype(np.float64), want.astype(np.float64)
        rel = np.abs(g - w) / np.maximum(np.abs(w), 1e-30)
        assert np.all((rel <= 1e-6) | (g == w)), f"{what}: max rel {rel.max()}"
        same = (got.view(np.uint32) == want.view(np.uint32)) if signed_zero else ((g == w) | (np.isnan(g) & np.isnan(w)))
        n_diff = int((~same).sum())
    assert n_diff == 0, f"{what}: {n_diff} elements differ from the oracle (within tolerance, but not identical)"


def tensor_mask(fam):
    """bool mask of elements covered by tensors (gap elements are never written)"""
    offs, nums, total = fam.layout()
    m = np.zeros(total, bool)
    for o, n in zip(offs.tolist(), nums.tolist()):
        m[o:o + n] = True
    return m


def ops_for(K, kinds=("avg", "ta", "ties", "ties1", "dare")):
    out = []
    for k in kinds:
        if k == "avg":
            out.append(("avg", mp.make_op(mp.MP_OP_AVG, alpha=[1.0 / K] * K),
                        oracle.Op(oracle.AVG, K, alpha=[1.0 / K] * K)))
        elif k == "ta":
            out.append(("ta", mp.make_op(mp.MP_OP_TA, alpha=[0.3] * K), oracle.Op(oracle.TA, K, alpha=[0.3] * K)))
        elif k == "ties":
            out.append(("ties", mp.make_op(mp.MP_OP_TIES, lam=1.0, density=0.2, trim_scope=0),
                        oracle.Op(oracle.TIES, K, lam=1.0, density=0.2, trim_scope=0)))
        elif k == "ties1":
            out.append(("ties1", mp.make_op(mp.MP_OP_TIES, lam=0.7, density=0.35, trim_scope=1),
                        oracle.Op(oracle.TIES, K, lam=0.7, density=0.35, trim_scope=1)))
        elif k == "dare":
            alpha = [1.0 / K] * K
            out.append(("dare", mp.make_op(mp.MP_OP_DARE, alpha=alpha, drop_p=0.9, seed=1234567),
                        oracle.Op(oracle.DARE, K, alpha=alpha, drop_p=0.9, seed=1234567)))
        elif k == "ta_pb":   # score per byte (ragged blocks have different costs)
            alpha = [0.3 + 0.1 * i for i in range(K)]
            out.append(("ta_pb", mp.make_op(mp.MP_OP_TA, alpha=alpha, score_mode=1),
                        oracle.Op(oracle.TA, K, alpha=alpha, score_mode=1)))
        elif k == "avg_renorm":   # App. A.1's selected-only average
            alpha = [(i + 1) / (K * (K + 1) / 2) for i in range(K)]
            out.append(("avg_renorm", mp.make_op(mp.MP_OP_AVG_RENORM, alpha=alpha),
                        oracle.Op(oracle.AVG_RENORM, K, alpha=alpha)))
        elif k == "dare_ties":
            out.append(("dare_ties", mp.make_op(mp.MP_OP_DARE_TIES, lam=0.8, drop_p=0.7, seed=424242),
                        oracle.Op(oracle.DARE_TIES, K, lam=0.8, drop_p=0.7, seed=424242)))
        elif k == "ties_masked":   # App. A.1: TIES after masking (threshold of the masked deltas)
            out.append(("ties_masked", mp.make_op(mp.MP_OP_TIES_MASKED, lam=1.0, density=0.2),
                        oracle.Op(oracle.TIES_MASKED, K, lam=1.0, density=0.2)))
        elif k == "ties_masked1":
            out.append(("ties_masked1", mp.make_op(mp.MP_OP_TIES_MASKED, lam=0.7, density=0.35, trim_scope=1),
                        oracle.Op(oracle.TIES_MASKED, K, lam=0.7, density=0.35, trim_scope=1)))
        elif k == "ta_tiny":   # coefficients small enough that products of subnormals underflow to +-0
            alpha = [2.0 ** -20, -(2.0 ** -21), 2.0 ** -18][:K] + [2.0 ** -19] * max(0, K - 3)
            out.append(("ta_tiny", mp.make_op(mp.MP_OP_TA, alpha=alpha), oracle.Op(oracle.TA, K, alpha=alpha)))
        elif k == "dare_tiny":
            alpha = [2.0 ** -20, -(2.0 ** -21), 2.0 ** -18][:K] + [2.0 ** -19] * max(0, K - 3)
            out.append(("dare_tiny", mp.make_op(mp.MP_OP_DARE, alpha=alpha, drop_p=0.5, seed=77),
                        oracle.Op(oracle.DARE, K, alpha=alpha, drop_p=0.5, seed=77)))
        elif k == "ties_neg":   # a negative lambda: lambda * +0 = -0 where no sign wins
            out.append(("ties_neg", mp.make_op(mp.MP_OP_TIES, lam=-0.5, density=0.3),
                        oracle.Op(oracle.TIES, K, lam=-0.5, density=0.3)))
        elif k == "dare_ties_neg":
            out.append(("dare_ties_neg", mp.make_op(mp.MP_OP_DARE_TIES, lam=-0.75, drop_p=0.5, seed=99),
                        oracle.Op(oracle.DARE_TIES, K, lam=-0.75, drop_p=0.5, seed=99)))
        elif k == "ties_pb":
            out.append(("ties_pb", mp.make_op(mp.MP_OP_TIES, lam=1.0, density=0.2, score_mode=1),
                        oracle.Op(oracle.TIES, K, lam=1.0, density=0.2, score_mode=1)))
    return out


def run_case(fam, base, experts, kinds, fracs, check_merge=True, host_experts=False):
    mf, b, ex = upload(fam, base, experts, host_experts)
    covered = tensor_mask(fam)
    bo, bl, bt = fam.block_table()
    es = fam.elem_size
    C_full = fam.K * fam.n_params * es
    for name, gop, oop in ops_for(fam.K, kinds):
        masked = oop.kind == oracle.TIES_MASKED
        scope = oop.trim_scope if oop.kind in (oracle.TIES, oracle.TIES_MASKED) else 0
        of = oracle_family(fam, base, experts, trim_scope=scope)
        idx = mp.mp_index_blocks(mf, gop)
        norm, maxabs, nnz, tau = mp.mp_index_stats(idx)
        o_norm, o_max, o_nnz = oracle.index(of)
        assert np.array_equal(nnz, o_nnz), name
        assert np.array_equal(maxabs.view(np.uint32), o_max.view(np.uint32)), name
        assert np.array_equal(norm.view(np.uint32), o_norm.view(np.uint32)), name
        o_tau = None
        if oop.kind in (oracle.TIES, oracle.TIES_MASKED):
            o_tau = oracle.ties_thresholds(of, oop.density)
            assert np.array_equal(tau, o_tau), name
        for f in fracs:
            B = mp.mp_budget_from_fraction(mf, f) if f <= 1.0 else C_full + int(f)
            assert B == (math.floor(f * C_full) if f <= 1.0 else B)
            plan = mp.mp_plan(idx, gop, B)
            pi = mp.mp_plan_info(plan, idx)
            ng = of.n_groups
            opl = oracle.plan(fam.K, bl, of.blk_group, ng, es, oop, o_norm, o_max, o_nnz, None if masked else o_tau, B)
            what = f"{fam.name}/{name}/f={f}"
            assert pi["chat"] == opl["chat"] <= B, what
            assert pi["n_sel"] == opl["n_sel"], what
            assert pi["n_cand"] == opl["n_cand"], what
            assert np.array_equal(pi["mask"], opl["mask"]), what
            assert np.array_equal(pi["order"], opl["order"]), what
            assert pi["digest"] == opl["digest"], what
            if not check_merge:
                plan.free()
                continue
            out = torch.full_like(b, float("nan"))
            man = mp.mp_merge(mf, idx, plan, out)
            mi = mp.mp_manifest_info(man, fam.K)
            assert mi["realized_total"] == opl["chat"], what          # Prop. 1, realized = planned
            assert mi["touched"] == int((opl["mask"] != 0).sum()), what
            assert mi["digest"] == opl["digest"], what
            m_tau = oracle.ties_masked_thresholds(of, oop.density, opl["mask"]) if masked else o_tau
            want = oracle.merge(of, oop, tau=m_tau, mask=opl["mask"])
            got = host(fam, out)
            assert_merge_close(fam, got[covered], want[covered], what)
            if masked:   # the threshold pass re-reads only selected blocks
                assert 0 <= mp.mp_manifest_threshold_reads(man) <= opl["chat"], what
            if f >= 1.0:   # Eq. 5: full budget reproduces the unmasked operator
                # in value: the full read also adds the zero deltas of the blocks the plan
                # leaves out (nnz = 0), and adding a +0 can turn an accumulated -0 into +0
                phi = oracle.merge(of, oop, tau=o_tau, mask=None)
                assert_merge_close(fam, got[covered], phi[covered], what + " vs Phi", signed_zero=False)
            man.free()
            plan.free()
        idx.free()


# ---- families -------------------------------------------------------------------------------------

def fam_ragged_bf16():
    return synth.custom([5000, 70001, 65536, 8, 131072 + 17, 300, 4096], dtype=synth.BF16, block_elems=4096, K=3,
                        active_frac=0.5, name="ragged-bf16")


def fam_ragged_f32():
    return synth.custom([4096 * 3 + 5, 1000, 77, 2048], dtype=synth.F32, block_elems=1024, K=5, active_frac=0.4,
                        name="ragged-f32", log_mu=math.log(1e-3))


def fam_k9():
    return synth.custom([30000, 12345, 65536 * 2 + 100], dtype=synth.BF16, block_elems=8192, K=9, active_frac=0.5,
                        per_expert_active=True, name="k9")


def fam_k7():
    # K = 7: the whole-chunk merges for up to 8 experts (bf16)
    return synth.custom([30000, 8191, 65536 + 8], dtype=synth.BF16, block_elems=4096, K=7, active_frac=0.6,
                        per_expert_active=True, name="k7")


def fam_k16():
    # K = 16 with most blocks active for every expert: chunks of 17 fills fill the 17-slot ring
    return synth.custom([40000, 4097, 24576], dtype=synth.BF16, block_elems=4096, K=16, active_frac=0.9,
                        name="k16")


def fam_k17():
    return synth.custom([20000, 7777, 40000], dtype=synth.BF16, block_elems=2048, K=17, active_frac=0.3,
                        per_expert_active=True, name="k17")


def fam_k1():
    # K = 1, the smallest family (one-expert catalog groups, one-bit masks)
    return synth.custom([12000, 4096, 777], dtype=synth.BF16, block_elems=2048, K=1, active_frac=0.6, name="k1")


def fam_k32():
    # K = 32, the largest family: the access mask uses its top bit
    return synth.custom([9000, 4099, 16384], dtype=synth.BF16, block_elems=2048, K=32, active_frac=0.3,
                        per_expert_active=True, name="k32")


def fam_big_blocks():
    # 4 Mi-element blocks (a whole block is thousands of chunks), ragged tails, K = 2
    return synth.custom([(1 << 22) + (1 << 20) + 5, 3000, 1 << 22], dtype=synth.BF16, block_elems=1 << 22, K=2,
                        active_frac=0.7, name="big-blocks")


def fam_max_block():
    # the largest block the ABI allows (2^24 elements), one expert, fp32
    return synth.custom([(1 << 24) + 12], dtype=synth.F32, block_elems=1 << 24, K=1, active_frac=1.0, name="max-block",
                        log_mu=math.log(1e-3))


FRACS = [0.0, 0.1, 0.25, 0.5, 0.9, 1.0, 1000.0]


@pytest.mark.parametrize("make", [fam_ragged_bf16, fam_ragged_f32, fam_k7, fam_k9, fam_k16, fam_k17, fam_k32, fam_k1],
                         ids=lambda f: f.__name__)
def test_parity_small_families(make):
    fam = make()
    base, experts = fam.host_arrays()
    run_case(fam, base, experts, ("avg", "ta", "ties", "ties1", "dare", "ta_pb", "ties_pb", "avg_renorm", "dare_ties",
                                  "ties_masked", "ties_masked1"), FRACS)


@pytest.mark.parametrize("make", [fam_big_blocks, fam_max_block], ids=lambda f: f.__name__)
def test_parity_largest_blocks(make):
    """blocks of 2^22 and 2^24 elements: the canonical norm order over thousands of chunks,
    TIES thresholds and DARE masks at block offsets beyond 2^24"""
    fam = make()
    base, experts = fam.host_arrays()
    run_case(fam, base, experts, ("avg", "ta", "ties", "dare", "ta_pb"), [0.3, 0.6, 1.0])


def test_parity_tiny_config():
    """8 fp32 512x512 tensors, K=4: AVG, TIES rho=0.2, DARE p=0.9 at budgets 1.0/0.5/0.25"""
    fam = synth.tiny()
    base, experts = fam.host_arrays()
    run_case(fam, base, experts, ("avg", "ties", "dare"), [1.0, 0.5, 0.25])


def signed_zero_family(dtype, K=3):
    """every element drawn from +-0, +-(the smallest subnormal), +-(twice it) and +-1, the
    experts equal to the base at 40 % of the elements and over whole blocks for some
    (block, expert) pairs: signed zeros in the base, deltas of +0, -0 results of underflowing
    products, ties of equal magnitudes in the TIES trim, and zero-delta blocks the plan omits"""
    fam = synth.custom([3 * 1024 + 77, 2048, 515], dtype=dtype, block_elems=1024, K=K,
                        name=f"signed-zero-{dtype}-k{K}")
    _, _, total = fam.layout()
    rng = np.random.default_rng(2605)
    if dtype == synth.BF16:
        pal = np.array([0x0000, 0x8000, 0x0001, 0x8001, 0x0002, 0x8002, 0x3F80, 0xBF80], np.uint16)
    else:
        pal = np.array([0x00000000, 0x80000000, 0x00000001, 0x80000001, 0x00000002, 0x80000002, 0x3F800000,
                        0xBF800000], np.uint32).view(np.float32)
    base = pal[rng.integers(0, 6, total)]
    bo, bl, _ = fam.block_table()
    experts = []
    for i in range(fam.K):
        e = np.where(rng.random(total) < 0.4, base, pal[rng.integers(0, len(pal), total)])
        for b in range(i % 3, fam.n_blocks, 3):   # whole blocks equal to the base: nnz = 0
            e[int(bo[b]):int(bo[b] + bl[b])] = base[int(bo[b]):int(bo[b] + bl[b])]
        experts.append(e.astype(base.dtype))
    return fam, base, experts


@pytest.mark.parametrize("dtype,K,host_experts", [(synth.BF16, 3, False), (synth.F32, 3, False), (synth.BF16, 17, False),
                                                  (synth.BF16, 3, True)],
                         ids=["bf16", "f32", "bf16-k17", "bf16-host-pool"])
def test_signed_zeros_and_subnormals_bit_for_bit(dtype, K, host_experts):
    """the kernels reach the oracle's result bit for bit, the sign of every zero included, on
    inputs made of signed zeros and subnormals: the merge adds each selected (and, for DARE,
    kept) term in the oracle's order and omits the rest, and an unselected block is M_0 plus
    the zero the operator adds.  K = 17 takes the streaming merges for every operator; the
    host-pool case gathers the experts from pinned host memory"""
    fam, base, experts = signed_zero_family(dtype, K)
    run_case(fam, base, experts, ("avg", "ta", "ta_tiny", "ties", "ties_neg", "dare", "dare_tiny", "avg_renorm",
                                  "dare_ties", "dare_ties_neg", "ties_masked"), [0.0, 0.3, 1.0],
             host_experts=host_experts)


def test_device_fill_matches_host_fill():
    fam = fam_k9()
    base, experts = fam.host_arrays()
    db, dex = fam.device_arrays()
    assert np.array_equal(host(fam, db), base)
    for e, d in zip(experts, dex):
        assert np.array_equal(host(fam, d), e)


# ---- semantics on the GPU -------------------------------------------------------------------------

def test_non_anticipation_unselected_blocks_never_read():
    """Sec. 2: omitted entries enter only through the mask.  Poison every unselected
    expert block with NaN after planning: the merged output must not change."""
    fam = fam_ragged_bf16()
    base, experts = fam.host_arrays()
    mf, b, ex = upload(fam, base, experts)
    bo, bl, _ = fam.block_table()
    for name, gop, _ in ops_for(fam.K, ("ta", "ties", "dare")):
        idx = mp.mp_index_blocks(mf, gop)
        plan = mp.mp_plan(idx, gop, mp.mp_budget_from_fraction(mf, 0.3))
        mask = mp.mp_plan_info(plan, idx)["mask"]
        out1 = torch.empty_like(b)
        mp.mp_merge(mf, idx, plan, out1).free()
        poisoned = [e.clone() for e in ex]
        for bb in range(fam.n_blocks):
            for i in range(fam.K):
                if not (mask[bb] >> i) & 1:
                    poisoned[i][int(bo[bb]):int(bo[bb] + bl[bb])] = float("nan")
        offs, nums, _ = fam.layout()
        mf2 = mp.family(list(zip(offs.tolist(), nums.tolist())), b, poisoned, fam.block_elems, fam.dtype, 0)
        out2 = torch.empty_like(b)
        mp.mp_merge(mf2, idx, plan, out2).free()
        cov = torch.from_numpy(tensor_mask(fam)).cuda()
        assert torch.equal(out1.view(torch.int16)[cov], out2.view(torch.int16)[cov]), name
        assert not torch.isnan(out2[cov].float()).any(), name
        plan.free()
        idx.free()


def test_nonfinite_delta_reported():
    fam = synth.custom([9000], dtype=synth.BF16, block_elems=2048, K=2)
    base, experts = fam.host_arrays()
    experts[1] = experts[1].copy()
    experts[1][4321] = 0x7FC0  # NaN
    mf, b, ex = upload(fam, base, experts)
    op = mp.make_op(mp.MP_OP_AVG, alpha=[0.5, 0.5])
    idx = mp.mp_index_blocks(mf, op)
    with pytest.raises(mp.MergePipeError) as ei:
        mp.mp_index_stats(idx)
    assert ei.value.status == -4
    plan = mp.mp_plan(idx, op, 10 ** 9)
    with pytest.raises(mp.MergePipeError) as ei:
        mp.mp_plan_info(plan)
    assert ei.value.status == -4


def test_invalid_arguments_rejected():
    fam = synth.custom([4096], dtype=synth.BF16, block_elems=1024, K=2)
    base, experts = fam.host_arrays()
    mf, b, ex = upload(fam, base, experts)
    op = mp.make_op(mp.MP_OP_AVG, alpha=[0.5, 0.5])
    bad = mp.family([(0, 4096)], b, ex, 1004, mp.MP_BF16, 0)       # block size not a multiple of 8
    with pytest.raises(mp.MergePipeError) as ei:
        mp.mp_index_blocks(bad, op)
    assert ei.value.status == -1
    bad = mp.family([(3, 4000)], b, ex, 1024, mp.MP_BF16, 0)       # tensor not 16-byte aligned
    with pytest.raises(mp.MergePipeError):
        mp.mp_index_blocks(bad, op)
    with pytest.raises(mp.MergePipeError):                          # alpha missing
        mp.mp_index_blocks(mf, mp.make_op(mp.MP_OP_AVG))
    idx = mp.mp_index_blocks(mf, op)
    with pytest.raises(mp.MergePipeError) as ei:                    # TIES plan on a non-TIES index
        mp.mp_plan(idx, mp.make_op(mp.MP_OP_TIES, density=0.2), 100)
    assert ei.value.status == -8
    plan = mp.mp_plan(idx, op, 10 ** 6)
    with pytest.raises(mp.MergePipeError):                          # out aliases the base
        mp.mp_merge(mf, idx, plan, b)
    host_base = torch.zeros_like(b, device="cpu")
    with pytest.raises(mp.MergePipeError):                          # out on the host
        mp.mp_merge(mf, idx, plan, host_base)


def test_replay_is_bit_identical():
    """A manifest's plan replayed gives the same bytes (replayable manifests, Sec. 3)."""
    fam = fam_k9()
    base, experts = fam.host_arrays()
    mf, b, ex = upload(fam, base, experts)
    _, gop, _ = ops_for(fam.K, ("dare",))[0]
    idx = mp.mp_index_blocks(mf, gop)
    plan = mp.mp_plan(idx, gop, mp.mp_budget_from_fraction(mf, 0.4))
    o1, o2 = torch.empty_like(b), torch.empty_like(b)
    m1 = mp.mp_merge(mf, idx, plan, o1)
    m2 = mp.mp_merge(mf, idx, plan, o2)
    cov = torch.from_numpy(tensor_mask(fam)).cuda()   # padding between tensors is never written
    assert torch.equal(o1.view(torch.int16)[cov], o2.view(torch.int16)[cov])
    assert mp.mp_manifest_info(m1, fam.K)["digest"] == mp.mp_manifest_info(m2, fam.K)["digest"]


def test_manifest_records_lineage():
    """Sec. 3: the manifest records the lineage of the merged checkpoint (the caller's ids of
    M_0..M_K as given with the family); without ids it records zeros"""
    fam = fam_ragged_bf16()
    base, experts = fam.host_arrays()
    b, ex = dev(fam, base), [dev(fam, e) for e in experts]
    offs, nums, _ = fam.layout()
    ids = [0xB0, 11, 22, 0xFFFFFFFFFFFFFFFF][: fam.K + 1]
    gop = mp.make_op(mp.MP_OP_AVG, alpha=[1.0 / fam.K] * fam.K)
    for lin in (ids, None):
        mf = mp.family(list(zip(offs.tolist(), nums.tolist())), b, ex, fam.block_elems, fam.dtype, 0, lineage_ids=lin)
        idx = mp.mp_index_blocks(mf, gop)
        plan = mp.mp_plan(idx, gop, mp.mp_budget_from_fraction(mf, 0.5))
        man = mp.mp_merge(mf, idx, plan, torch.empty_like(b))
        got = mp.mp_manifest_lineage(man, fam.K).tolist()
        assert got == (ids if lin is not None else [0] * (fam.K + 1))
        for h in (man, plan, idx):
            h.free()
