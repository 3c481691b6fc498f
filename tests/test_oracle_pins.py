"""Pins of the CPU oracle to things other than itself (no GPU needed).

Each test ties one oracle function to a library routine, a closed form, a
hand-worked example, brute force on tiny inputs or a published test vector, so
that a dropped term, a wrong sign or index, or a transposed operand fails.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle
from conftest import oracle_family

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def bf16_bits_torch(x: np.ndarray) -> np.ndarray:
    t = torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def bf16_to_f32(h: np.ndarray) -> np.ndarray:
    return (h.astype(np.uint32) << 16).view(np.float32)


def to_bf16(values) -> np.ndarray:
    return bf16_bits_torch(np.asarray(values, np.float32))


# ---- element conversion ------------------------------------------------------------------------

def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(1)
    vals = np.concatenate([
        rng.standard_normal(4000).astype(np.float32) * np.float32(0.02),
        rng.standard_normal(2000).astype(np.float32) * np.float32(1e-30),
        (rng.integers(0, 2**32, 4000, dtype=np.uint64).astype(np.uint32)).view(np.float32),
        # exact ties between two bf16 values (round to even both ways)
        ((np.arange(0, 512, dtype=np.uint32) << 16) | 0x8000).view(np.float32),
        np.array([0.0, -0.0, np.inf, -np.inf, 3.4e38, -3.4e38, 1e-45], np.float32),
    ])
    vals = vals[~np.isnan(vals)]
    ref = bf16_bits_torch(vals)
    got = np.array([oracle.bf16_bits(float(v)) for v in vals], np.uint16)
    assert np.array_equal(got, ref)


def test_bf16_rounding_keeps_nan_a_nan():
    """IEEE: a NaN converts to a NaN, also one whose payload lies only in the 16 bits that
    bf16 drops (cutting them would leave an infinity).  The float32 bits go to the C
    function unchanged (a Python float round trip would quiet a signalling NaN)."""
    import ctypes
    import struct

    pats = [0x7F800001, 0xFF800001, 0x7F80FFFF, 0x7FC00000, 0x7FBFFFFF, 0xFFC00001, 0x7F801234]
    for bits in pats:
        x = ctypes.c_float.from_buffer_copy(struct.pack("<I", bits))
        h = int(oracle.lib().orc_f32_to_bf16(x))
        t = torch.from_numpy(np.array([bits], np.uint32).view(np.float32)).to(torch.bfloat16)
        assert bool(torch.isnan(t).item())
        assert (h & 0x7F80) == 0x7F80 and (h & 0x007F) != 0, hex(bits)   # a bf16 NaN


def test_ties_key_is_bf16_magnitude():
    rng = np.random.default_rng(2)
    d = (rng.standard_normal(3000) * 10.0 ** rng.uniform(-8, 2, 3000)).astype(np.float32)
    ref = bf16_bits_torch(np.abs(d)) & 0x7FFF
    got = np.array([oracle.ties_key(float(v)) for v in d], np.uint32)
    assert np.array_equal(got, ref.astype(np.uint32))


# ---- block statistics -----------------------------------------------------------------------------

@pytest.mark.parametrize("n", [65536, 65536 - 3, 4096 + 5, 1, 7, 2048 * 8 + 9])
def test_block_stats_integer_closed_form(n):
    """integer deltas: every partial sum is exact, so the norm is sqrt(sum k^2) in any order"""
    rng = np.random.default_rng(n)
    k = rng.integers(-3, 4, n)
    base = np.zeros(n, np.float32)
    expert = k.astype(np.float32)
    nrm, mx, nz, ss = oracle.block_stats(oracle.BF16, to_bf16(base), to_bf16(expert))
    s = int((k * k).sum())
    assert ss == float(s)
    assert nrm == np.float32(math.sqrt(s))
    assert mx == float(np.abs(k).max())
    assert nz == int((k != 0).sum())


def test_block_stats_single_element_positions():
    """one nonzero delta at every lane/vector position is found and counted once"""
    n = 4096 * 2 + 3
    for pos in [0, 7, 8, 255 * 8, 256 * 8, 256 * 8 + 1, n - 1]:
        e = np.zeros(n, np.float32)
        e[pos] = 3.0
        nrm, mx, nz, ss = oracle.block_stats(oracle.BF16, to_bf16(np.zeros(n)), to_bf16(e))
        assert (nrm, mx, nz, ss) == (3.0, 3.0, 1, 9.0), pos


@pytest.mark.parametrize("dtype", [oracle.BF16, oracle.F32])
def test_block_stats_against_fp64(dtype):
    rng = np.random.default_rng(3 + dtype)
    n = 65536 - 11
    base32 = (rng.standard_normal(n) * 0.02).astype(np.float32)
    exp32 = base32 + (rng.standard_normal(n) * 1e-3).astype(np.float32)
    z = rng.random(n) < 0.2
    exp32[z] = base32[z]
    if dtype == oracle.BF16:
        b, e = to_bf16(base32), to_bf16(exp32)
        d = bf16_to_f32(e) - bf16_to_f32(b)
    else:
        b, e = base32, exp32
        d = e - b
    nrm, mx, nz, ss = oracle.block_stats(dtype, b, e)
    exact = float(np.sqrt(np.sum(d.astype(np.float64) ** 2)))
    per_lane = math.ceil(n / (8 if dtype == oracle.BF16 else 4) / 256) * (8 if dtype == oracle.BF16 else 4)
    bound = (per_lane + 8 + 1) * 2.0 ** -24
    assert abs(nrm - exact) <= bound * exact
    assert mx == float(np.abs(d).max())
    assert nz == int(np.count_nonzero(d))
    assert ss == pytest.approx(exact * exact, rel=1e-12)


def test_block_stats_rejects_nonfinite():
    b = to_bf16(np.zeros(64))
    for bad in [np.nan, np.inf, -np.inf]:
        e = np.zeros(64, np.float32)
        e[17] = bad
        with pytest.raises(oracle.OracleError) as ei:
            oracle.block_stats(oracle.BF16, b, to_bf16(e))
        assert ei.value.rc == oracle.ENONFINITE


def test_ties_key_histogram_rejects_nonfinite():
    """a non-finite delta has no magnitude key: the TIES threshold pass refuses it, as the
    statistics pass does (the library reports MP_ERR_NONFINITE)"""
    b = to_bf16(np.zeros(64))
    for bad in [np.nan, np.inf, -np.inf]:
        e = np.zeros(64, np.float32)
        e[40] = bad
        with pytest.raises(oracle.OracleError) as ei:
            oracle.key_hist(oracle.BF16, b, to_bf16(e))
        assert ei.value.rc == oracle.ENONFINITE
        fam = oracle.Family(oracle.BF16, [0], [64], [0], 1, b, [to_bf16(np.zeros(64)), to_bf16(e)])
        with pytest.raises(oracle.OracleError) as ei:
            oracle.ties_thresholds(fam, 0.5)
        assert ei.value.rc == oracle.ENONFINITE


def test_index_family_layout(tiny_family):
    """per-unit statistics land at [expert, block] for every block of every tensor"""
    fam, base, experts = tiny_family
    of = oracle_family(fam, base, experts)
    norm, maxabs, nnz = oracle.index(of)
    bo, bl, _ = fam.block_table()
    rng = np.random.default_rng(0)
    for b in rng.choice(fam.n_blocks, 12, replace=False):
        for i in range(fam.K):
            s = slice(int(bo[b]), int(bo[b]) + int(bl[b]))
            d = experts[i][s] - base[s]
            assert nnz[i, b] == np.count_nonzero(d)
            assert maxabs[i, b] == np.abs(d).max()
            assert norm[i, b] == pytest.approx(np.sqrt((d.astype(np.float64) ** 2).sum()), rel=2e-5)


# ---- TIES thresholds --------------------------------------------------------------------------------

@pytest.mark.parametrize("density", [0.2, 0.5, 0.9, 1.0, 1e-9, 0.0])
def test_tau_is_kth_largest_key(density):
    rng = np.random.default_rng(7)
    n = 5000
    base = to_bf16(rng.standard_normal(n) * 0.02)
    d = rng.standard_normal(n) * 1e-3
    d[rng.random(n) < 0.3] = 0.0
    exp = to_bf16(bf16_to_f32(base) + d.astype(np.float32))
    delta = bf16_to_f32(exp) - bf16_to_f32(base)
    keys = (bf16_bits_torch(np.abs(delta)) & 0x7FFF).astype(np.int64)
    k = int(math.floor(float(np.float32(density)) * n))
    want = oracle.TAU_NONE if k == 0 else int(np.sort(keys)[::-1][k - 1])
    hist = oracle.key_hist(oracle.BF16, base, exp)
    assert int(hist.sum()) == n
    assert oracle.tau_from_hist(hist, n, density) == want
    if k > 0:
        assert (keys >= want).sum() >= k          # every key tied at tau is kept
        assert (keys > want).sum() < k


def test_tau_per_tensor_and_per_expert_scope(tiny_family):
    fam, base, experts = tiny_family
    bo, bl, bt = fam.block_table()
    for scope in (0, 1):
        of = oracle_family(fam, base, experts, trim_scope=scope)
        tau = oracle.ties_thresholds(of, 0.2)
        offs, nums, _ = fam.layout()
        for i in (0, fam.K - 1):
            if scope == 0:
                for t in (0, len(fam.tensors) - 1):
                    s = slice(int(offs[t]), int(offs[t] + nums[t]))
                    keys = (bf16_bits_torch(np.abs(experts[i][s] - base[s])) & 0x7FFF).astype(np.int64)
                    k = int(math.floor(float(np.float32(0.2)) * keys.size))
                    assert tau[i, t] == np.sort(keys)[::-1][k - 1]
            else:
                keys = (bf16_bits_torch(np.abs(experts[i] - base)) & 0x7FFF).astype(np.int64)
                k = int(math.floor(float(np.float32(0.2)) * keys.size))
                assert tau[i, 0] == np.sort(keys)[::-1][k - 1]


# ---- merge operators: worked examples -----------------------------------------------------------------

def _load(name):
    with open(os.path.join(GOLD, name)) as f:
        return json.load(f)


def test_ties_worked_example():
    g = _load("ties_worked.json")
    base = np.array(g["base"], np.float32)
    experts = [to_bf16(base + np.array(d, np.float32)) for d in g["deltas"]]
    b = to_bf16(base)
    for e, d in zip(experts, g["deltas"]):
        assert np.array_equal(bf16_to_f32(e) - bf16_to_f32(b), np.array(d, np.float32))
    tau = [oracle.tau_from_hist(oracle.key_hist(oracle.BF16, b, e), 6, g["density"]) for e in experts]
    assert tau == [oracle.ties_key(v) for v in g["tau_keys_of"]]
    op = oracle.Op(oracle.TIES, 3, lam=1.0, density=g["density"])
    full = oracle.merge_block(oracle.BF16, 0, b, experts, 0b111, op, tau)
    assert np.array_equal(bf16_to_f32(full), np.array(g["expected_full"], np.float32))
    part = oracle.merge_block(oracle.BF16, 0, b, [experts[0], None, experts[2]], g["mask_partial"], op, tau)
    assert np.array_equal(bf16_to_f32(part), np.array(g["expected_partial"], np.float32))
    # the omitted expert counts as zero whatever its data: the same result with it present
    wild = to_bf16(np.full(6, 1000.0))
    for omitted in (experts[1], wild):
        part = oracle.merge_block(oracle.BF16, 0, b, [experts[0], omitted, experts[2]], g["mask_partial"], op, tau)
        assert np.array_equal(bf16_to_f32(part), np.array(g["expected_partial"], np.float32))


def test_avg_worked_example():
    g = _load("avg_worked.json")
    base = np.array(g["base"], np.float32)
    experts = [to_bf16(base + np.array(d, np.float32)) for d in g["deltas"]]
    b = to_bf16(base)
    op = oracle.Op(oracle.AVG, 3, alpha=g["alpha"])
    full = oracle.merge_block(oracle.BF16, 0, b, experts, 0b111, op)
    assert np.array_equal(bf16_to_f32(full), np.array(g["expected_full"], np.float32))
    part = oracle.merge_block(oracle.BF16, 0, b, [experts[0], experts[1], None], g["mask_partial"], op)
    assert np.array_equal(bf16_to_f32(part), np.array(g["expected_partial"], np.float32))
    # the omitted expert counts as zero whatever its data: the same result with it present
    wild = to_bf16(np.full(len(base), -1000.0))
    for omitted in (experts[2], wild):
        part = oracle.merge_block(oracle.BF16, 0, b, [experts[0], experts[1], omitted], g["mask_partial"], op)
        assert np.array_equal(bf16_to_f32(part), np.array(g["expected_partial"], np.float32))


def test_ties_special_cases():
    rng = np.random.default_rng(11)
    n = 777
    base = to_bf16(rng.standard_normal(n) * 0.02)
    # K = 1, rho = 1: every delta kept, its sign elected, mean = itself -> the expert back
    e = to_bf16(bf16_to_f32(base) + (rng.standard_normal(n) * 1e-2).astype(np.float32))
    op = oracle.Op(oracle.TIES, 1, lam=1.0, density=1.0)
    tau = [oracle.tau_from_hist(oracle.key_hist(oracle.BF16, base, e), n, 1.0)]
    out = oracle.merge_block(oracle.BF16, 0, base, [e], 1, op, tau)
    assert np.array_equal(out, e)
    # all experts same-signed: result is base + mean of the kept (nonzero) deltas
    mags = [np.abs(rng.standard_normal(n)).astype(np.float32) * np.float32(2.0 ** -8) for _ in range(3)]
    mags = [np.round(m * 1024) / 1024 for m in mags]   # dyadic, exact sums
    mags[1][::3] = 0.0
    bz = to_bf16(np.zeros(n))
    ex = [to_bf16(m) for m in mags]
    op3 = oracle.Op(oracle.TIES, 3, lam=1.0, density=1.0)
    tau3 = [0, 0, 0]
    out = bf16_to_f32(oracle.merge_block(oracle.BF16, 0, bz, ex, 0b111, op3, tau3))
    dm = np.stack([bf16_to_f32(x) for x in ex]).astype(np.float64)
    cnt = (dm > 0).sum(0)
    want = np.where(cnt > 0, dm.sum(0) / np.maximum(cnt, 1), 0.0)
    assert np.array_equal(out, bf16_to_f32(to_bf16(want.astype(np.float32))))


# ---- Eq. 5: full-budget Psi equals an fp64 restatement of Phi -----------------------------------------

def _fp64_avg(base, experts, alpha):
    x0 = bf16_to_f32(base).astype(np.float64)
    acc = sum(a * (bf16_to_f32(e).astype(np.float64) - x0) for a, e in zip(alpha, experts))
    return x0 + acc


def test_full_read_avg_within_one_ulp_of_fp64(tiny_family):
    rng = np.random.default_rng(5)
    n = 20000
    base = to_bf16(rng.standard_normal(n) * 0.02)
    experts = [to_bf16(bf16_to_f32(base) + (rng.standard_normal(n) * 10 ** rng.uniform(-4, -2)).astype(np.float32))
               for _ in range(5)]
    alpha = np.full(5, 0.3, np.float32)
    op = oracle.Op(oracle.TA, 5, alpha=alpha)
    out = bf16_to_f32(oracle.merge_block(oracle.BF16, 0, base, experts, 0b11111, op)).astype(np.float64)
    ref = _fp64_avg(base, experts, alpha.astype(np.float64))
    ulp = np.abs(bf16_to_f32(to_bf16(ref.astype(np.float32)))).astype(np.float64) * 2.0 ** -7
    assert np.all(np.abs(out - ref) <= ulp + 1e-30)


def test_full_read_ties_matches_fp64_away_from_sign_ties():
    rng = np.random.default_rng(6)
    n, K = 20000, 4
    base = to_bf16(rng.standard_normal(n) * 0.02)
    experts = [to_bf16(bf16_to_f32(base) + (rng.standard_normal(n) * 3e-3).astype(np.float32)) for _ in range(K)]
    dens = 0.3
    taus = [oracle.tau_from_hist(oracle.key_hist(oracle.BF16, base, e), n, dens) for e in experts]
    op = oracle.Op(oracle.TIES, K, lam=1.0, density=dens)
    out = bf16_to_f32(oracle.merge_block(oracle.BF16, 0, base, experts, (1 << K) - 1, op, taus)).astype(np.float64)
    x0 = bf16_to_f32(base).astype(np.float64)
    d = np.stack([bf16_to_f32(e).astype(np.float64) - x0 for e in experts])
    keys = np.stack([(bf16_bits_torch(np.abs(di.astype(np.float32))) & 0x7FFF) for di in d]).astype(np.int64)
    dh = np.where(keys >= np.array(taus)[:, None], d, 0.0)
    S = dh.sum(0)
    pos, neg = (dh > 0), (dh < 0)
    m = np.where(S > 0, (dh * pos).sum(0) / np.maximum(pos.sum(0), 1),
                 np.where(S < 0, (dh * neg).sum(0) / np.maximum(neg.sum(0), 1), 0.0))
    ref = x0 + m
    safe = np.abs(S) > 1e-6 * np.abs(dh).sum(0) + 1e-30
    safe |= (dh == 0).all(0)
    assert safe.mean() > 0.99
    ulp = np.abs(ref) * 2.0 ** -7 + 1e-30
    assert np.all(np.abs(out - ref)[safe] <= ulp[safe])


def test_ties_per_tensor_trim_is_separable(tiny_family):
    """With one trim group per tensor, each tensor's trim, election and mean involve that
    tensor alone: the whole family's TIES merge equals, tensor by tensor, the merge of that
    tensor taken as a family of its own (its own threshold, its own element numbering)."""
    fam, base, experts = tiny_family
    of = oracle_family(fam, base, experts)
    bo, bl, bt = fam.block_table()
    dens = 0.2
    tau = oracle.ties_thresholds(of, dens)
    assert len(set(tau[0].tolist())) > 1            # the tensors' thresholds differ
    op = oracle.Op(oracle.TIES, fam.K, lam=0.8, density=dens)
    whole = oracle.merge(of, op, tau=tau)
    for t in range(len(fam.tensors)):
        blocks = np.nonzero(bt == t)[0]
        lo, hi = int(bo[blocks[0]]), int(bo[blocks[-1]] + bl[blocks[-1]])
        sub = oracle.Family(fam.dtype, bo[blocks] - lo, bl[blocks], np.zeros(len(blocks), np.uint32), 1,
                            base[lo:hi], [e[lo:hi] for e in experts])
        alone = oracle.merge(sub, op, tau=oracle.ties_thresholds(sub, dens))
        assert np.array_equal(whole[lo:hi].view(np.uint32), alone.view(np.uint32)), t


# ---- Prop. 2: additive omission bound ------------------------------------------------------------------

def test_additive_omission_bound(tiny_family):
    fam, base, experts = tiny_family
    of = oracle_family(fam, base, experts)
    norm, maxabs, nnz = oracle.index(of)
    bo, bl, bt = fam.block_table()
    alpha = np.full(fam.K, 0.25, np.float32)
    op = oracle.Op(oracle.AVG, fam.K, alpha=alpha)
    full = oracle.merge(of, op).astype(np.float64)
    x0 = base.astype(np.float64)
    exact_norm = np.zeros((fam.K, fam.n_blocks))
    for i in range(fam.K):
        d = experts[i].astype(np.float64) - x0
        for b in range(fam.n_blocks):
            s = slice(int(bo[b]), int(bo[b] + bl[b]))
            exact_norm[i, b] = np.sqrt((d[s] ** 2).sum())
    C_full = fam.K * fam.total_elems * 4
    for f in (1.0, 0.5, 0.25, 0.1, 0.0):
        B = int(math.floor(f * C_full))
        pl = oracle.plan(fam.K, bl, bt, len(fam.tensors), 4, op, norm, maxabs, nnz, None, B)
        assert pl["chat"] <= B
        out = oracle.merge(of, op, mask=pl["mask"]).astype(np.float64)
        A = ((pl["mask"][None, :] >> np.arange(fam.K)[:, None]) & 1).astype(np.float64)
        q = ((1 - A) * np.abs(alpha[:, None]) * exact_norm).sum(0)
        lhs = np.sqrt(((full - out) ** 2).sum())
        slack = 4 * 2.0 ** -24 * np.sqrt((full ** 2).sum())
        assert lhs <= np.sqrt((q ** 2).sum()) + slack
        assert np.sqrt((q ** 2).sum()) <= q.sum() + 1e-12
        if f == 1.0:
            assert lhs == 0.0


# ---- DARE --------------------------------------------------------------------------------------------

def test_dare_p0_equals_avg():
    rng = np.random.default_rng(9)
    n = 3001
    base = to_bf16(rng.standard_normal(n) * 0.02)
    experts = [to_bf16(bf16_to_f32(base) + (rng.standard_normal(n) * 1e-3).astype(np.float32)) for _ in range(3)]
    alpha = [0.25, 0.5, 0.25]
    a = oracle.merge_block(oracle.BF16, 123, base, experts, 0b111, oracle.Op(oracle.AVG, 3, alpha=alpha))
    d = oracle.merge_block(oracle.BF16, 123, base, experts, 0b111,
                           oracle.Op(oracle.DARE, 3, alpha=alpha, drop_p=0.0, seed=99))
    assert np.array_equal(a, d)


def test_dare_keep_fraction_binomial_band():
    p = 0.9
    T = math.floor(p * 65536)
    q = 1.0 - T / 65536.0
    n = 40000
    for expert in (0, 5):
        kept = sum(oracle.dare_keep(1234, expert, j, p) for j in range(n))
        sd = math.sqrt(n * q * (1 - q))
        assert abs(kept - n * q) < 5 * sd


def test_dare_mean_over_seeds_tends_to_avg():
    rng = np.random.default_rng(10)
    n = 512
    base = (rng.standard_normal(n) * 0.02).astype(np.float32)
    experts = [base + (rng.standard_normal(n) * 1e-2).astype(np.float32) for _ in range(2)]
    alpha = [0.5, 0.5]
    seeds = 400
    acc = np.zeros(n)
    for s in range(seeds):
        o = oracle.merge_block(oracle.F32, 0, base, experts, 0b11, oracle.Op(oracle.DARE, 2, alpha=alpha, drop_p=0.5, seed=s))
        acc += o.astype(np.float64) - base
    avg = oracle.merge_block(oracle.F32, 0, base, experts, 0b11, oracle.Op(oracle.AVG, 2, alpha=alpha)).astype(np.float64) - base
    # per element: mean of 400 draws of sum_i a_i * 2 * Bern(.5) * d_i; sd of the mean <= sum |a_i d_i| / sqrt(400)
    sd = sum(abs(a) * np.abs(e.astype(np.float64) - base) for a, e in zip(alpha, experts)) / math.sqrt(seeds)
    assert np.all(np.abs(acc / seeds - avg) <= 5 * sd + 1e-9)


def test_dare_p0_never_drops_over_many_entries():
    """p = 0 drops nothing, whatever the random word: over 2^21 + 6 entries (so every 16-bit
    word value, 0 included, comes up many times) DARE is AVG bit for bit"""
    rng = np.random.default_rng(21)
    n = (1 << 20) + 3
    base = (rng.standard_normal(n) * 0.02).astype(np.float32)
    experts = [base + (rng.standard_normal(n) * 1e-3).astype(np.float32) for _ in range(2)]
    alpha = [0.5, 0.5]
    a = oracle.merge_block(oracle.F32, 77, base, experts, 0b11, oracle.Op(oracle.AVG, 2, alpha=alpha))
    d = oracle.merge_block(oracle.F32, 77, base, experts, 0b11,
                           oracle.Op(oracle.DARE, 2, alpha=alpha, drop_p=0.0, seed=5))
    assert np.array_equal(a.view(np.uint32), d.view(np.uint32))


def test_dare_drops_independently_across_blocks():
    """App. A.1's DARE drops each entry at random: two blocks holding the same deltas at
    different places in the checkpoint get different drop patterns (at p = 0.5 the chance
    that 4096 independent draws agree is 2^-4096)"""
    rng = np.random.default_rng(22)
    E = 4096
    b = (rng.standard_normal(E) * 0.02).astype(np.float32)
    e = b + (rng.standard_normal(E) * 1e-2).astype(np.float32)
    base, expert = np.concatenate([b, b]), np.concatenate([e, e])
    fam = oracle.Family(oracle.F32, [0, E], [E, E], [0, 0], 1, base, [expert])
    out = oracle.merge(fam, oracle.Op(oracle.DARE, 1, alpha=[1.0], drop_p=0.5, seed=3))
    kept0, kept1 = out[:E] != b, out[E:] != b
    assert 0.4 < kept0.mean() < 0.6 and 0.4 < kept1.mean() < 0.6
    assert not np.array_equal(kept0, kept1)


def test_philox_word_statistics():
    """uniform 16-bit words, independent across counters (chi-square on 256 bins, 4 outputs)"""
    words = []
    for g in range(4096):
        w = oracle.philox4x32_10([g, 0, 3, 0x44415245], [17, 0])
        for x in w:
            words += [int(x) & 0xFFFF, int(x) >> 16]
    h = np.bincount(np.array(words) >> 8, minlength=256)
    exp = len(words) / 256
    chi2 = ((h - exp) ** 2 / exp).sum()
    assert chi2 < 255 + 5 * math.sqrt(2 * 255)
    a = oracle.philox4x32_10([0, 0, 0, 0], [0, 0])
    b = oracle.philox4x32_10([1, 0, 0, 0], [0, 0])
    c = oracle.philox4x32_10([0, 0, 0, 0], [1, 0])
    assert not np.array_equal(a, b) and not np.array_equal(a, c)


def _curand_host():
    """cuRAND's host-side generator library (it runs on the CPU; no GPU is touched)"""
    import ctypes
    import ctypes.util
    names = [os.path.join(os.environ.get("CUDA_HOME", "/usr/local/cuda"), "lib64", "libcurand.so"),
             ctypes.util.find_library("curand")]
    for n in names:
        if n and (os.path.exists(n) or not os.path.isabs(n)):
            try:
                return ctypes.CDLL(n)
            except OSError:
                pass
    pytest.skip("libcurand is not available")


def _curand_host_philox(L, seed, offset, n_words):
    import ctypes
    gen = ctypes.c_void_p()
    assert L.curandCreateGeneratorHost(ctypes.byref(gen), 161) == 0  # CURAND_RNG_PSEUDO_PHILOX4_32_10
    try:
        assert L.curandSetPseudoRandomGeneratorSeed(gen, ctypes.c_ulonglong(seed)) == 0
        assert L.curandSetGeneratorOffset(gen, ctypes.c_ulonglong(offset)) == 0
        out = np.zeros(n_words, np.uint32)
        assert L.curandGenerate(gen, out.ctypes.data_as(ctypes.c_void_p), ctypes.c_size_t(n_words)) == 0
    finally:
        L.curandDestroyGenerator(gen)
    return out


def test_philox_matches_curand_host_generator():
    """Philox4x32-10 against an independent implementation of the same published generator:
    cuRAND's host generator, run on the CPU.  For seed s it emits 4-word blocks; block j
    (j = the starting offset / 4 + the block's position) is Philox of the counter
    (lo32(j >> 16), hi32(j >> 16), j & 0xFFFF, 0) under the key (lo32(s), hi32(s)).  That
    reaches counter words 0-2 and both key words; word 3, which the DARE stream fixes to a
    tag, is pinned against cuRAND's device generator in the GPU suite."""
    L = _curand_host()

    def ctr_of(j):
        r = j >> 16
        return [r & 0xFFFFFFFF, r >> 32, j & 0xFFFF, 0]

    for seed in (0, 1, 2605, 0x0123456789ABCDEF, 0xFFFFFFFFFFFFFFFF):
        key = [seed & 0xFFFFFFFF, seed >> 32]
        # a run of blocks across the first change of counter word 0 (j = 65535 -> 65536)
        j0 = 65536 - 3
        got = _curand_host_philox(L, seed, 4 * j0, 4 * 6).reshape(-1, 4)
        for b in range(6):
            assert np.array_equal(oracle.philox4x32_10(ctr_of(j0 + b), key), got[b]), (seed, j0 + b)
        # large offsets: counter words 0 and 1 both nonzero, and all ones in word 0
        for j in ((5 << 48) + (7 << 16) + 9, (1 << 61) + 3, (0xFFFFFFFF << 16) + 11, (1 << 62) - 1):
            got = _curand_host_philox(L, seed, 4 * j, 4)
            assert np.array_equal(oracle.philox4x32_10(ctr_of(j), key), got), (seed, hex(j))


# ---- Alg. 1 PlanGen ------------------------------------------------------------------------------------

def _tiny_plan_case(rng, K, nb, uniform):
    blk_len = np.full(nb, 8, np.uint32) if uniform else rng.integers(1, 9, nb).astype(np.uint32)
    norm = rng.choice([0.5, 1.0, 1.5, 2.0, 3.0], (K, nb)).astype(np.float32)
    nnz = (rng.random((K, nb)) > 0.2).astype(np.uint32) * 5
    maxabs = norm.copy()
    alpha = rng.choice([0.25, 0.5, 1.0], K).astype(np.float32)
    return blk_len, norm, maxabs, nnz, alpha


def test_plan_brute_force_tiny():
    rng = np.random.default_rng(12)
    for trial in range(60):
        K, nb = int(rng.integers(1, 4)), int(rng.integers(1, 5))
        uniform = trial % 2 == 0
        blk_len, norm, maxabs, nnz, alpha = _tiny_plan_case(rng, K, nb, uniform)
        op = oracle.Op(oracle.AVG, K, alpha=alpha)
        units = [(b, i) for b in range(nb) for i in range(K) if nnz[i, b] > 0]
        score = {u: np.float32(abs(alpha[u[1]])) * norm[u[1], u[0]] for u in units}
        cost = {u: int(blk_len[u[0]]) * 2 for u in units}
        total = sum(cost.values())
        for B in sorted(set([0, total, total // 2, total // 3, int(rng.integers(0, total + 1))])):
            pl = oracle.plan(K, blk_len, np.zeros(nb, np.uint32), 1, 2, op, norm, maxabs, nnz, None, B)
            sel = [(b, i) for b in range(nb) for i in range(K) if (pl["mask"][b] >> i) & 1]
            assert set(sel) <= set(units)
            assert pl["chat"] == sum(cost[u] for u in sel) <= B          # Prop. 1
            assert pl["n_cand"] == len(units) and pl["n_sel"] == len(sel)
            # traversal order: decreasing score, ties by ascending unit id b*K+i
            order = [(int(u) // K, int(u) % K) for u in pl["order"]]
            assert sorted(order) == sorted(units)
            assert all((-score[x], x[0] * K + x[1]) < (-score[y], y[0] * K + y[1]) for x, y in zip(order, order[1:]))
            # greedy-with-skip characterisation along that order
            run = 0
            for u in order:
                if u in sel:
                    assert run + cost[u] <= B
                    run += cost[u]
                else:
                    assert run + cost[u] > B
            if B >= total:
                assert set(sel) == set(units)
            if uniform and units:
                # equal costs: greedy is optimal for Eq. 6 (cardinality knapsack); brute force
                best = 0.0
                for r in range(len(units) + 1):
                    for comb in itertools.combinations(units, r):
                        if sum(cost[u] for u in comb) <= B:
                            best = max(best, sum(float(score[u]) for u in comb))
                got = sum(float(score[u]) for u in sel)
                assert got == pytest.approx(best, rel=1e-6)


def test_plan_monotone_in_budget_with_equal_costs():
    rng = np.random.default_rng(13)
    K, nb = 3, 40
    blk_len, norm, maxabs, nnz, alpha = _tiny_plan_case(rng, K, nb, True)
    op = oracle.Op(oracle.TA, K, alpha=alpha)
    prev_sel, prev_c = set(), 0
    for B in range(0, 16 * K * nb + 1, 16 * 3):
        pl = oracle.plan(K, blk_len, np.zeros(nb, np.uint32), 1, 2, op, norm, maxabs, nnz, None, B)
        sel = {(b, i) for b in range(nb) for i in range(K) if (pl["mask"][b] >> i) & 1}
        assert pl["chat"] >= prev_c and prev_sel <= sel
        prev_sel, prev_c = sel, pl["chat"]


def test_plan_ties_prunes_fully_trimmed_units():
    K, nb = 2, 3
    blk_len = np.full(nb, 4, np.uint32)
    norm = np.ones((K, nb), np.float32)
    maxabs = np.array([[0.5, 0.25, 1.0], [2.0 ** -20, 0.5, 0.5]], np.float32)
    nnz = np.full((K, nb), 4, np.uint32)
    tau = np.array([[oracle.ties_key(0.5)], [oracle.ties_key(0.5)]], np.uint32)
    op = oracle.Op(oracle.TIES, K, lam=1.0, density=0.2)
    pl = oracle.plan(K, blk_len, np.zeros(nb, np.uint32), 1, 2, op, norm, maxabs, nnz, tau, 10 ** 9)
    assert list(pl["mask"]) == [0b01, 0b10, 0b11]


def test_plan_ties_candidates_are_units_with_a_surviving_entry(tiny_family):
    """TIES pruning is exact, per trim group: with one group per tensor, a unit is a
    candidate iff some entry of it survives its own tensor's trim, i.e. the largest bf16
    magnitude key among its deltas (computed here with torch from the data) reaches tau of
    (its expert, its tensor).  The tensors' thresholds differ, so a unit judged against
    another tensor's tau shows."""
    fam, base, experts = tiny_family
    of = oracle_family(fam, base, experts)
    bo, bl, bt = fam.block_table()
    norm, maxabs, nnz = oracle.index(of)
    dens = 0.2
    tau = oracle.ties_thresholds(of, dens)
    assert len(set(tau[0].tolist())) > 1
    want = set()
    for i, e in enumerate(experts):
        d = e.astype(np.float32) - base.astype(np.float32)
        keys = (bf16_bits_torch(np.abs(d)) & 0x7FFF).astype(np.int64)
        for b in range(len(bl)):
            blk = keys[int(bo[b]):int(bo[b] + bl[b])]
            if nnz[i, b] > 0 and blk.max() >= tau[i, bt[b]]:
                want.add(b * fam.K + i)
    op = oracle.Op(oracle.TIES, fam.K, lam=1.0, density=dens)
    full = fam.K * int(bl.sum()) * 4
    p = oracle.plan(fam.K, bl, bt, len(fam.tensors), 4, op, norm, maxabs, nnz, tau, full)
    assert 0 < len(want) < fam.K * len(bl)
    assert set(p["order"].tolist()) == want and p["n_cand"] == len(want) and p["n_sel"] == len(want)


def test_plan_is_invariant_under_relabelling():
    """Alg. 1 looks only at scores and costs: with distinct scores, relabelling the experts
    (statistics and coefficients together) or reordering the blocks relabels the selection,
    the traversal order and C_hat in the same way"""
    rng = np.random.default_rng(41)
    for trial in range(25):
        K, nb = int(rng.integers(2, 6)), int(rng.integers(3, 30))
        blk_len = rng.integers(1, 9, nb).astype(np.uint32)
        norm = rng.uniform(0.1, 4.0, (K, nb)).astype(np.float32)
        nnz = (rng.random((K, nb)) > 0.15).astype(np.uint32) * 3
        alpha = rng.uniform(0.2, 1.0, K).astype(np.float32)
        pe, pb = rng.permutation(K), rng.permutation(nb)      # expert i -> pe[i], block b -> pb[b]
        norm2, nnz2 = np.empty_like(norm), np.empty_like(nnz)
        norm2[pe[:, None], pb[None, :]] = norm
        nnz2[pe[:, None], pb[None, :]] = nnz
        alpha2 = np.empty_like(alpha)
        alpha2[pe] = alpha
        len2 = np.empty_like(blk_len)
        len2[pb] = blk_len
        total = int(blk_len.sum()) * K * 2
        for B in (0, total // 5, total // 2, total):
            a = oracle.plan(K, blk_len, np.zeros(nb, np.uint32), 1, 2, oracle.Op(oracle.TA, K, alpha=alpha),
                            norm, norm, nnz, None, B)
            b = oracle.plan(K, len2, np.zeros(nb, np.uint32), 1, 2, oracle.Op(oracle.TA, K, alpha=alpha2),
                            norm2, norm2, nnz2, None, B)
            sel_a = {(int(pb[bb]), int(pe[i])) for bb in range(nb) for i in range(K) if (a["mask"][bb] >> i) & 1}
            sel_b = {(bb, i) for bb in range(nb) for i in range(K) if (b["mask"][bb] >> i) & 1}
            assert sel_a == sel_b and a["chat"] == b["chat"] and a["n_cand"] == b["n_cand"]
            order_a = [(int(pb[u // K]), int(pe[u % K])) for u in a["order"].tolist()]
            order_b = [(u // K, u % K) for u in b["order"].tolist()]
            assert order_a == order_b


def test_plan_depends_on_coefficient_magnitudes_only():
    """The utility of a unit is |coef| * ||Delta|| (Prop. 2): flipping the sign of some
    experts' coefficients leaves the order and the selection unchanged, and scaling one
    expert's coefficient moves its units in the order"""
    rng = np.random.default_rng(31)
    for trial in range(20):
        K, nb = 3, 12
        blk_len, norm, maxabs, nnz, alpha = _tiny_plan_case(rng, K, nb, trial % 2 == 0)
        signs = np.where(rng.random(K) < 0.5, -1.0, 1.0).astype(np.float32)
        signs[0] = -1.0
        B = int(rng.integers(0, int(blk_len.sum()) * K * 2 + 1))
        for sm in (0, 1):
            a = oracle.plan(K, blk_len, np.zeros(nb, np.uint32), 1, 2, oracle.Op(oracle.TA, K, alpha=alpha, score_mode=sm),
                            norm, maxabs, nnz, None, B)
            b = oracle.plan(K, blk_len, np.zeros(nb, np.uint32), 1, 2,
                            oracle.Op(oracle.TA, K, alpha=alpha * signs, score_mode=sm), norm, maxabs, nnz, None, B)
            assert np.array_equal(a["order"], b["order"]) and np.array_equal(a["mask"], b["mask"])
            assert a["chat"] == b["chat"] and a["set_hash"] == b["set_hash"]
    # expert 1's coefficient x 4 lifts its unit above expert 0's (norms 1.0 vs 2.0, unit ids 0 and 1)
    blk_len = np.full(1, 4, np.uint32)
    norm = np.array([[2.0], [1.0]], np.float32)
    nnz = np.full((2, 1), 4, np.uint32)
    for al, want in (([1.0, 1.0], [0, 1]), ([1.0, -4.0], [1, 0])):
        p = oracle.plan(2, blk_len, np.zeros(1, np.uint32), 1, 2, oracle.Op(oracle.TA, 2, alpha=al), norm, norm, nnz,
                        None, 8)
        assert p["order"].tolist() == want and p["mask"].tolist() == [1 << want[0]]


# ---- digest ----------------------------------------------------------------------------------------------

def test_fnv1a_published_vectors():
    assert oracle.fnv1a64(b"") == 0xCBF29CE484222325
    assert oracle.fnv1a64(b"a") == 0xAF63DC4C8601EC8C
    assert oracle.fnv1a64(b"foobar") == 0x85944171F73967E8


def test_splitmix64_reference_output():
    assert oracle.splitmix64(0) == 0xE220A8397B1DCDAF


def test_digest_tracks_selection():
    rng = np.random.default_rng(14)
    K, nb = 3, 30
    blk_len, norm, maxabs, nnz, alpha = _tiny_plan_case(rng, K, nb, False)
    op = oracle.Op(oracle.AVG, K, alpha=alpha)
    g = np.zeros(nb, np.uint32)
    p1 = oracle.plan(K, blk_len, g, 1, 2, op, norm, maxabs, nnz, None, 200)
    p2 = oracle.plan(K, blk_len, g, 1, 2, op, norm, maxabs, nnz, None, 200)
    p3 = oracle.plan(K, blk_len, g, 1, 2, op, norm, maxabs, nnz, None, 150)
    assert p1["digest"] == p2["digest"]
    assert p1["digest"] != p3["digest"]
    sel = [b * K + i for b in range(nb) for i in range(K) if (p1["mask"][b] >> i) & 1]
    assert p1["set_hash"] == sum(oracle.splitmix64(u) for u in sel) % 2 ** 64


def test_plan_score_per_byte_worked_example():
    """Hand-worked: one expert, three blocks of 50, 25 and 25 bf16 elements (costs 100, 50 and
    50 bytes) with norms 10, 6 and 6, budget 100 bytes.  By score the order is block 0, 1, 2:
    block 0 fills the budget and the others are skipped (utility 10).  By score per byte the
    densities are 0.10, 0.12 and 0.12: blocks 1 and 2 come first and both fit (utility 12)."""
    blk_len = [50, 25, 25]
    norm = np.array([[10.0, 6.0, 6.0]], np.float32)
    maxabs = np.ones((1, 3), np.float32)
    nnz = np.ones((1, 3), np.uint32)
    args = (1, blk_len, [0, 0, 0], 1, 2)
    by_score = oracle.plan(*args, oracle.Op(oracle.AVG, 1, alpha=[1.0]), norm, maxabs, nnz, None, 100)
    per_byte = oracle.plan(*args, oracle.Op(oracle.AVG, 1, alpha=[1.0], score_mode=1), norm, maxabs, nnz, None, 100)
    assert by_score["mask"].tolist() == [1, 0, 0] and by_score["chat"] == 100 and by_score["order"].tolist() == [0, 1, 2]
    assert per_byte["mask"].tolist() == [0, 1, 1] and per_byte["chat"] == 100 and per_byte["order"].tolist() == [1, 2, 0]
    assert by_score["digest"] != per_byte["digest"]   # the mode is part of the plan's identity


def test_plan_score_per_byte_equal_power_of_two_costs_same_selection():
    """with every block of the same power-of-two byte cost, dividing by it is an exact scaling
    of every score, so the order and the selection equal those of the plain score"""
    rng = np.random.default_rng(11)
    K, nb = 3, 40
    blk_len = [4096] * nb
    norm = rng.lognormal(size=(K, nb)).astype(np.float32)
    norm[0, :5] = norm[1, :5]          # ties are broken the same way
    maxabs = np.ones((K, nb), np.float32)
    nnz = np.ones((K, nb), np.uint32)
    nnz[2, ::7] = 0
    for budget in (0, 8192 * 10, 8192 * 33, 8192 * K * nb):
        a = oracle.plan(K, blk_len, [0] * nb, 1, 2, oracle.Op(oracle.TA, K, alpha=[0.3, -0.7, 1.1]), norm, maxabs, nnz,
                        None, budget)
        b = oracle.plan(K, blk_len, [0] * nb, 1, 2, oracle.Op(oracle.TA, K, alpha=[0.3, -0.7, 1.1], score_mode=1), norm,
                        maxabs, nnz, None, budget)
        assert np.array_equal(a["mask"], b["mask"]) and np.array_equal(a["order"], b["order"])
        assert a["chat"] == b["chat"] and a["n_sel"] == b["n_sel"]


# ---- operator variants (App. A.1): renormalised AVG, DARE-TIES ----------------------------------------

def test_avg_renorm_worked_example():
    """Hand-worked, fp32 (every value dyadic, every step exact): alpha = (0.5, 0.25, 0.25).
    Experts 1 and 2 selected: s = 0.5, beta = (0, 0.5, 0.5), so out = base + (D1 + D2) / 2.
    All three selected: s = 1, beta = alpha (the plain average)."""
    base = np.array([1.0, -2.0, 0.5, 0.0], np.float32)
    e0 = np.array([9.0, 9.0, 9.0, 9.0], np.float32)      # omitted below: must not matter
    e1 = np.array([2.0, -1.0, 0.5, 1.0], np.float32)     # D1 = ( 1,  1, 0,  1)
    e2 = np.array([1.0, -3.0, 1.5, -1.0], np.float32)    # D2 = ( 0, -1, 1, -1)
    op = oracle.Op(oracle.AVG_RENORM, 3, alpha=[0.5, 0.25, 0.25])
    out = oracle.merge_block(oracle.F32, 0, base, [e0, e1, e2], 0b110, op)
    assert out.tolist() == [1.5, -2.0, 1.0, 0.0]
    out_all = oracle.merge_block(oracle.F32, 0, base, [e0, e1, e2], 0b111, op)
    # base + 0.5*(8,11,8.5,9) + 0.25*(1,1,0,1) + 0.25*(0,-1,1,-1)
    assert out_all.tolist() == [5.25, 3.5, 5.0, 4.5]
    out_none = oracle.merge_block(oracle.F32, 0, base, [e0, e1, e2], 0, op)
    assert out_none.tolist() == base.tolist()


def test_avg_renorm_needs_positive_coefficients():
    """the renormalised average divides by the sum of the taking-part coefficients, which
    needs every coefficient > 0 (else the sum can vanish or flip sign): a zero or negative
    alpha is refused, as the library refuses it"""
    base = np.zeros(8, np.float32)
    ex = [np.full(8, 1.0, np.float32), np.full(8, 2.0, np.float32)]
    for alpha in ([0.5, 0.0], [0.5, -0.5], [-1.0, 1.0]):
        with pytest.raises(oracle.OracleError) as ei:
            oracle.merge_block(oracle.F32, 0, base, ex, 0b11, oracle.Op(oracle.AVG_RENORM, 2, alpha=alpha))
        assert ei.value.rc == oracle.EINVAL
    out = oracle.merge_block(oracle.F32, 0, base, ex, 0b11, oracle.Op(oracle.AVG_RENORM, 2, alpha=[0.5, 0.5]))
    assert out.tolist() == [1.5] * 8


def test_avg_renorm_full_budget_equals_avg(tiny_family):
    """with sum alpha = 1 exactly (0.25 x 4), the full-read renormalised average divides by 1"""
    fam, base, experts = tiny_family
    of = oracle_family(fam, base, experts)
    a = [0.25] * fam.K
    r = oracle.merge(of, oracle.Op(oracle.AVG_RENORM, fam.K, alpha=a))
    m = oracle.merge(of, oracle.Op(oracle.AVG, fam.K, alpha=a))
    assert np.array_equal(r.view(np.uint32), m.view(np.uint32))


def test_avg_renorm_full_budget_plan_equals_avg(tiny_family):
    """Through the plan, as the pipeline runs it: at the full budget the mask holds every
    unit with nnz > 0 but no unit whose delta is exactly zero (those are not candidates).
    The renormalised AVG over that mask, told the zero deltas by the catalog's nnz (or
    finding them in the data), still divides by the sum of all K coefficients, so it equals
    the full-read AVG (Eq. 5).  Each expert here has its own blocks set equal to the base."""
    fam, base, experts = tiny_family
    bo, bl, _ = fam.block_table()
    experts = [e.copy() for e in experts]
    for i, e in enumerate(experts):
        for blk in range(i, len(bl), 7 + i):
            e[int(bo[blk]):int(bo[blk] + bl[blk])] = base[int(bo[blk]):int(bo[blk] + bl[blk])]
    of = oracle_family(fam, base, experts)
    norm, maxabs, nnz = oracle.index(of)
    assert (nnz == 0).any(axis=1).all() and ((nnz == 0).sum(axis=0) < fam.K).all()
    a = [0.25] * fam.K
    op = oracle.Op(oracle.AVG_RENORM, fam.K, alpha=a)
    full = fam.K * int(bl.sum()) * 4
    pl = oracle.plan(fam.K, bl, np.zeros(len(bl), np.uint32), 1, 4, op, norm, maxabs, nnz, None, full)
    assert pl["n_sel"] == int((nnz > 0).sum())
    m = oracle.merge(of, oracle.Op(oracle.AVG, fam.K, alpha=a))
    for catalog in (nnz, None):
        r = oracle.merge(of, op, mask=pl["mask"], nnz=catalog)
        assert np.array_equal(r.view(np.uint32), m.view(np.uint32))


def test_avg_renorm_coefficient_drift_bound(tiny_family):
    """App. A.1: ||M_full - M_A||_2 <= sqrt(sum_b r_b^2), r_b = sum_i |alpha_i - beta_i(A)| ||Delta_i,b||_2,
    checked in fp64 on plans at several budgets (slack for the fp32 arithmetic)"""
    fam, base, experts = tiny_family
    of = oracle_family(fam, base, experts)
    norm, maxabs, nnz = oracle.index(of)
    bo, bl, bt = fam.block_table()
    alpha = np.array([0.4, 0.3, 0.2, 0.1], np.float32)[: fam.K]
    alpha = alpha / alpha.sum()
    op = oracle.Op(oracle.AVG_RENORM, fam.K, alpha=alpha)
    full = oracle.merge(of, op).astype(np.float64)
    x0 = base.astype(np.float64)
    exact_norm = np.zeros((fam.K, fam.n_blocks))
    for i in range(fam.K):
        d = experts[i].astype(np.float64) - x0
        for b in range(fam.n_blocks):
            s = slice(int(bo[b]), int(bo[b] + bl[b]))
            exact_norm[i, b] = np.sqrt((d[s] ** 2).sum())
    C_full = fam.K * fam.total_elems * 4
    checked_drift = False
    for f in (1.0, 0.6, 0.3, 0.1):
        B = int(math.floor(f * C_full))
        pl = oracle.plan(fam.K, bl, bt, len(fam.tensors), 4, op, norm, maxabs, nnz, None, B)
        out = oracle.merge(of, op, mask=pl["mask"]).astype(np.float64)
        A = ((pl["mask"][None, :] >> np.arange(fam.K)[:, None]) & 1).astype(np.float64)
        ssel = (A * alpha.astype(np.float64)[:, None]).sum(0)
        beta = np.where(ssel > 0, A * alpha.astype(np.float64)[:, None] / np.where(ssel > 0, ssel, 1.0), 0.0)
        r = (np.abs(alpha.astype(np.float64)[:, None] - beta) * exact_norm).sum(0)
        lhs = np.sqrt(((full - out) ** 2).sum())
        slack = 8 * 2.0 ** -24 * np.sqrt((full ** 2).sum())
        assert lhs <= np.sqrt((r ** 2).sum()) + slack, f
        checked_drift |= lhs > slack
    assert checked_drift   # some budget actually moved the result


def test_dare_ties_p0_equals_ties_density_one():
    """p = 0 keeps every delta with sigma = 1, and TIES at density 1 trims nothing: the two
    are the same operator (election, disjoint mean, lambda)"""
    rng = np.random.default_rng(21)
    n, K = 1500, 5
    base = to_bf16(rng.standard_normal(n) * 0.02)
    ex = [to_bf16(bf16_to_f32(base) + (rng.standard_normal(n) * 1e-2 * (k + 1)).astype(np.float32)) for k in range(K)]
    for k in range(K):
        z = rng.random(n) < 0.3
        ex[k][z] = base[z]   # some exact zero deltas
    taus = [oracle.tau_from_hist(oracle.key_hist(oracle.BF16, base, e), n, 1.0) for e in ex]
    for mask in (0b11111, 0b10110, 0b00001):
        t = oracle.merge_block(oracle.BF16, 0, base, ex, mask, oracle.Op(oracle.TIES, K, lam=0.7, density=1.0), taus)
        d = oracle.merge_block(oracle.BF16, 0, base, ex, mask,
                               oracle.Op(oracle.DARE_TIES, K, lam=0.7, drop_p=0.0, seed=5))
        assert np.array_equal(t, d), mask


def test_dare_ties_uses_the_dare_mask():
    """an element whose every selected delta is dropped by the (cuRAND-pinned) keep mask
    stays at the base; an element with exactly one kept nonzero delta gets
    fma(lambda, delta * sigma, base), the mean of a single entry"""
    rng = np.random.default_rng(22)
    n, K, p, seed, j0 = 4096, 3, 0.6, 77, 8 * 1000
    base = to_bf16(rng.standard_normal(n) * 0.02)
    ex = [to_bf16(bf16_to_f32(base) + (rng.standard_normal(n) * 1e-2).astype(np.float32)) for _ in range(K)]
    op = oracle.Op(oracle.DARE_TIES, K, lam=0.9, drop_p=p, seed=seed)
    out = bf16_to_f32(oracle.merge_block(oracle.BF16, j0, base, ex, 0b111, op))
    keep = np.array([[oracle.dare_keep(seed, i, j0 + k, p) for k in range(n)] for i in range(K)])
    x0 = bf16_to_f32(base)
    d = np.stack([bf16_to_f32(e) - x0 for e in ex])
    sigma = np.float32(1.0 / (1.0 - p))
    none = ~keep.any(0)
    assert none.any() and np.array_equal(out[none], x0[none])
    one = (keep & (d != 0)).sum(0) == 1
    assert one.any()
    for k in np.nonzero(one)[0][:200]:
        i = int(np.nonzero(keep[:, k] & (d[:, k] != 0))[0][0])
        v = np.float32(d[i, k] * sigma)
        want = np.float32(np.float64(np.float32(0.9)) * np.float64(v) + np.float64(x0[k]))  # one rounding (fma)
        assert out[k] == bf16_to_f32(to_bf16(np.array([want], np.float32)))[0], k


# ---- tensor-level fallback (Sec. 3 Planner; Alg. 1 scoring with fallback metadata) -----------------------

MISS = oracle.NNZ_MISSING


def _fallback_worked_catalog():
    """two experts over two tensors: t0 = blocks 0-2, t1 = blocks 3-4, 4 bf16 elements (8 bytes)
    each.  Expert 0 has no statistics for block 2, expert 1 none for block 4."""
    blk_len = np.full(5, 4, np.uint32)
    blk_tensor = np.array([0, 0, 0, 1, 1], np.uint32)
    norm = np.array([[3.0, 4.0, 99.0, 1.0, 2.0],
                     [1.0, 1.0, 1.0, 6.0, 99.0]], np.float32)
    nnz = np.array([[4, 4, MISS, 4, 4],
                    [4, 4, 4, 4, MISS]], np.uint32)
    return blk_len, blk_tensor, norm, nnz


def _fallback_plan(budget, score_mode=0):
    blk_len, bt, norm, nnz = _fallback_worked_catalog()
    op = oracle.Op(oracle.AVG, 2, alpha=[1.0, 1.0], score_mode=score_mode)
    return oracle.plan(2, blk_len, bt, 2, 2, op, norm, np.ones_like(norm), nnz, None, budget, blk_tensor=bt)


def test_fallback_worked_example():
    """Hand-worked.  The pairs (0, t0) and (1, t1) fall back to one unit each:
    (0, t0): id 0*2+0 = 0, cost 24, score sqrt(3^2 + 4^2) = 5 (block 2's 99 is not used);
    (1, t1): id 3*2+1 = 7, cost 16, score sqrt(6^2) = 6.
    Block units: (1,b0) id 1, (1,b1) id 3, (1,b2) id 5, (0,b3) id 6 with score 1 and (0,b4) id
    8 with score 2, cost 8 each.  Order by score: 7, 0, 8, then 1, 3, 5, 6.
    B = 40: 7 (16), 0 (40), then nothing fits.  B = 30: 7 (16), 0 skipped, 8 (24), the rest
    skipped.  Per byte the scores are 6/16, 5/24, 2/8 and 1/8: order 7, 8, 0, 1, 3, 5, 6; B = 48
    takes 7, 8 and 0 (48).  B = 80 (everything) takes every unit."""
    p = _fallback_plan(40)
    assert p["order"].tolist() == [7, 0, 8, 1, 3, 5, 6] and p["n_cand"] == 7
    assert p["mask"].tolist() == [1, 1, 1, 2, 2] and p["chat"] == 40 and p["n_sel"] == 2
    assert p["set_hash"] == (oracle.splitmix64(7) + oracle.splitmix64(0)) % 2 ** 64
    p = _fallback_plan(30)
    assert p["mask"].tolist() == [0, 0, 0, 2, 3] and p["chat"] == 24 and p["n_sel"] == 2
    p = _fallback_plan(48, score_mode=1)
    assert p["order"].tolist() == [7, 8, 0, 1, 3, 5, 6]
    assert p["mask"].tolist() == [1, 1, 1, 2, 3] and p["chat"] == 48
    p = _fallback_plan(30, score_mode=1)
    assert p["mask"].tolist() == [0, 0, 0, 2, 3] and p["chat"] == 24
    p = _fallback_plan(80)
    assert p["mask"].tolist() == [3] * 5 and p["chat"] == 80 and p["n_sel"] == 7


def test_fallback_worked_example_with_unequal_coefficients():
    """Hand-worked, the catalog above under TA with alpha = (0.25, -2): scores are |alpha_i|
    times the norm.  (0, t0) id 0: 0.25 * 5 = 1.25; (1, t1) id 7: 2 * 6 = 12; (1, b0..b2)
    ids 1, 3, 5: 2 each; (0, b4) id 8: 0.5; (0, b3) id 6: 0.25.  Order 7, 1, 3, 5, 0, 8, 6.
    B = 40: 7 (16), 1, 3, 5 (40), then nothing fits: bit 1 on every block."""
    blk_len, bt, norm, nnz = _fallback_worked_catalog()
    op = oracle.Op(oracle.TA, 2, alpha=[0.25, -2.0])
    p = oracle.plan(2, blk_len, bt, 2, 2, op, norm, np.ones_like(norm), nnz, None, 40, blk_tensor=bt)
    assert p["order"].tolist() == [7, 1, 3, 5, 0, 8, 6]
    assert p["mask"].tolist() == [2] * 5 and p["chat"] == 40 and p["n_sel"] == 4


def test_fallback_needs_the_tensor_map():
    blk_len, bt, norm, nnz = _fallback_worked_catalog()
    op = oracle.Op(oracle.AVG, 2, alpha=[1.0, 1.0])
    with pytest.raises(Exception):
        oracle.plan(2, blk_len, bt, 2, 2, op, norm, np.ones_like(norm), nnz, None, 40)
    with pytest.raises(Exception):   # a tensor's blocks must be contiguous
        oracle.plan(2, blk_len, bt, 2, 2, op, norm, np.ones_like(norm), nnz, None, 40,
                    blk_tensor=np.array([0, 1, 0, 1, 1], np.uint32))


def test_fallback_without_missing_entries_is_the_block_plan(tiny_family):
    """the tensor map changes nothing while every entry has statistics"""
    fam, base, experts = tiny_family
    of = oracle_family(fam, base, experts)
    norm, maxabs, nnz = oracle.index(of)
    _, bl, bt = fam.block_table()
    for kind, kw in ((oracle.TA, dict(alpha=[0.3, -0.5, 0.7, 1.0][:fam.K])), (oracle.AVG, dict(alpha=[0.25] * fam.K))):
        for sm in (0, 1):
            op = oracle.Op(kind, fam.K, score_mode=sm, **kw)
            for f in (0.1, 0.5, 1.0):
                B = int(f * fam.K * fam.total_elems * 4)
                a = oracle.plan(fam.K, bl, bt, len(fam.tensors), 4, op, norm, maxabs, nnz, None, B)
                b = oracle.plan(fam.K, bl, bt, len(fam.tensors), 4, op, norm, maxabs, nnz, None, B, blk_tensor=bt)
                assert a["digest"] == b["digest"] and np.array_equal(a["mask"], b["mask"])
                assert np.array_equal(a["order"], b["order"])


def test_fallback_score_is_the_known_part_norm_of_the_deltas(tiny_family):
    """Against the deltas themselves: with one expert, a fallback tensor t competes with one
    block whose catalog norm is set 0.1 % above or below ||Delta_t|| over t's known blocks
    (fp64, from the data).  The budget fits either but not both, so the winner shows the
    order: the block wins when above, the tensor when below."""
    fam, base, experts = tiny_family
    of = oracle_family(fam, base[:], [experts[0]])
    norm, maxabs, nnz = oracle.index(of)
    bo, bl, bt = fam.block_table()
    counts = np.bincount(bt)
    t = int(np.argmax(counts))                      # the tensor with most blocks
    blocks = np.nonzero(bt == t)[0]
    assert len(blocks) >= 3
    other = int(np.nonzero(bt != t)[0][0])
    miss = int(blocks[1])
    nnz = nnz.copy()
    keep = np.zeros(nnz.shape[1], bool)
    keep[blocks] = True
    keep[other] = True
    nnz[0, ~keep] = 0                               # nothing else competes
    nnz[0, miss] = MISS
    d = experts[0].astype(np.float64) - base.astype(np.float64)
    known = [int(b) for b in blocks if int(b) != miss]
    exact = math.sqrt(sum(float((d[int(bo[b]):int(bo[b] + bl[b])] ** 2).sum()) for b in known))
    t_cost = int(bl[blocks].sum()) * 4
    B = max(t_cost, int(bl[other]) * 4)
    assert B < t_cost + int(bl[other]) * 4
    op = oracle.Op(oracle.TA, 1, alpha=[1.0])
    for factor, tensor_wins in ((1.001, False), (0.999, True)):
        nm = norm.copy()
        nm[0, other] = np.float32(exact * factor)
        p = oracle.plan(1, bl, bt, len(fam.tensors), 4, op, nm, maxabs, nnz, None, B, blk_tensor=bt)
        assert bool(p["mask"][blocks[0]]) == tensor_wins
        assert bool(p["mask"][other]) == (not tensor_wins)
        # all or nothing over the tensor
        assert len(set(int(p["mask"][b]) for b in blocks)) == 1


def test_fallback_properties_on_random_catalogs():
    """For random catalogs with missing entries: a fallback pair is read all or nothing;
    C_hat is the bytes the mask reads and never exceeds B (Prop. 1); the candidates are the
    fallback pairs plus the other units with nnz > 0; the full budget reads every candidate
    block; along the order, the greedy takes a unit iff it still fits."""
    rng = np.random.default_rng(31)
    for trial in range(40):
        K = int(rng.integers(1, 5))
        n_t = int(rng.integers(1, 6))
        per_t = rng.integers(1, 5, n_t)
        bt = np.repeat(np.arange(n_t), per_t).astype(np.uint32)
        nb = bt.size
        bl = rng.integers(1, 9, nb).astype(np.uint32)
        norm = rng.choice([0.5, 1.0, 2.0, 3.0], (K, nb)).astype(np.float32)
        nnz = (rng.random((K, nb)) > 0.25).astype(np.uint32) * 3
        nnz[rng.random((K, nb)) < 0.2] = MISS
        op = oracle.Op(oracle.TA, K, alpha=rng.choice([-1.0, 0.5, 2.0], K), score_mode=trial % 2)
        fb = np.zeros((K, n_t), bool)
        for i in range(K):
            for b in range(nb):
                fb[i, bt[b]] |= nnz[i, b] == MISS
        first = {int(t): int(np.nonzero(bt == t)[0][0]) for t in range(n_t)}
        cost = {}
        for b in range(nb):
            for i in range(K):
                if fb[i, bt[b]]:
                    if b == first[int(bt[b])]:
                        cost[b * K + i] = int(bl[bt == bt[b]].sum()) * 2
                elif nnz[i, b] > 0:
                    cost[b * K + i] = int(bl[b]) * 2
        total = sum(cost.values())
        for B in (0, total // 3, total // 2, total):
            p = oracle.plan(K, bl, np.zeros(nb, np.uint32), 1, 2, op, norm, np.ones_like(norm), nnz, None, B,
                            blk_tensor=bt)
            A = (p["mask"][None, :] >> np.arange(K)[:, None]) & 1
            for i in range(K):
                for t in range(n_t):
                    if fb[i, t]:
                        assert len(set(A[i, bt == t].tolist())) == 1
            assert p["chat"] == int((A * bl[None, :]).sum()) * 2 <= B
            assert p["n_cand"] == len(cost) and sorted(p["order"].tolist()) == sorted(cost)
            run = 0
            for u in p["order"].tolist():
                b, i = u // K, u % K
                if A[i, b]:
                    assert run + cost[u] <= B
                    run += cost[u]
                else:
                    assert run + cost[u] > B
            assert run == p["chat"]
            if B == total:
                want = fb[:, bt] | ((nnz > 0) & (nnz != MISS))
                assert np.array_equal(A.astype(bool), want)


def test_fallback_plan_at_full_budget_merges_like_the_full_read(tiny_family):
    """A = 1 over every block that can change the output recovers the full-read operator
    (Eq. 5), whatever entries lack statistics"""
    fam, base, experts = tiny_family
    of = oracle_family(fam, base, experts)
    norm, maxabs, nnz = oracle.index(of)
    _, bl, bt = fam.block_table()
    rng = np.random.default_rng(32)
    nnz = nnz.copy()
    nnz[rng.random(nnz.shape) < 0.15] = MISS
    for op in (oracle.Op(oracle.TA, fam.K, alpha=[0.4] * fam.K), oracle.Op(oracle.AVG_RENORM, fam.K, alpha=[1.0] * fam.K)):
        B = fam.K * fam.total_elems * 4
        p = oracle.plan(fam.K, bl, bt, len(fam.tensors), 4, op, norm, maxabs, nnz, None, B, blk_tensor=bt)
        got = oracle.merge(of, op, mask=p["mask"], nnz=nnz)
        want = oracle.merge(of, op)
        assert np.array_equal(got.view(np.uint32), want.view(np.uint32))


# ---- block content hash (catalog hashes; Alg. 2 validates them) -------------------------------------------

M64 = 2 ** 64


def _words_to_bytes(words):
    return np.asarray(words, np.uint64).tobytes()


def test_block_hash_detects_every_single_word_change():
    """odd keys are units mod 2^64: changing any one 64-bit word by any nonzero amount
    (including 2^63, which an even key would annihilate) changes the hash"""
    rng = np.random.default_rng(41)
    words = rng.integers(0, 2 ** 63, 64, dtype=np.uint64) * np.uint64(2) + np.uint64(1)
    h0 = oracle.block_hash(_words_to_bytes(words))
    for j in range(words.size):
        for d in (1, 2 ** 63, int(rng.integers(1, 2 ** 62))):
            w = words.copy()
            w[j] = np.uint64((int(w[j]) + d) % M64)
            assert oracle.block_hash(_words_to_bytes(w)) != h0, (j, d)


def test_block_hash_depends_on_position_and_word_order():
    rng = np.random.default_rng(42)
    words = rng.integers(0, 2 ** 63, 32, dtype=np.uint64)
    h0 = oracle.block_hash(_words_to_bytes(words))
    sw = words.copy()
    sw[[0, 1, 2, 3]] = sw[[2, 3, 0, 1]]           # swap vectors 0 and 1
    assert oracle.block_hash(_words_to_bytes(sw)) != h0
    hl = words.copy()
    hl[[4, 5]] = hl[[5, 4]]                       # swap the two words of vector 2
    assert oracle.block_hash(_words_to_bytes(hl)) != h0


def test_block_hash_sum_is_additive_over_disjoint_support():
    """H is a sum of per-word terms, so blocks with disjoint nonzero words add (mod 2^64),
    and an all-zero block has H = 0 (its hash is SplitMix64 of the length alone)"""
    rng = np.random.default_rng(43)
    for n_words in (2, 6, 64, 2 * 257):
        a = rng.integers(0, 2 ** 63, n_words, dtype=np.uint64)
        pick = rng.random(n_words) < 0.5
        x = np.where(pick, a, 0).astype(np.uint64)
        y = np.where(pick, 0, a).astype(np.uint64)
        hx, hy, ha = (oracle.block_hash_sum(_words_to_bytes(v)) for v in (x, y, a))
        assert (hx + hy) % M64 == ha
        assert oracle.block_hash_sum(bytes(8 * n_words)) == 0
        assert oracle.block_hash(bytes(8 * n_words)) == oracle.splitmix64(8 * n_words)


def test_block_hash_pads_to_vectors_and_mixes_the_length():
    """a ragged block is hashed as if zero-padded to 16 bytes (same H), but the length is
    mixed in, so the padded and unpadded blocks differ"""
    data = bytes(range(1, 23))                    # 22 bytes: one full vector and 6 bytes
    padded = data + bytes(10)
    assert oracle.block_hash_sum(data) == oracle.block_hash_sum(padded)
    assert oracle.block_hash(data) != oracle.block_hash(padded)


def test_index_hashes_are_content_addressed(tiny_family):
    """the catalog's hash of a block depends on its bytes only: an expert block equal to the
    base block has the base's hash, and every block matches hashing its bytes directly"""
    fam, base, experts = tiny_family
    e0 = experts[0].copy()
    bo, bl, _ = fam.block_table()
    s0 = slice(int(bo[1]), int(bo[1] + bl[1]))
    e0[s0] = base[s0]
    of = oracle_family(fam, base, [e0] + list(experts[1:]))
    bh, eh = oracle.index_hashes(of)
    assert eh[0, 1] == bh[1]
    for b in (0, 1, fam.n_blocks - 1):
        s = slice(int(bo[b]), int(bo[b] + bl[b]))
        assert bh[b] == oracle.block_hash(base[s].tobytes())
        assert eh[1, b] == oracle.block_hash(experts[1][s].tobytes())
    assert len(set(bh.tolist())) > fam.n_blocks // 2


def test_avg_single_expert_unit_weight_reproduces_the_expert():
    """K = 1, AVG with alpha = 1: out = round(M_0 + (M_1 - M_0)) is M_1 itself wherever the
    fp32 delta is exact (checked against fp64), bit for bit, masked-in; masked out it is M_0"""
    rng = np.random.default_rng(51)
    n = 5000
    base = to_bf16(rng.standard_normal(n) * 0.02)
    ex = to_bf16(bf16_to_f32(base) + (rng.standard_normal(n) * 1e-3).astype(np.float32))
    b64, e64 = bf16_to_f32(base).astype(np.float64), bf16_to_f32(ex).astype(np.float64)
    exact = (bf16_to_f32(ex) - bf16_to_f32(base)).astype(np.float64) == e64 - b64
    assert exact.mean() > 0.99
    op = oracle.Op(oracle.AVG, 1, alpha=[1.0])
    out = oracle.merge_block(oracle.BF16, 0, base, [ex], 1, op)
    assert np.array_equal(out[exact], ex[exact])
    out0 = oracle.merge_block(oracle.BF16, 0, base, [ex], 0, op)
    assert np.array_equal(out0.view(np.uint16) & 0x7FFF, base.view(np.uint16) & 0x7FFF)


# ---- TIES after masking (App. A.1) ----------------------------------------------------------------------

def test_ties_masked_thresholds_brute_force(tiny_family):
    """the threshold of the zero-completed masked deltas is the k-th largest key when every
    entry of an unselected block counts as a zero (sorted directly in numpy from the
    deltas' bf16 keys); the full mask gives the ordinary thresholds, the empty mask keys 0"""
    fam, base, experts = tiny_family
    of = oracle_family(fam, base, experts)
    bo, bl, bt = fam.block_table()
    rng = np.random.default_rng(61)
    for density in (0.05, 0.2, 0.6):
        full = oracle.ties_thresholds(of, density)
        assert np.array_equal(oracle.ties_masked_thresholds(of, density, np.full(fam.n_blocks, 0xF, np.uint32)), full)
        for trial in range(2):
            mask = rng.integers(0, 16, fam.n_blocks).astype(np.uint32)
            got = oracle.ties_masked_thresholds(of, density, mask)
            for i in range(fam.K):
                d = experts[i].astype(np.float32) - base.astype(np.float32)
                keys = bf16_bits_torch(np.abs(d)).astype(np.int64) & 0x7FFF
                for t in range(len(fam.tensors)):
                    parts = []
                    for b in np.nonzero(bt == t)[0]:
                        s_ = slice(int(bo[b]), int(bo[b] + bl[b]))
                        parts.append(keys[s_] if (mask[b] >> i) & 1 else np.zeros(int(bl[b]), np.int64))
                    allk = np.sort(np.concatenate(parts))[::-1]
                    k = int(math.floor(density * allk.size))
                    want = oracle.TAU_NONE if k == 0 else int(allk[k - 1])
                    assert got[i, t] == want, (density, i, t)
        zero = oracle.ties_masked_thresholds(of, density, np.zeros(fam.n_blocks, np.uint32))
        assert (zero == 0).all()


def test_ties_masked_full_mask_merges_like_ties(tiny_family):
    """with every block selected the masked operator is standard TIES (Eq. 5)"""
    fam, base, experts = tiny_family
    of = oracle_family(fam, base, experts)
    full_mask = np.full(fam.n_blocks, 0xF, np.uint32)
    tau = oracle.ties_thresholds(of, 0.2)
    tm = oracle.ties_masked_thresholds(of, 0.2, full_mask)
    a = oracle.merge(of, oracle.Op(oracle.TIES, fam.K, lam=1.0, density=0.2), tau=tau, mask=full_mask)
    b = oracle.merge(of, oracle.Op(oracle.TIES_MASKED, fam.K, lam=1.0, density=0.2), tau=tm, mask=full_mask)
    assert np.array_equal(a.view(np.uint32), b.view(np.uint32))


def test_ties_masked_thresholds_per_expert_scope(tiny_family):
    """trim scope 1 (one group per expert): the k-th largest masked key over the whole
    checkpoint, brute force"""
    fam, base, experts = tiny_family
    of = oracle_family(fam, base, experts, trim_scope=1)
    bo, bl, _ = fam.block_table()
    rng = np.random.default_rng(62)
    mask = rng.integers(0, 16, fam.n_blocks).astype(np.uint32)
    for density in (0.1, 0.5):
        got = oracle.ties_masked_thresholds(of, density, mask)
        assert got.shape == (fam.K, 1)
        for i in range(fam.K):
            d = experts[i].astype(np.float32) - base.astype(np.float32)
            keys = bf16_bits_torch(np.abs(d)).astype(np.int64) & 0x7FFF
            parts = [keys[int(bo[b]):int(bo[b] + bl[b])] if (mask[b] >> i) & 1 else np.zeros(int(bl[b]), np.int64)
                     for b in range(fam.n_blocks)]
            allk = np.sort(np.concatenate(parts))[::-1]
            k = int(math.floor(density * allk.size))
            assert got[i, 0] == (oracle.TAU_NONE if k == 0 else int(allk[k - 1])), (density, i)


def _dare_seed_keeping_first_dropping_second(p):
    for seed in range(100000):
        if oracle.dare_keep(seed, 0, 0, p) and not oracle.dare_keep(seed, 1, 0, p):
            return seed
    raise AssertionError("no seed found")


def test_dare_omits_a_dropped_entry_even_in_the_sign_of_zero():
    """R13: a dropped entry is left out of the sum, as an unselected one is.  Expert 1's kept
    product underflows to -0 (alpha 2^-20 times -2^-132), so the sum is -0; expert 2 is dropped
    with alpha > 0.  Omitting it keeps -0 and the output is M_0 + (-0) = -0 for M_0 = -0;
    adding its zero instead would give +0 + (-0) = +0 and the output +0."""
    p = 0.5
    seed = _dare_seed_keeping_first_dropping_second(p)
    base = np.array([0x8000], np.uint16)            # -0
    e0 = np.array([0x8001], np.uint16)              # -2^-133, the smallest bf16 subnormal
    e1 = np.array([0x3F80], np.uint16)              # 1.0 (dropped)
    op = oracle.Op(oracle.DARE, 2, alpha=[2.0 ** -20, 0.5], drop_p=p, seed=seed)
    out = oracle.merge_block(oracle.BF16, 0, base, [e0, e1], 0b11, op)
    assert out[0] == 0x8000
    # with expert 2 kept (p = 0) its contribution is an ordinary nonzero term
    op0 = oracle.Op(oracle.DARE, 2, alpha=[2.0 ** -20, 0.5], drop_p=0.0, seed=seed)
    assert oracle.merge_block(oracle.BF16, 0, base, [e0, e1], 0b11, op0)[0] == 0x3F00  # 0.5
