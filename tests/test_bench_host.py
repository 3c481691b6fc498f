"""Host logic of bench.py that needs no GPU: the affine read-time model fit, the seeded
pattern of catalog entries without statistics, the fidelity columns, the agreement of the
library's and the oracle's operator for every workload, and the clock record."""
import math
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def test_time_model_fit_recovers_an_affine_model():
    """merge times generated from T(f) = a + b f are fitted back exactly (r^2 = 1), and the
    model's slope and intercept follow from C_full, 2 N s and the bandwidth"""
    import bench

    c_full, ckpt = 8_000_000_000, 1_000_000_000
    a, b = 0.31, 1.07
    per = [{"planned_bytes": int(f * c_full), "merge_ms": a + b * f} for f in (1.0, 0.5, 0.25, 0.1)]
    fit = bench.time_model_fit([1.0, 0.5, 0.25, 0.1], per, ckpt, c_full, 6800.0, False)
    assert math.isclose(fit["slope_ms"], b, rel_tol=1e-9) and math.isclose(fit["intercept_ms"], a, rel_tol=1e-9)
    assert math.isclose(fit["r2"], 1.0, rel_tol=1e-12)
    assert math.isclose(fit["model_slope_ms"], c_full / 6800e9 * 1e3)
    assert math.isclose(fit["model_intercept_ms"], 2 * ckpt / 6800e9 * 1e3)
    assert math.isclose(fit["bw_from_slope_gbs"], c_full / (b / 1e3) / 1e9)
    # the touched-only merge has no fixed 2 N s term; one budget gives no line
    assert bench.time_model_fit([1.0, 0.5], per[:2], ckpt, c_full, 6800.0, True)["model_intercept_ms"] is None
    assert bench.time_model_fit([1.0], per[:1], ckpt, c_full, 6800.0, False) is None


def test_missing_entries_pattern_is_seeded_and_pair_dominated():
    """the same pattern on every call; the largest tensor of expert 0 is missing whole; every
    tensor with a missing pair is missing for all its blocks of that expert"""
    from paper_2605_29489_gb300 import synth

    fam = synth.qwen25_05b(layers=2)
    a = synth.missing_entries(fam, fam.K)
    b = synth.missing_entries(fam, fam.K)
    assert a.shape == (fam.K, fam.n_blocks) and np.array_equal(a, b)
    _, _, bt = fam.block_table()
    big = int(np.argmax(np.bincount(bt)))
    assert a[0, bt == big].all()
    c = synth.missing_entries(fam, fam.K, pair_frac=0.0, entry_frac=0.0)
    assert c.sum() == int((bt == big).sum())     # only the forced pair
    assert 0.0 < a.mean() < 0.5


def test_fidelity_columns_match_their_definitions():
    """Tab. 3's fidelity columns as bench.py reports them, against the definitions written
    out over the blocks: rel. l2 = ||M_A - M_full|| / ||M_full|| over the whole checkpoint;
    P95 = the 95th percentile (linear interpolation) over blocks of ||d_b|| / ||M_full[b]||.
    The family has a ragged last block in every tensor; perturbations sit in a few blocks."""
    import torch

    import bench

    class Fam:
        block_elems = 64
        tensors = [(0, 300), (304, 130), (448, 64)]

        def layout(self):
            offs = np.array([o for o, _ in self.tensors], np.int64)
            nums = np.array([n for _, n in self.tensors], np.int64)
            return offs, nums, 512

    fam = Fam()
    rng = np.random.default_rng(7)
    full = torch.from_numpy(rng.standard_normal(512).astype(np.float32))
    budgets = [1.0, 0.5, 0.25]
    outs = [full.clone()]
    for scale in (1e-3, 1e-2):
        o = full.clone()
        idx = torch.from_numpy(rng.choice(512, 40, replace=False))
        o[idx] += torch.from_numpy((rng.standard_normal(40) * scale).astype(np.float32))
        outs.append(o)
    per = [{} for _ in budgets]
    bench.fidelity_vs_full(fam, budgets, outs, False, per)
    F = full.double().numpy()
    for k, out in enumerate(outs):
        D = out.double().numpy() - F
        num = den = 0.0
        rel = []
        for o, n in fam.tensors:
            for s in range(0, n, fam.block_elems):
                e = min(n, s + fam.block_elems)
                d, f = D[o + s:o + e], F[o + s:o + e]
                num += float(d @ d)
                den += float(f @ f)
                rel.append(math.sqrt(float(d @ d) / float(f @ f)))
        assert math.isclose(per[k]["rel_l2_vs_full"], math.sqrt(num / den), rel_tol=1e-12)
        assert math.isclose(per[k]["p95_block_dev_vs_full"], float(np.percentile(np.float32(rel), 95)),
                            rel_tol=1e-6, abs_tol=1e-12)
    assert per[0]["rel_l2_vs_full"] == 0.0 and per[0]["p95_block_dev_vs_full"] == 0.0
    # no full-read budget in the sweep (or one shared output buffer): nothing is reported
    per = [{}]
    bench.fidelity_vs_full(fam, [0.5], outs[1:2], False, per)
    assert per == [{}]


def test_every_workload_gives_the_library_and_the_oracle_the_same_operator():
    """bench.py builds each workload's operator twice, for the library and for the oracle
    (the CPU baseline); both must describe the same merge: kind, coefficients, lambda,
    density, trim scope, drop probability, seed and score mode"""
    import bench

    for name, w in bench.workloads().items():
        fam = w["make"]()
        g, o = bench.make_ops(w, fam.K)
        c = g.c
        assert c.kind == o.kind, name
        if o.alpha is None:
            assert g.alpha is None, name
        else:
            assert np.array_equal(g.alpha, o.alpha) and len(o.alpha) == fam.K, name
        assert np.float32(c.lambda_) == np.float32(o.lam) and np.float32(c.density) == np.float32(o.density), name
        assert (c.trim_scope, c.drop_p, c.seed, c.score_mode) == (o.trim_scope, o.drop_p, o.seed, o.score_mode), name


def test_clock_sampler_summary():
    """the clock record the bench line carries: median SM clock under load, the maximum, and
    every throttle reason seen active in any sample (malformed lines are skipped)"""
    import bench

    class Done:
        def terminate(self):
            pass

        def wait(self, timeout=None):
            return 0

    cs = bench.ClockSampler(0)
    cs.proc = Done()
    cs.lines = [
        "0, 2070, 2070, 900.1, 0x0, Not Active, Not Active, Not Active, Not Active",
        "0, 2055, 2070, 1390.0, 0x4, Not Active, Not Active, Not Active, Active",
        "garbage line",
        "0, 1980, 2070, 1400.0, 0x4, Not Active, Not Active, Not Active, Active",
        "0, [N/A], 2070, 1400.0, 0x0, Not Active, Not Active, Not Active, Not Active",
    ]
    s = cs.stop()
    assert s == {"sm_mhz": 2055.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"], "samples": 3}
    cs = bench.ClockSampler(0)
    cs.proc = Done()
    cs.lines = ["0, 1500, 2070, 800.0, 0x40, Active, Not Active, Active, Not Active"]
    assert cs.stop()["reasons"] == ["hw_slowdown", "sw_thermal_slowdown"]
    cs = bench.ClockSampler(0)             # nvidia-smi could not be started: no record
    assert cs.stop() is None


def test_interval_union_and_overlap_of_the_host_timeline():
    """the timeline's busy time is the length of a union of intervals (overlaps counted
    once, gaps not at all), and a kernel's time under gathers is its intersection with it"""
    import bench

    iv = [(0.0, 2.0), (1.0, 3.0), (5.0, 6.0), (5.5, 5.7), (8.0, 8.0)]
    assert bench._union_ms(iv) == 4.0
    assert bench._union_ms([]) == 0.0
    assert bench._overlap_ms(2.5, 5.5, iv) == 1.0   # [2.5, 3] and [5, 5.5]
    assert bench._overlap_ms(3.0, 5.0, iv) == 0.0
    assert bench._overlap_ms(-1.0, 10.0, iv) == bench._union_ms(iv)


def test_host_memory_reading():
    """MemAvailable in bytes: positive, and no more than MemTotal"""
    import bench

    avail = bench.host_mem_available()
    total = None
    with open("/proc/meminfo") as f:
        for line in f:
            if line.startswith("MemTotal:"):
                total = float(line.split()[1]) * 1024.0
    assert 0 < avail <= total
