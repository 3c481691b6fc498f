#!/usr/bin/env python3
"""Benchmark of the budgeted, mask-aware merge on GB300.

One step = one pass of the whole hot path over the workload: the catalog pass
(mp_index_blocks), then for every budget of the sweep the access plan (mp_plan)
and the budgeted merge (mp_merge).  Inputs are seeded synthetic checkpoint
families with the published tensor shapes, generated on the device before the
timed region; every checkpoint is larger than L2, so no flush is needed.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--impl native|reference]

Prints one JSON line.  `value` is merged parameters per second over the sweep
(budgets x params / step time), device-timed with CUDA events; `e2e` is the same
metric with the inputs copied from pinned host memory and the merged outputs
copied back inside the timed region.  `--impl reference` times the CPU oracle on
the host cores on a bounded sample of the same workload.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import re
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "accessed-expert GB/s vs HBM peak; merged params/s per budget (1 GB300)"
UNIT = "params/s"
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0


def workloads():
    from paper_2605_29489_gb300 import synth

    return {
        "qwen2.5-0.5b-ta": dict(make=lambda: synth.qwen25_05b(), op="ta", lam=0.3, budgets=[1.0, 0.5, 0.25, 0.1],
                                desc="Qwen2.5-0.5B-shaped bf16 family, K=8, task arithmetic lambda=0.3, 64Ki-element blocks"),
        "qwen2.5-0.5b-ta-2l": dict(make=lambda: synth.qwen25_05b(layers=2), op="ta", lam=0.3,
                                   budgets=[1.0, 0.5, 0.25, 0.1],
                                   desc="Qwen2.5-0.5B shapes cut to 2 layers (profiling case), K=8, TA lambda=0.3"),
        "qwen2.5-0.5b-ties-2l": dict(make=lambda: synth.qwen25_05b(layers=2, K=4), op="ties", density=0.2,
                                     budgets=[1.0, 0.5, 0.25, 0.1],
                                     desc="Qwen2.5-0.5B shapes cut to 2 layers (profiling case), K=4, TIES density 0.2"),
        "llama-3-8b-ties": dict(make=lambda: synth.llama3_8b(), op="ties", density=0.2, budgets=[1.0, 0.5, 0.25, 0.1],
                                desc="Llama-3-8B-shaped bf16 family, K=4, TIES density 0.2, 64Ki-element blocks"),
        "llama-3-8b-ties-1l": dict(make=lambda: synth.llama3_8b(layers=1), op="ties", density=0.2,
                                   budgets=[1.0, 0.5, 0.25, 0.1],
                                   desc="one Llama-3-8B transformer layer (no embedding or lm_head; profiling "
                                        "case), K=4, TIES density 0.2"),
        "llama-3-8b-ties-masked": dict(make=lambda: synth.llama3_8b(), op="ties_masked", density=0.2,
                                       budgets=[1.0, 0.5, 0.25, 0.1],
                                       desc="Llama-3-8B-shaped bf16 family, K=4, TIES applied after masking (threshold "
                                            "of the zero-completed masked deltas, App. A.1) density 0.2"),
        "qwen2.5-1.5b-dare": dict(make=lambda: synth.qwen25_15b(), op="dare", drop_p=0.9, budgets=[0.25],
                                  desc="Qwen2.5-1.5B-shaped bf16 family, K=16, DARE p=0.9 then AVG, per-expert active sets"),
        "qwen2.5-0.5b-avg-renorm": dict(make=lambda: synth.qwen25_05b(), op="avg_renorm", budgets=[1.0, 0.5, 0.25, 0.1],
                                        desc="Qwen2.5-0.5B-shaped bf16 family, K=8, AVG renormalised over the selected "
                                             "experts (App. A.1)"),
        "qwen2.5-1.5b-dare-ties": dict(make=lambda: synth.qwen25_15b(), op="dare_ties", drop_p=0.9, budgets=[0.25],
                                       desc="Qwen2.5-1.5B-shaped bf16 family, K=16, DARE-TIES p=0.9 lambda=1, "
                                            "per-expert active sets"),
        "qwen2.5-1.5b-dare-2l": dict(make=lambda: synth.qwen25_15b(layers=2), op="dare", drop_p=0.9, budgets=[0.25],
                                     desc="Qwen2.5-1.5B shapes cut to 2 layers (profiling case), K=16, DARE p=0.9"),
        "qwen2.5-1.5b-dare-ties-2l": dict(make=lambda: synth.qwen25_15b(layers=2), op="dare_ties", drop_p=0.9,
                                          budgets=[0.25],
                                          desc="Qwen2.5-1.5B shapes cut to 2 layers (profiling case), K=16, DARE-TIES "
                                               "p=0.9"),
        "llama-3-8b-hostpool-avg": dict(make=lambda: synth.llama3_8b(K=8), op="avg", budgets=[1.0, 0.25, 0.1],
                                        host_pool=True,
                                        desc="Llama-3-8B-shaped bf16 base in HBM, K=8 experts (128 GB) in pinned host "
                                             "memory, AVG, planned blocks gathered over NVLink-C2C"),
        "llama-3-8b-hostpool-ties": dict(make=lambda: synth.llama3_8b(K=8), op="ties", density=0.2,
                                         budgets=[1.0, 0.25, 0.1], host_pool=True,
                                         desc="Llama-3-8B-shaped bf16 base in HBM, K=8 experts (128 GB) in pinned host "
                                              "memory, TIES density 0.2"),
        "qwen2.5-0.5b-ta-touched": dict(make=lambda: synth.qwen25_05b(), op="ta", lam=0.3,
                                        budgets=[1.0, 0.5, 0.25, 0.1], touched=True,
                                        desc="as qwen2.5-0.5b-ta, merged with mp_merge_touched: only touched blocks "
                                             "are read and written (Alg. 2 WriteBlockOrReference)"),
        "llama-3-8b-ta-fallback": dict(make=lambda: synth.llama3_8b(), op="ta", lam=0.3,
                                       budgets=[1.0, 0.5, 0.25, 0.1], fallback=True,
                                       desc="Llama-3-8B-shaped bf16 family, K=4, TA lambda=0.3, planned from an "
                                            "imported catalog without statistics for 10 % of the (expert, tensor) "
                                            "pairs (the embedding of expert 0 among them) and 0.1 % of the other "
                                            "entries: tensor-level fallback plan (Sec. 3 Planner)"),
        "tiny-avg": dict(make=lambda: synth.tiny(), op="avg", budgets=[1.0, 0.5, 0.25],
                         desc="8 fp32 512x512 tensors, K=4, AVG, 4Ki-element blocks"),
    }


DEFAULT_WORKLOAD = "llama-3-8b-ties"


def make_ops(w, K):
    import oracle
    import paper_2605_29489_gb300 as mp

    if w["op"] == "ta":
        a = [w["lam"]] * K
        return mp.make_op(mp.MP_OP_TA, alpha=a), oracle.Op(oracle.TA, K, alpha=a)
    if w["op"] == "avg":
        a = [1.0 / K] * K
        return mp.make_op(mp.MP_OP_AVG, alpha=a), oracle.Op(oracle.AVG, K, alpha=a)
    if w["op"] == "ties":
        return (mp.make_op(mp.MP_OP_TIES, lam=1.0, density=w["density"]),
                oracle.Op(oracle.TIES, K, lam=1.0, density=w["density"]))
    if w["op"] == "ties_masked":
        return (mp.make_op(mp.MP_OP_TIES_MASKED, lam=1.0, density=w["density"]),
                oracle.Op(oracle.TIES_MASKED, K, lam=1.0, density=w["density"]))
    if w["op"] == "dare":
        a = [1.0 / K] * K
        return (mp.make_op(mp.MP_OP_DARE, alpha=a, drop_p=w["drop_p"], seed=20260),
                oracle.Op(oracle.DARE, K, alpha=a, drop_p=w["drop_p"], seed=20260))
    if w["op"] == "avg_renorm":
        a = [1.0 / K] * K
        return mp.make_op(mp.MP_OP_AVG_RENORM, alpha=a), oracle.Op(oracle.AVG_RENORM, K, alpha=a)
    if w["op"] == "dare_ties":
        return (mp.make_op(mp.MP_OP_DARE_TIES, lam=1.0, drop_p=w["drop_p"], seed=20260),
                oracle.Op(oracle.DARE_TIES, K, lam=1.0, drop_p=w["drop_p"], seed=20260))
    raise ValueError(w["op"])


def fallback_missing(fam, K):
    """the fallback workloads' catalog entries without statistics (seeded; bool [K, n_blocks])"""
    from paper_2605_29489_gb300 import synth

    return synth.missing_entries(fam, K)


# ---- clocks ---------------------------------------------------------------------------------------

class ClockSampler:
    """nvidia-smi clock / throttle-reason samples taken during the timed region"""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.lines: list[str] = []
        self.proc = None
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()
        time.sleep(0.25)

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.15)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        if self.thread:
            self.thread.join(timeout=2)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# ---- measured peaks / profiles ------------------------------------------------------------------

def hbm_peak():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def merge_source_hash() -> str:
    h = hashlib.sha256()
    for name in ("merge.cu", "philox.cuh", "small_div.cuh", "tma.cuh"):
        with open(os.path.join(ROOT, "paper_2605_29489_gb300", "csrc", name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def profiled_traffic(workload: str, alg_bytes_per_launch: float):
    """DRAM bytes per merge launch from the committed ncu summary, if it was taken on the
    current merge kernel source (else None): either captured on this workload itself
    (traffic_per_launch), or on a smaller case of the same kernel whose DRAM bytes per
    algorithmic byte (traffic_ratio) scale to a full launch (traffic grows in proportion to
    the bytes a launch moves)"""
    path = os.path.join(ROOT, "profiles", "merge_kernel_traffic.md")
    if not os.path.exists(path):
        return None
    txt = open(path).read()
    src = re.search(r"source_hash:\s*([0-9a-f]+)", txt)
    if not src or src.group(1) != merge_source_hash():
        return None
    m = re.search(rf"traffic_per_launch\[{re.escape(workload)}\]:\s*([0-9.eE+]+)", txt)
    if m:
        return float(m.group(1))
    m = re.search(rf"traffic_ratio\[{re.escape(workload)}\]:\s*([0-9.eE+]+)", txt)
    return float(m.group(1)) * alg_bytes_per_launch if m else None


# ---- CPU oracle sample ----------------------------------------------------------------------------

def oracle_sample(w, fam, target_s: float):
    """A bounded sample of the workload for the CPU oracle: blocks evenly spaced over the
    family, as many as about target_s seconds of oracle work (index, then plan and merge at
    every budget) take, regenerated on the host once.  Returns (run, description); run()
    times one full pass of the oracle over the sample and returns (merged params/s, seconds).
    The oracle keeps nothing between passes, so every pass does the whole work again."""
    import numpy as np
    import oracle

    _, oop = make_ops(w, fam.K)
    bo, bl, bt = fam.block_table()
    budgets = w["budgets"]
    miss_all = fallback_missing(fam, fam.K) if w.get("fallback") else None
    es = fam.elem_size

    def prepare(blocks):
        data = [fam.block_host(int(b)) for b in blocks]
        lens = np.array([bl[b] for b in blocks], np.uint32)
        offs = np.zeros(len(blocks), np.uint64)
        o = 0
        for k, b in enumerate(blocks):
            offs[k] = o
            o += int(bl[b])
        base = np.concatenate([d[0] for d in data])
        experts = [np.concatenate([d[1][i] for d in data]) for i in range(fam.K)]
        groups = np.zeros(len(blocks), np.uint32)
        of = oracle.Family(fam.dtype, offs, lens, groups, 1, base, experts)
        catalog = None
        if miss_all is not None:
            # the catalog is imported, not computed: built before any clock starts
            norm, maxabs, nnz = oracle.index(of)
            nnz = nnz.copy()
            nnz[miss_all[:, blocks]] = oracle.NNZ_MISSING
            tmap = np.unique(bt[blocks], return_inverse=True)[1].astype(np.uint32)
            catalog = (norm, maxabs, nnz, tmap)
        return of, lens, groups, catalog

    def timed(sample):
        of, lens, groups, catalog = sample
        full = fam.K * int(lens.sum()) * es
        t0 = time.perf_counter()
        if catalog is None:
            norm, maxabs, nnz = oracle.index(of)
            tmap = None
        else:
            norm, maxabs, nnz, tmap = catalog
        tau = oracle.ties_thresholds(of, oop.density) if oop.kind == oracle.TIES else None
        for f in budgets:
            pl = oracle.plan(fam.K, lens, groups, 1, es, oop, norm, maxabs, nnz, tau, math.floor(f * full),
                             blk_tensor=tmap)
            m_tau = oracle.ties_masked_thresholds(of, oop.density, pl["mask"]) if oop.kind == oracle.TIES_MASKED else tau
            oracle.merge(of, oop, tau=m_tau, mask=pl["mask"], nnz=nnz if tmap is not None else None)
        return time.perf_counter() - t0

    nb = fam.n_blocks
    # per-block cost from an evenly spaced probe (active and inactive blocks differ in cost)
    probe = sorted(set(int(x) for x in np.linspace(0, nb - 1, min(nb, 8))))
    dt1 = timed(prepare(probe))
    n = max(1, min(nb, int(target_s / max(dt1 / len(probe), 1e-6))))
    blocks = sorted(set(int(x) for x in np.linspace(0, nb - 1, n)))
    sample = prepare(blocks)
    params = int(sample[1].sum())
    first = "catalog imported (computed before timing)" if miss_all is not None else "oracle index"
    desc = (f"{len(blocks)} of {nb} blocks ({params} params) evenly spaced over the family, regenerated on the "
            f"host once; {first} + plan and merge at budgets {budgets} (budget relative to the sample)")

    def run():
        dt = timed(sample)
        return len(budgets) * params / dt, dt

    return run, desc


def oracle_sample_run(w, fam, target_s: float):
    """One timed pass of the oracle over a bounded sample (oracle_sample):
    (merged params/s, seconds, sample description)"""
    run, desc = oracle_sample(w, fam, target_s)
    v, dt = run()
    return v, dt, desc


def cpu_info():
    model = ""
    try:
        out = subprocess.run(["lscpu"], stdout=subprocess.PIPE, text=True).stdout
        m = re.search(r"Model name:\s*(.+)", out)
        model = m.group(1).strip() if m else ""
    except Exception:
        pass
    return model, os.cpu_count()


# ---- native arm -----------------------------------------------------------------------------------

def native(args, rank, world, local_rank):
    import numpy as np
    import torch
    import paper_2605_29489_gb300 as mp

    torch.cuda.set_device(local_rank)
    W = workloads()[args.workload]
    fam = W["make"]()
    gop, _ = make_ops(W, fam.K)
    budgets = W["budgets"]
    base, experts = fam.device_arrays()
    host_pool = bool(W.get("host_pool"))
    link = None
    if host_pool:
        # the experts live in pinned host memory; only the base (and the output) stay in HBM
        experts_h = []
        for e in experts:
            h = torch.empty(e.shape, dtype=e.dtype, pin_memory=True)
            h.copy_(e)
            experts_h.append(h)
        del e
        experts = experts_h
        torch.cuda.empty_cache()
        link = measure_h2d(experts[0])
    offs, nums, total = fam.layout()
    tensors = list(zip(offs.tolist(), nums.tolist()))
    mf = mp.family(tensors, base, experts, fam.block_elems, fam.dtype, 1 if host_pool else 0)
    es = fam.elem_size
    N = fam.n_params
    free_b, _ = torch.cuda.mem_get_info()
    shared_out = free_b < (len(budgets) + 2) * total * es
    outs = [torch.empty_like(base)] if shared_out else [torch.empty_like(base) for _ in budgets]
    Bs = [mp.mp_budget_from_fraction(mf, f) for f in budgets]
    stream = torch.cuda.current_stream()
    touched_mode = bool(W.get("touched"))
    merge_fn = mp.mp_merge_touched if touched_mode else mp.mp_merge
    catalog = None
    if W.get("fallback"):
        # a catalog saved earlier, with entries lacking statistics; each step imports it
        idx0 = mp.mp_index_blocks(mf, gop)
        c_norm, c_max, c_nnz, c_tau = mp.mp_index_stats(idx0)
        idx0.free()
        c_nnz[fallback_missing(fam, fam.K)] = mp.MP_NNZ_MISSING
        catalog = (c_norm, c_max, c_nnz, c_tau if gop.kind == mp.MP_OP_TIES else None)

    def make_index(fam_c):
        if catalog is not None:
            return mp.mp_index_import(fam_c, gop, *catalog, stream=stream)
        return mp.mp_index_blocks(fam_c, gop, stream)

    def step(fam_c, ev=None, st=None):
        st = stream if st is None else st
        hs = []
        if ev is not None:
            ev["i0"].record(st)
        idx = make_index(fam_c) if st is stream else mp.mp_index_blocks(fam_c, gop, st)
        hs.append(idx)
        if ev is not None:
            ev["i1"].record(st)
        for k, B in enumerate(Bs):
            if ev is not None:
                ev["p0"][k].record(st)
            plan = mp.mp_plan(idx, gop, B, st)
            if ev is not None:
                ev["p1"][k].record(st)
            man = merge_fn(fam_c, idx, plan, outs[0 if shared_out else k], st)
            if ev is not None:
                ev["m1"][k].record(st)
            hs += [plan, man]
        return hs

    def new_events():
        E = lambda: torch.cuda.Event(enable_timing=True)  # noqa: E731
        return {"i0": E(), "i1": E(), "p0": [E() for _ in Bs], "p1": [E() for _ in Bs], "m1": [E() for _ in Bs]}

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()

    for _ in range(args.warmup):
        hs = step(mf)
        torch.cuda.synchronize()
        for h in hs:
            h.free()

    # ---- timed region (device) ----
    evs = [new_events() for _ in range(args.steps)]
    clocks = ClockSampler(local_rank)
    barrier()
    torch.cuda.synchronize()
    clocks.start()
    launches0 = mp.mp_kernel_launch_count()
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t_start.record(stream)
    handles = []
    for s in range(args.steps):
        handles.append(step(mf, evs[s]))
    t_end.record(stream)
    torch.cuda.synchronize()
    barrier()
    launches = mp.mp_kernel_launch_count() - launches0
    clk = clocks.stop()
    elapsed_ms = t_start.elapsed_time(t_end)

    idx_ms = statistics.mean(e["i0"].elapsed_time(e["i1"]) for e in evs)
    plan_ms = [statistics.mean(e["p0"][k].elapsed_time(e["p1"][k]) for e in evs) for k in range(len(Bs))]
    merge_ms = [statistics.mean(e["p1"][k].elapsed_time(e["m1"][k]) for e in evs) for k in range(len(Bs))]
    last = handles[-1]
    per_budget = []
    blk_len = fam.block_table()[1]
    for k, f in enumerate(budgets):
        pi = mp.mp_plan_info(last[1 + 2 * k], last[0] if touched_mode else None, with_arrays=touched_mode)
        mi = mp.mp_manifest_info(last[2 + 2 * k], fam.K)
        per_budget.append(dict(f=f, budget_bytes=Bs[k], planned_bytes=pi["chat"], realized_bytes=mi["realized_total"],
                               n_selected=pi["n_sel"], n_candidates=pi["n_cand"], touched_blocks=mi["touched"],
                               touched_ratio=pi["chat"] / (fam.K * N * es), plan_ms=plan_ms[k], merge_ms=merge_ms[k]))
        if touched_mode:
            per_budget[-1]["touched_elements"] = int(np.asarray(blk_len)[np.asarray(pi["mask"]) != 0].sum())
        if gop.kind == mp.MP_OP_TIES_MASKED:   # the masked threshold's second read of selected blocks
            per_budget[-1]["threshold_read_bytes"] = mp.mp_manifest_threshold_reads(last[2 + 2 * k])
    timeline = host_timeline(mp, step, mf, budgets, args.trace_out) if host_pool else None
    hashes = None
    if not host_pool and not args.no_hash:
        hashes = time_hashes(mp, fam, mf, last, outs, shared_out, per_budget, stream)
    for hs in handles:
        for h in hs:
            h.free()
    graph = None
    # device-resident families whose calls enqueue only kernels (TIES after masking and
    # imported catalogs copy host arrays in, which a capture cannot hold)
    if not host_pool and catalog is None and gop.kind != mp.MP_OP_TIES_MASKED:
        graph = graph_replay(mp, step, mf)

    if not touched_mode:   # touched-only outputs hold only the touched blocks
        fidelity_vs_full(fam, budgets, outs, shared_out, per_budget)

    peak, peak_kind = hbm_peak()
    # base read + output write of every materialised element, plus the planned expert reads
    alg_bytes = [2 * (pb["touched_elements"] if touched_mode else N) * es + pb["planned_bytes"] for pb in per_budget]
    for pb, ab in zip(per_budget, alg_bytes):
        s = pb["merge_ms"] / 1e3
        pb.update(merged_params_per_s=N / s, expert_gbs=pb["planned_bytes"] / s / 1e9, hbm_bytes=ab,
                  hbm_gbs=ab / s / 1e9, hbm_frac_measured=ab / s / 1e9 / peak,
                  hbm_frac_nominal=ab / s / 1e9 / NOMINAL_HBM_GBS)
    merge_total_s = sum(merge_ms) / 1e3
    achieved = sum(alg_bytes) / merge_total_s / 1e9
    t_model = time_model_fit(budgets, per_budget, N * es, fam.K * N * es, peak, touched_mode) if not host_pool else None

    # ---- e2e: pinned host inputs in, merged outputs back, inside the timed region ----
    e2e = None
    # the end-to-end leg pins the inputs and the outputs in host memory on every rank: it runs
    # only where each rank's share of the host's available memory holds them (with one output
    # buffer shared by the budgets if four do not fit); the decision is the same on every rank
    out_bufs = len(budgets)
    if not args.no_e2e and not host_pool:
        share = host_mem_available() / max(1, int(os.environ.get("LOCAL_WORLD_SIZE", world)))
        in_b, out_b = (fam.K + 1) * total * es, total * es
        if in_b + out_bufs * out_b > 0.85 * share:
            out_bufs = 1
        fits = in_b + out_bufs * out_b <= 0.85 * share
        # every rank must agree: the slowest rank's (largest) need decides
        need = _max_over_ranks(0.0 if fits else 1.0, world)
        if need > 0.0:
            e2e = {"skipped": f"host memory: the inputs and outputs need {(in_b + out_b) / 1e9:.0f} GB pinned per "
                              f"rank, {share / 1e9:.0f} GB is available per rank"}
            out_bufs = 0
    if not args.no_e2e and not host_pool and out_bufs > 0:
        def pinned_copy(t):
            h = torch.empty(t.shape, dtype=t.dtype, pin_memory=True)
            h.copy_(t)
            return h

        base_h = pinned_copy(base)
        experts_h = [pinned_copy(e) for e in experts]
        outs_h = [torch.empty(outs[0].shape, dtype=outs[0].dtype, pin_memory=True) for _ in range(out_bufs)]
        outs_h = [outs_h[min(k, out_bufs - 1)] for k in range(len(budgets))]  # one buffer: reused in order
        # the device-resident inputs of the timed leg are not needed any more: the end-to-end
        # leg brings its own copies in from the pinned host buffers
        shape, dt = base.shape, base.dtype
        del mf, base, experts
        torch.cuda.synchronize()
        torch.cuda.empty_cache()
        set_bytes = (fam.K + 1) * total * es
        free_b, _ = torch.cuda.mem_get_info()
        # two device copies of the inputs when they fit: step s + 1's inputs come in on their
        # own stream while step s computes and its outputs go back (the link is full duplex)
        n_sets = 2 if free_b > 2 * set_bytes + (4 << 30) else 1
        sets = []
        for _ in range(n_sets):
            bd = torch.empty(shape, dtype=dt, device="cuda")
            ed = [torch.empty(shape, dtype=dt, device="cuda") for _ in range(fam.K)]
            sets.append((bd, ed, mp.family(tensors, bd, ed, fam.block_elems, fam.dtype, 0)))
        e2e_steps = max(3, min(args.steps, 10))
        E = lambda: torch.cuda.Event()  # noqa: E731
        in_ready = [E() for _ in range(n_sets)]  # the set's inputs have arrived
        in_free = [E() for _ in range(n_sets)]   # the last merge reading the set is done
        h2d_stream = torch.cuda.Stream() if n_sets > 1 else stream

        # each budget's output goes back on a copy stream while the next budget is planned and
        # merged (separate output buffers); with a shared output buffer the copies stay in order.
        # A budget's merge waits only for the previous step's copy of its own output buffer.
        copy_stream = torch.cuda.Stream() if not shared_out else stream
        out_copied = [E() for _ in Bs]  # the previous step's copy of output k has read it
        for ev in out_copied:
            ev.record(copy_stream)

        def issue_inputs(j):
            h2d_stream.wait_event(in_free[j])
            with torch.cuda.stream(h2d_stream):
                sets[j][0].copy_(base_h, non_blocking=True)
                for d, h in zip(sets[j][1], experts_h):
                    d.copy_(h, non_blocking=True)
            in_ready[j].record(h2d_stream)

        def compute(j):
            stream.wait_event(in_ready[j])
            mf_d = sets[j][2]
            hs = []
            idx = make_index(mf_d)
            hs.append(idx)
            for k, B in enumerate(Bs):
                plan = mp.mp_plan(idx, gop, B, stream)
                out = outs[0 if shared_out else k]
                stream.wait_event(out_copied[0 if shared_out else k])
                man = mp.mp_merge(mf_d, idx, plan, out, stream)
                copy_stream.wait_stream(stream)
                with torch.cuda.stream(copy_stream):
                    outs_h[k].copy_(out, non_blocking=True)
                out_copied[0 if shared_out else k].record(copy_stream)
                hs += [plan, man]
            in_free[j].record(stream)
            return hs

        def run(n_steps, start_event=None):
            if start_event is not None:
                h2d_stream.wait_event(start_event)
            issue_inputs(0)
            hl = []
            for st in range(n_steps):
                if n_sets > 1 and st + 1 < n_steps:
                    issue_inputs((st + 1) % n_sets)
                hl.append(compute(st % n_sets))
                if n_sets == 1 and st + 1 < n_steps:
                    issue_inputs(0)
            stream.wait_stream(copy_stream)  # the last copies end inside the timed region
            return hl

        # the first passes over freshly pinned host buffers run well below the link rate
        # (translations are set up on first use): warm up like the device-timed leg
        for hs in run(args.warmup):
            torch.cuda.synchronize()
            for h in hs:
                h.free()
        barrier()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        hl = run(e2e_steps, a)
        b.record(stream)
        torch.cuda.synchronize()
        barrier()
        e2e_ms = a.elapsed_time(b) / e2e_steps
        for hs in hl:
            for h in hs:
                h.free()
        e2e_ms = _max_over_ranks(e2e_ms, world)
        e2e = {"value": world * len(budgets) * N / (e2e_ms / 1e3), "unit": UNIT,
               "h2d_bytes_per_step": (fam.K + 1) * N * es, "d2h_bytes_per_step": len(budgets) * N * es,
               "ms_per_step": e2e_ms, "input_sets": n_sets, "host_output_buffers": out_bufs}
        del base_h, experts_h, outs_h, sets

    elapsed_ms = _max_over_ranks(elapsed_ms, world)
    ms_per_step = elapsed_ms / args.steps
    value = replica_value(len(budgets) * N, world, ms_per_step)

    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16" if fam.dtype == 0 else "f32", "data": "synthetic",
        "config": {"workload": args.workload, "description": W["desc"], "params": N, "K": fam.K,
                   "blocks": fam.n_blocks, "block_elems": fam.block_elems, "budgets": budgets,
                   "parallelism": f"replicas x{world}", "l2": "inputs larger than L2 (no flush)",
                   "step": ("catalog import" if catalog is not None else "index") + " + (plan + merge) per budget"},
        "accessed_expert_gbs": sum(pb["planned_bytes"] for pb in per_budget) / merge_total_s / 1e9,
        "index_ms": idx_ms, "per_budget": per_budget, "time_model": t_model, "block_hashes": hashes,
        "roofline": {"bound": "hbm", "kernel": merge_kernel_name(W["op"], fam.dtype, fam.K), "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "peak_kind": peak_kind,
                     "frac_of_nominal_8tbs": achieved / NOMINAL_HBM_GBS,
                     "traffic": profiled_traffic(args.workload, sum(alg_bytes) / len(alg_bytes)),
                     "algorithmic_bytes": ("per materialised (touched) parameter" if touched_mode else
                                           "per merged parameter") + " 2*s + s*(selected experts); summed over the "
                                          "budget sweep's launches / their summed CUDA-event time"},
        "gpu_launches": launches,
        "host_timeline": timeline,
        "graph": graph,
        "host_link": None if link is None else dict(
            h2d_gbs_measured=link, gathered_bytes=[pb["planned_bytes"] for pb in per_budget],
            gathered_gbs=[pb["planned_bytes"] / (pb["merge_ms"] / 1e3) / 1e9 for pb in per_budget],
            frac_of_link=[pb["planned_bytes"] / (pb["merge_ms"] / 1e3) / 1e9 / link for pb in per_budget],
            index_reads_gbs=fam.K * N * es / (idx_ms / 1e3) / 1e9),
        "clocks": clk,
        "e2e": e2e,
    }
    if catalog is not None:
        miss = catalog[2] == mp.MP_NNZ_MISSING
        bt = np.asarray(fam.block_table()[2])
        pairs = np.zeros((fam.K, int(bt.max()) + 1), bool)
        for i in range(fam.K):
            pairs[i, np.unique(bt[miss[i]])] = True
        line["config"]["catalog"] = {"entries_missing": int(miss.sum()), "entries": int(miss.size),
                                     "fallback_pairs": int(pairs.sum()), "pairs": int(pairs.size)}
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        v, dt, desc = oracle_sample_run(W, fam, args.cpu_seconds)
        model, ncpu = cpu_info()
        line["cpu_baseline"] = {"value": v, "unit": UNIT, "cores": 1, "kind": "oracle", "sample": desc,
                                "seconds": dt, "host_cpu": model, "host_cores_available": ncpu}
    return line


def merge_kernel_name(op: str, dtype: int, K: int) -> str:
    """the merge kernel instance a workload's operator launches: whole-chunk consumers for
    TIES with up to 8 experts and DARE / DARE-TIES with up to 16, streaming consumers
    otherwise"""
    inst = {"ta": "AVG/TA", "avg": "AVG/TA", "ties": "TIES", "ties_masked": "TIES", "dare": "DARE",
            "avg_renorm": "AVG_RENORM", "dare_ties": "DARE_TIES"}[op]
    chunk = (inst == "TIES" and K <= 8) or (inst in ("DARE", "DARE_TIES") and K <= 16)
    return f"{'merge_chunk_kernel' if chunk else 'merge_tma_kernel'}<{'bf16' if dtype == 0 else 'f32'}, {inst}>"


def graph_replay(mp, step, mf, reps=20):
    """One step captured into a CUDA graph (catalog, plans and merges, on a capture stream)
    and replayed: the per-step time without the host's launch work.  Not part of `value`,
    which times the eager calls."""
    import torch
    torch.cuda.synchronize()
    s = torch.cuda.Stream()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        hs = step(mf, st=s)
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(s):
        g.replay()
        a.record(s)
        for _ in range(reps):
            g.replay()
        b.record(s)
    torch.cuda.synchronize()
    ms = a.elapsed_time(b) / reps
    for h in hs:  # the handles' memory first, then the graph
        h.free()
    del g
    return {"replay_ms_per_step": ms, "reps": reps}


def _union_ms(iv):
    """total length of a union of intervals [(t0, t1), ...]"""
    tot, end = 0.0, None
    for a, b in sorted(iv):
        if end is None or a > end:
            tot += b - a
            end = b
        elif b > end:
            tot += b - end
            end = b
    return tot


def _overlap_ms(a, b, iv):
    """length of [a, b] covered by the union of the intervals iv"""
    return _union_ms([(max(a, x), min(b, y)) for x, y in iv if min(b, y) > max(a, x)])


def host_timeline(mp, step, mf, budgets, trace_out=None):
    """One more step, untimed, with the device-time trace on: per call (the index, each
    budget's merge), the wall time, how busy the gather stream kept the host link, and how
    much of the segment kernels' time ran while a gather was in flight."""
    import torch
    torch.cuda.synchronize()
    mp.mp_trace_start(1 << 16)
    hs = step(mf)
    torch.cuda.synchronize()
    ranges = mp.mp_trace_stop()
    for h in hs:
        h.free()
    if trace_out:
        with open(trace_out, "w") as fo:
            fo.write("kind,segment,stream,t0_ms,t1_ms\n")
            for r in ranges:
                fo.write(f"{r['kind']},{r['segment']},{r['stream']},{r['t0_ms']:.4f},{r['t1_ms']:.4f}\n")
    calls = []   # ranges in enqueue order: a segment range belongs to the call begun before it
    for r in ranges:
        if r["kind"] in (mp.MP_TRACE_INDEX, mp.MP_TRACE_MERGE):
            calls.append({"call": r, "g": [], "k": []})
        elif r["kind"] == mp.MP_TRACE_GATHER and calls:
            calls[-1]["g"].append((r["t0_ms"], r["t1_ms"]))
        elif r["kind"] == mp.MP_TRACE_SEGMENT and calls:
            calls[-1]["k"].append((r["t0_ms"], r["t1_ms"]))
    out = []
    for c, name in zip(calls, ["index"] + [f"merge f={f}" for f in budgets]):
        wall = c["call"]["t1_ms"] - c["call"]["t0_ms"]
        kern = sum(b - a for a, b in c["k"])
        under = sum(_overlap_ms(a, b, c["g"]) for a, b in c["k"])
        out.append(dict(call=name, segments=len(c["g"]), wall_ms=wall, gather_busy_ms=_union_ms(c["g"]),
                        gather_busy_frac=_union_ms(c["g"]) / wall if wall > 0 else None, kernel_ms=kern,
                        kernel_under_gather_frac=under / kern if kern > 0 else None))
    return out


def time_hashes(mp, fam, mf, last, outs, shared_out, per_budget, stream, reps=3):
    """The catalog's block hashes (one pass over the K + 1 checkpoints) and Alg. 2's hash
    validation of the last budget's merge (base + selected expert blocks + output), timed
    with CUDA events after the timed region; not part of the step."""
    import torch

    idx, k = last[0], len(per_budget) - 1
    plan, man = last[1 + 2 * k], last[2 + 2 * k]
    out = outs[0 if shared_out else k]
    es, N = fam.elem_size, fam.n_params
    E = lambda: torch.cuda.Event(enable_timing=True)  # noqa: E731
    mp.mp_index_hashes(mf, idx, stream)
    mp.mp_manifest_validate(mf, idx, plan, out, man, stream)
    torch.cuda.synchronize()
    t_cat, t_val = [], []
    for _ in range(reps):
        a, b, c = E(), E(), E()
        a.record(stream)
        mp.mp_index_hashes(mf, idx, stream)
        b.record(stream)
        mp.mp_manifest_validate(mf, idx, plan, out, man, stream)
        c.record(stream)
        torch.cuda.synchronize()
        t_cat.append(a.elapsed_time(b))
        t_val.append(b.elapsed_time(c))
    v = mp.mp_manifest_validation(man, fam.n_blocks)
    peak, _ = hbm_peak()
    cat_bytes = (fam.K + 1) * N * es
    val_bytes = 2 * N * es + per_budget[k]["planned_bytes"]
    cat_ms, val_ms = statistics.median(t_cat), statistics.median(t_val)
    return {"catalog_ms": cat_ms, "catalog_bytes": cat_bytes, "catalog_gbs": cat_bytes / cat_ms / 1e6,
            "catalog_frac": cat_bytes / cat_ms / 1e6 / peak, "validate_f": per_budget[k]["f"],
            "validate_ms": val_ms, "validate_bytes": val_bytes, "validate_gbs": val_bytes / val_ms / 1e6,
            "validate_frac": val_bytes / val_ms / 1e6 / peak, "blocks_checked": v["checked"],
            "mismatched": v["mismatched"]}


def time_model_fit(budgets, per_budget, ckpt_bytes, c_full, peak_gbs, touched_mode):
    """The merge time against the affine model T(f) = (2 N s + f C_full) / BW: a least-squares
    line through the measured (planned fraction, merge ms) points, next to the model's slope
    C_full / BW and intercept 2 N s / BW at the measured copy bandwidth."""
    if len(budgets) < 2:
        return None
    x = [pb["planned_bytes"] / c_full for pb in per_budget]
    y = [pb["merge_ms"] for pb in per_budget]
    n = len(x)
    mx, my = sum(x) / n, sum(y) / n
    sxx = sum((a - mx) ** 2 for a in x)
    if sxx <= 0:
        return None
    slope = sum((a - mx) * (b - my) for a, b in zip(x, y)) / sxx
    icpt = my - slope * mx
    res = [b - (icpt + slope * a) for a, b in zip(x, y)]
    ss_tot = sum((b - my) ** 2 for b in y)
    r2 = 1.0 - sum(r * r for r in res) / ss_tot if ss_tot > 0 else 1.0
    return {"x": "planned expert bytes / C_full", "slope_ms": slope, "intercept_ms": icpt, "r2": r2,
            "model_slope_ms": c_full / (peak_gbs * 1e9) * 1e3,
            "model_intercept_ms": None if touched_mode else 2 * ckpt_bytes / (peak_gbs * 1e9) * 1e3,
            "bw_from_slope_gbs": c_full / (slope / 1e3) / 1e9 if slope > 0 else None}


def fidelity_vs_full(fam, budgets, outs, shared_out, per_budget):
    """Tab. 3's fidelity columns for every budget against the full-read merge of the same
    step (budget 1.0): relative L2 deviation ||M_A - M_full|| / ||M_full|| and the 95th
    percentile over blocks of ||d_b|| / ||M_full[b]||.  Reporting only: computed after the
    timed region, per tensor, in fp64 (the merge itself never runs here)."""
    import torch

    if shared_out or 1.0 not in budgets:
        return
    full = outs[budgets.index(1.0)]
    offs, nums, _ = fam.layout()
    E = fam.block_elems
    num2 = [0.0] * len(budgets)
    den2 = 0.0
    blk_rel = [[] for _ in budgets]
    for o, n in zip(offs.tolist(), nums.tolist()):
        nb = (n + E - 1) // E
        pad = nb * E - n

        def rows(t):
            x = t[o:o + n].double()
            return torch.nn.functional.pad(x, (0, pad)).view(nb, E)

        fr = rows(full)
        fb2 = (fr * fr).sum(1)
        den2 += float(fb2.sum())
        for k in range(len(budgets)):
            d = rows(outs[k]) - fr
            db2 = (d * d).sum(1)
            num2[k] += float(db2.sum())
            blk_rel[k].append(torch.sqrt(db2 / torch.clamp(fb2, min=1e-300)))
    for k, pb in enumerate(per_budget):
        rel = torch.cat(blk_rel[k]).float().cpu()
        pb["rel_l2_vs_full"] = (num2[k] / den2) ** 0.5 if den2 > 0 else 0.0
        pb["p95_block_dev_vs_full"] = float(torch.quantile(rel, 0.95)) if rel.numel() <= (1 << 24) else \
            float(rel.kthvalue(max(1, int(0.95 * rel.numel()))).values)


def measure_h2d(pinned_src) -> float:
    """host -> device copy bandwidth (GB/s) from the pinned pool: 256 MiB copies, best of 10"""
    import torch

    n = min(pinned_src.numel(), (256 << 20) // pinned_src.element_size())
    src = pinned_src[:n]
    dst = torch.empty(n, dtype=pinned_src.dtype, device="cuda")
    best = 0.0
    for _ in range(10):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        dst.copy_(src, non_blocking=True)
        b.record()
        b.synchronize()
        best = max(best, n * pinned_src.element_size() / (a.elapsed_time(b) / 1e3) / 1e9)
    return best


def host_mem_available() -> float:
    """bytes of host memory available now (MemAvailable), or +inf where it cannot be read"""
    try:
        with open("/proc/meminfo") as f:
            for line in f:
                if line.startswith("MemAvailable:"):
                    return float(line.split()[1]) * 1024.0
    except OSError:
        pass
    return float("inf")


def _max_over_ranks(x: float, world: int) -> float:
    """the largest x over the replicas (the slowest rank's time is the job's time)"""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist

    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def replica_value(units_per_rank: float, world: int, ms_per_step: float) -> float:
    """whole-job throughput of N independent replicas: every rank processes the same units
    per step, the step takes the slowest rank's time"""
    return world * units_per_rank / (ms_per_step / 1e3)


# ---- K-scaling at a fixed absolute budget (Cor. 1) --------------------------------------------------

def k_sweep(args):
    """Cor. 1: with the expert-read budget B fixed in bytes, the bytes a merge reads from the
    experts stay at most B however many experts the family has, while a full read grows as K.
    For Qwen2.5-0.5B-shaped families with K = 4 ... 32 and the operators of Tab. 1 (AVG, TIES,
    DARE), time the catalog, then plan + merge at the full budget (the naive full read) and at
    the fixed budget, all with CUDA events on the launching stream."""
    import torch
    import paper_2605_29489_gb300 as mp
    from paper_2605_29489_gb300 import synth

    torch.cuda.set_device(0)
    stream = torch.cuda.current_stream()
    ks = [int(k) for k in args.k_list.split(",")]
    rows = []
    launches0 = mp.mp_kernel_launch_count()
    clocks = ClockSampler(0)
    clocks.start()
    for K in ks:
        fam = synth.qwen25_05b(K=K)
        base, experts = fam.device_arrays()
        offs, nums, total = fam.layout()
        mf = mp.family(list(zip(offs.tolist(), nums.tolist())), base, experts, fam.block_elems, fam.dtype, 0)
        N, es = fam.n_params, fam.elem_size
        B_fixed = int(args.k_budget_experts * N * es)
        out = torch.empty_like(base)
        for opn in ("avg", "ties", "dare"):
            W = {"op": opn, "density": 0.2, "drop_p": 0.9}
            gop, _ = make_ops(W, K)
            t = {"index": [], "plan_full": [], "merge_full": [], "plan_fixed": [], "merge_fixed": []}
            info = {}
            for it in range(args.warmup + args.steps):
                ev = [torch.cuda.Event(enable_timing=True) for _ in range(6)]
                ev[0].record(stream)
                idx = mp.mp_index_blocks(mf, gop, stream)
                ev[1].record(stream)
                hs = [idx]
                for j, B in enumerate((mp.mp_budget_from_fraction(mf, 1.0), B_fixed)):
                    plan = mp.mp_plan(idx, gop, B, stream)
                    ev[2 + 2 * j].record(stream)
                    man = mp.mp_merge(mf, idx, plan, out, stream)
                    ev[3 + 2 * j].record(stream)
                    hs += [plan, man]
                torch.cuda.synchronize()
                if it >= args.warmup:
                    t["index"].append(ev[0].elapsed_time(ev[1]))
                    t["plan_full"].append(ev[1].elapsed_time(ev[2]))
                    t["merge_full"].append(ev[2].elapsed_time(ev[3]))
                    t["plan_fixed"].append(ev[3].elapsed_time(ev[4]))
                    t["merge_fixed"].append(ev[4].elapsed_time(ev[5]))
                if it == args.warmup + args.steps - 1:
                    for name, (pl, mn) in (("full", (hs[1], hs[2])), ("fixed", (hs[3], hs[4]))):
                        pi = mp.mp_plan_info(pl, with_arrays=False)
                        mi = mp.mp_manifest_info(mn, K)
                        info[name] = dict(planned_bytes=pi["chat"], realized_bytes=mi["realized_total"],
                                          touched_blocks=mi["touched"], n_selected=pi["n_sel"])
                for h in hs:
                    h.free()
            med = {k: statistics.median(v) for k, v in t.items()}
            rows.append(dict(K=K, op=opn, budget_fixed_bytes=B_fixed, c_full_bytes=K * N * es,
                             index_ms=med["index"],
                             full=dict(plan_ms=med["plan_full"], merge_ms=med["merge_full"], **info["full"]),
                             fixed=dict(plan_ms=med["plan_fixed"], merge_ms=med["merge_fixed"], **info["fixed"]),
                             io_reduction=1.0 - info["fixed"]["realized_bytes"] / max(1, info["full"]["realized_bytes"]),
                             merge_speedup=med["merge_full"] / med["merge_fixed"]))
        del base, experts, out, mf
        torch.cuda.empty_cache()
    clk = clocks.stop()
    launches = mp.mp_kernel_launch_count() - launches0
    fixed_ms = sum(r["fixed"]["merge_ms"] + r["fixed"]["plan_ms"] for r in rows)
    return {"metric": "merge time and expert-read bytes vs K at a fixed absolute budget (Cor. 1)",
            "value": statistics.mean(r["merge_speedup"] for r in rows), "unit": "x (full-read merge / fixed-budget merge)",
            "n_gpus": 1, "steps": args.steps, "warmup": args.warmup, "ms_per_step": fixed_ms / len(rows),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": "k-sweep", "family": "Qwen2.5-0.5B shapes", "K": ks,
                       "budget_fixed": f"{args.k_budget_experts} x one expert's bytes",
                       "ops": ["avg", "ties rho=0.2", "dare p=0.9"], "l2": "inputs larger than L2 (no flush)"},
            "rows": rows, "gpu_launches": launches, "clocks": clk}


# ---- reference arm (the CPU oracle) ----------------------------------------------------------------

def reference(args):
    W = workloads()[args.workload]
    fam = W["make"]()
    # about a minute of oracle work over all warm-up and timed steps, on one sample
    per_step = max(0.2, min(20.0, 60.0 / max(1, args.steps + args.warmup)))
    run, desc = oracle_sample(W, fam, per_step)
    for _ in range(args.warmup):
        run()
    vals, secs = [], []
    for _ in range(args.steps):
        v, dt = run()
        vals.append(v)
        secs.append(dt)
    v = statistics.mean(vals)
    model, ncpu = cpu_info()
    return {"impl": "reference", "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": 1, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1e3 * statistics.mean(secs), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16" if fam.dtype == 0 else "f32", "data": "synthetic",
            "config": {"workload": args.workload, "description": W["desc"], "budgets": W["budgets"]},
            "cpu_baseline": {"value": v, "unit": UNIT, "cores": 1, "kind": "oracle", "sample": desc,
                             "host_cpu": model, "host_cores_available": ncpu},
            "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1, help="GPUs (one process each under torchrun; independent replicas)")
    ap.add_argument("--steps", type=int, default=100, help="timed steps (one step = index, then plan + merge per budget)")
    ap.add_argument("--warmup", type=int, default=5, help="untimed warm-up steps (at least 3)")
    ap.add_argument("--impl", choices=["native", "reference"], default="native",
                    help="native: the CUDA path; reference: the CPU oracle on a bounded sample")
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=sorted(workloads().keys()),
                    help="synthetic family, operator and budgets")
    ap.add_argument("--no-e2e", action="store_true", help="skip the end-to-end leg (host buffers, copies timed)")
    ap.add_argument("--no-cpu-baseline", action="store_true", help="skip timing the CPU oracle")
    ap.add_argument("--no-hash", action="store_true", help="skip timing the block-hash passes")
    ap.add_argument("--cpu-seconds", type=float, default=15.0, help="CPU oracle work to time for cpu_baseline")
    ap.add_argument("--k-sweep", action="store_true",
                    help="K-scaling at a fixed absolute budget (Cor. 1) instead of the workload sweep")
    ap.add_argument("--k-list", default="4,8,16,32", help="expert counts of --k-sweep")
    ap.add_argument("--trace-out", default=None,
                    help="host-pool workloads: write the traced step's device-time ranges to this CSV")
    ap.add_argument("--k-budget-experts", type=float, default=0.25,
                    help="the fixed budget of --k-sweep, in units of one expert checkpoint's bytes")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        if rank == 0:
            print(json.dumps(reference(args)), flush=True)
        return
    if args.k_sweep:
        if rank == 0:
            print(json.dumps(k_sweep(args)), flush=True)
        return

    if world > 1:
        import torch
        import torch.distributed as dist

        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    line = native(args, rank, world, local_rank)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
