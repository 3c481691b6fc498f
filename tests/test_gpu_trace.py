"""Device-time trace of the calls (mp_trace_start / mp_trace_stop).

On device-resident inputs a traced index, plan and merge give one range each, in stream
order.  On a host-resident pool (Qwen2.5-0.5B shapes, 16 segments) every segment adds a
gather range on the side stream and a kernel range on the caller's stream; the trace then
shows the pipeline's two dependencies: a segment's kernels start after its gather ends
(the staging buffer is full), and the gather of segment s + 2 starts after the kernels of
segment s end (it refills the buffer they read)."""
import pytest
import torch

pytestmark = pytest.mark.gpu

import paper_2605_29489_gb300 as mp  # noqa: E402
from paper_2605_29489_gb300 import synth  # noqa: E402

TOL_MS = 0.01  # event timestamps are exact to about half a microsecond


def _by_kind(ranges, kind):
    return [r for r in ranges if r["kind"] == kind]


def test_trace_of_index_plan_merge_in_stream_order():
    fam = synth.custom([3 * 65536 + 17, 5 * 65536], dtype=synth.BF16, block_elems=65536, K=4, active_frac=0.5,
                       name="trace")
    base, experts = fam.device_arrays()
    offs, nums, _ = fam.layout()
    mf = mp.family(list(zip(offs.tolist(), nums.tolist())), base, experts, fam.block_elems, fam.dtype, 0)
    gop = mp.make_op(mp.MP_OP_TIES, density=0.2)
    mp.mp_trace_start(64)
    idx = mp.mp_index_blocks(mf, gop)
    pl = mp.mp_plan(idx, gop, mp.mp_budget_from_fraction(mf, 0.5))
    out = torch.empty_like(base)
    man = mp.mp_merge(mf, idx, pl, out)
    ranges = mp.mp_trace_stop()
    assert [r["kind"] for r in ranges] == [mp.MP_TRACE_INDEX, mp.MP_TRACE_PLAN, mp.MP_TRACE_MERGE]
    for r in ranges:
        assert 0.0 <= r["t0_ms"] <= r["t1_ms"] and r["stream"] == 0
    assert ranges[0]["t0_ms"] == 0.0
    for a, b in zip(ranges, ranges[1:]):
        assert a["t1_ms"] <= b["t0_ms"] + TOL_MS
    # nothing is recorded once the trace has stopped
    mp.mp_merge(mf, idx, pl, out).free()
    mp.mp_trace_start(8)
    assert mp.mp_trace_stop() == []
    for h in (man, pl, idx):
        h.free()


def test_trace_of_host_pool_segments_shows_the_pipeline_dependencies():
    fam = synth.qwen25_05b()
    base_d, experts_d = fam.device_arrays()
    experts_h = [e.cpu().pin_memory() for e in experts_d]
    del experts_d
    offs, nums, _ = fam.layout()
    mf = mp.family(list(zip(offs.tolist(), nums.tolist())), base_d, experts_h, fam.block_elems, fam.dtype, 1)
    gop = mp.make_op(mp.MP_OP_TA, alpha=[0.3] * fam.K)
    idx = mp.mp_index_blocks(mf, gop)
    pl = mp.mp_plan(idx, gop, mp.mp_budget_from_fraction(mf, 1.0))
    out = torch.empty_like(base_d)
    mp.mp_trace_start(1024)
    man = mp.mp_merge(mf, idx, pl, out)
    ranges = mp.mp_trace_stop()
    merge = _by_kind(ranges, mp.MP_TRACE_MERGE)
    gathers = _by_kind(ranges, mp.MP_TRACE_GATHER)
    kernels = _by_kind(ranges, mp.MP_TRACE_SEGMENT)
    assert len(merge) == 1
    n = len(gathers)
    assert n >= 8 and len(kernels) == n
    assert [g["segment"] for g in gathers] == list(range(n)) == [k["segment"] for k in kernels]
    assert all(g["stream"] == 1 for g in gathers) and all(k["stream"] == 0 for k in kernels)
    for s in range(n):
        assert kernels[s]["t0_ms"] >= gathers[s]["t1_ms"] - TOL_MS
        if s + 2 < n:
            assert gathers[s + 2]["t0_ms"] >= kernels[s]["t1_ms"] - TOL_MS
        assert merge[0]["t0_ms"] - TOL_MS <= gathers[s]["t0_ms"] and kernels[s]["t1_ms"] <= merge[0]["t1_ms"] + TOL_MS
    for h in (man, pl, idx):
        h.free()
