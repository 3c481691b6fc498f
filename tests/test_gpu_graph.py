"""A merge step captured into a CUDA graph and replayed.

The calls enqueue only kernels, stream-ordered allocations and event records, so one step
(catalog, a plan and a merge per budget) can be captured on a stream and replayed: every
replay recomputes the catalog, the plans and the merges from the current contents of the
family's buffers into the handles made during the capture.  The outputs of a replay must be
the eager step's, bit for bit — also after the experts' contents change between replays —
and the accessors of the captured handles must read the latest replay."""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

import paper_2605_29489_gb300 as mp  # noqa: E402
from paper_2605_29489_gb300 import synth  # noqa: E402


def _same(fam, a, b):
    """the elements of the family's tensors are equal bit for bit (the alignment gaps between
    tensors belong to no tensor and are never written)"""
    offs, nums, _ = fam.layout()
    return all(torch.equal(a[o:o + n].view(torch.int16), b[o:o + n].view(torch.int16))
               for o, n in zip(offs.tolist(), nums.tolist()))


def _family():
    fam = synth.custom([3 * 4096 + 77, 5 * 4096, 999], dtype=synth.BF16, block_elems=4096, K=3, active_frac=0.5,
                       name="graph")
    base, experts = fam.device_arrays()
    offs, nums, _ = fam.layout()
    mf = mp.family(list(zip(offs.tolist(), nums.tolist())), base, experts, fam.block_elems, fam.dtype, 0)
    return fam, base, experts, mf


@pytest.mark.parametrize("kind", ["ties", "ta", "dare"])
def test_captured_step_replays_the_eager_step(kind):
    fam, base, experts, mf = _family()
    gop = {"ties": mp.make_op(mp.MP_OP_TIES, density=0.2),
           "ta": mp.make_op(mp.MP_OP_TA, alpha=[0.3] * 3),
           "dare": mp.make_op(mp.MP_OP_DARE, alpha=[1 / 3] * 3, drop_p=0.9, seed=5)}[kind]
    Bs = [mp.mp_budget_from_fraction(mf, f) for f in (1.0, 0.25)]
    s = torch.cuda.Stream()

    def step(outs):
        hs = [mp.mp_index_blocks(mf, gop, s)]
        for k, B in enumerate(Bs):
            pl = mp.mp_plan(hs[0], gop, B, s)
            hs += [pl, mp.mp_merge(mf, hs[0], pl, outs[k], s)]
        return hs

    def eager():
        outs = [torch.empty_like(base) for _ in Bs]
        with torch.cuda.stream(s):
            hs = step(outs)
        s.synchronize()
        infos = [mp.mp_manifest_info(hs[2 + 2 * k], 3)["realized_total"] for k in range(len(Bs))]
        for h in hs:
            h.free()
        return [o.clone() for o in outs], infos

    want, want_info = eager()
    outs = [torch.zeros_like(base) for _ in Bs]
    with torch.cuda.stream(s):  # warm the library up on this stream before capturing
        for h in step(outs):
            h.free()
    s.synchronize()
    for o in outs:
        o.zero_()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        hs = step(outs)
    g.replay()
    torch.cuda.synchronize()
    for o, w in zip(outs, want):
        assert _same(fam, o, w)
    assert [mp.mp_manifest_info(hs[2 + 2 * k], 3)["realized_total"] for k in range(len(Bs))] == want_info

    # new expert contents, the same buffers: a replay gives the eager step on the new data
    experts[1].copy_(experts[2])
    experts[0].add_(torch.full_like(experts[0], 2.0 ** -7))
    want2, want2_info = eager()
    assert not all(_same(fam, a, b) for a, b in zip(want, want2))  # the new data changes the merge
    g.replay()
    torch.cuda.synchronize()
    for o, w in zip(outs, want2):
        assert _same(fam, o, w)
    assert [mp.mp_manifest_info(hs[2 + 2 * k], 3)["realized_total"] for k in range(len(Bs))] == want2_info
    norm = mp.mp_index_stats(hs[0])[0]
    assert np.all(np.isfinite(norm))
    torch.cuda.synchronize()
    for h in hs:  # the handles' memory first, then the graph
        h.free()
    del g


def test_capture_while_the_pinned_staging_is_in_use():
    """a family whose block table needs the largest pinned staging slot, captured while an
    eager index still holds the slot: the capture takes a new slot (a host allocation made in
    relaxed capture mode) and the replay gives the eager merge"""
    fam = synth.custom([2000 * 4096 + 123], dtype=synth.BF16, block_elems=4096, K=2, active_frac=0.5,
                       name="graph-big")
    base, experts = fam.device_arrays()
    offs, nums, _ = fam.layout()
    mf = mp.family(list(zip(offs.tolist(), nums.tolist())), base, experts, fam.block_elems, fam.dtype, 0)
    gop = mp.make_op(mp.MP_OP_TA, alpha=[0.5, 0.5])
    B = mp.mp_budget_from_fraction(mf, 0.25)
    s = torch.cuda.Stream()
    held = mp.mp_index_blocks(mf, gop)  # holds its staging slot until freed
    want = torch.empty_like(base)
    with torch.cuda.stream(s):
        idx_e = mp.mp_index_blocks(mf, gop, s)  # kept: every slot made so far stays taken
        pl = mp.mp_plan(idx_e, gop, B, s)
        man = mp.mp_merge(mf, idx_e, pl, want, s)
    s.synchronize()
    for h in (man, pl):
        h.free()
    out = torch.zeros_like(base)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        idx = mp.mp_index_blocks(mf, gop, s)
        pl = mp.mp_plan(idx, gop, B, s)
        man = mp.mp_merge(mf, idx, pl, out, s)
    g.replay()
    torch.cuda.synchronize()
    assert _same(fam, out, want)
    assert mp.mp_manifest_info(man, 2)["realized_total"] <= B
    for h in (man, pl, idx, idx_e, held):
        h.free()
    del g
