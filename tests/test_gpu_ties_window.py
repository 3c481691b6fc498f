"""TIES thresholds taken from predicted windows: both exact paths against the oracle.

For device-resident experts the catalog predicts, from a sample of every block of each
trim group, the coarse key bin that holds the threshold, and counts a window of 384 keys
around it at full resolution.  A pair whose threshold lies
outside its window takes the two-level select instead.  The families here are built so
that the sample mispredicts (the blocks it weighs most carry deltas far larger than the
others'), or so that the threshold is the key of an exact zero; thresholds,
plans and merges must still be the oracle's, bit for bit.
"""
import numpy as np
import pytest
import torch

import oracle
from conftest import oracle_family
from test_gpu_parity import run_case, upload

pytestmark = pytest.mark.gpu

import paper_2605_29489_gb300 as mp  # noqa: E402
from paper_2605_29489_gb300 import synth  # noqa: E402

E = 4096


def _bf16_bits(x):
    return torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(torch.bfloat16).view(torch.int16).numpy() \
        .view(np.uint16)


def _f32(bits):
    return (bits.astype(np.uint32) << 16).view(np.float32)


def _with_deltas(fam, scale_of_block, seed):
    """the family's base, and experts = bf16(base + scale(b) * N(0, 1)) per block b"""
    base, _ = fam.host_arrays()
    bo, bl, _ = fam.block_table()
    rng = np.random.default_rng(seed)
    b32 = _f32(base)
    experts = []
    for i in range(fam.K):
        d = np.zeros_like(b32)
        for b in range(fam.n_blocks):
            s = slice(int(bo[b]), int(bo[b] + bl[b]))
            d[s] = scale_of_block(i, b) * rng.standard_normal(int(bl[b])).astype(np.float32)
        experts.append(_bf16_bits(b32 + d))
    return base, experts


@pytest.mark.parametrize("host_experts", [False, True], ids=["device", "host_pool"])
def test_sample_that_misses_the_threshold_falls_back_to_the_two_level_select(host_experts):
    """The sample reads 32 vectors of every block longer than 4096 elements and every vector
    of a shorter one, so short blocks weigh far more in it.  Here the short blocks (a
    tensor's tail, small tensors) carry deltas about 10^4 times larger than the full
    blocks: the sample predicts a window among the large keys while the threshold lies
    among the small ones — for tensor 0 with per-tensor trim groups, and for the single
    group of trim scope 1.  The two-level select must give the oracle's thresholds — also
    with the experts in pinned host memory, where the sample reads them in place and the
    fallback walk's gathers run only because a pair was marked."""
    E = 65536
    shapes = [2 * E + 4000, 16 * E] + [4096] * 20 + [70001]
    fam = synth.custom(shapes, dtype=synth.BF16, block_elems=E, K=3, active_frac=0.5, name="window-miss")
    _, bl, bt = fam.block_table()

    def scale(i, b):
        t = int(bt[b])
        if t <= 1:
            return 0.5 if bl[b] <= 4096 else 1e-4
        if t < len(shapes) - 1:
            return 0.5
        return 1e-3 * (1 + i)

    base, experts = _with_deltas(fam, scale, seed=11)
    run_case(fam, base, experts, ("ties", "ties1"), [1.0, 0.5, 0.25], host_experts=host_experts)
    # the threshold of tensor 0 lies among its small deltas, far below the sampled ones
    mf, _, _ = upload(fam, base, experts, host_experts)
    idx = mp.mp_index_blocks(mf, mp.make_op(mp.MP_OP_TIES, lam=1.0, density=0.2))
    tau = mp.mp_index_stats(idx)[3]
    key_mid = int(_bf16_bits(np.float32([1e-2]))[0]) & 0x7FFF
    assert np.all(tau[:, 0] < key_mid)
    idx.free()


@pytest.mark.parametrize("host_experts", [False, True], ids=["device", "host_pool"])
@pytest.mark.parametrize("density", [0.5, 0.9, 1.0])
def test_threshold_at_the_key_of_an_exact_zero(density, host_experts):
    """nine blocks in ten have no delta at all: from density 0.5 on, the k-th largest key
    is the key 0 of an exact zero, reached through the window at the bottom of the keys"""
    fam = synth.custom([64 * E, 5 * E + 3], dtype=synth.BF16, block_elems=E, K=3, active_frac=0.5,
                       name="window-zero")
    base, experts = _with_deltas(fam, lambda i, b: 1e-2 if b % 10 == 3 else 0.0, seed=12)
    mf, _, _ = upload(fam, base, experts, host_experts)
    gop = mp.make_op(mp.MP_OP_TIES, lam=1.0, density=density)
    idx = mp.mp_index_blocks(mf, gop)
    tau = mp.mp_index_stats(idx)[3]
    want = oracle.ties_thresholds(oracle_family(fam, base, experts), density)
    assert np.array_equal(tau, want)
    assert np.all(want == 0)
    idx.free()
