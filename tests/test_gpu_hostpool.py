"""Host-resident expert pool: experts in pinned host memory, base and output in HBM.

The library walks the family in segments.  For each segment a gather kernel on a side
stream reads the expert blocks over the host mapping (every block for the index, only the
planned (block, expert) pairs for the merge) into double-buffered HBM staging, while the
index or merge kernel works on the previous segment.
The results must be exactly those of the oracle (and of the device-resident path)."""
import numpy as np
import pytest
import torch

import oracle
from conftest import oracle_family
from test_gpu_fullsize import oracle_catalog, pool  # noqa: F401  (pool: the oracle's process pool fixture)
from test_gpu_parity import FRACS, fam_k9, fam_k17, fam_ragged_bf16, fam_ragged_f32, host, ops_for, run_case

pytestmark = pytest.mark.gpu

import paper_2605_29489_gb300 as mp  # noqa: E402
from paper_2605_29489_gb300 import synth  # noqa: E402


@pytest.mark.parametrize("make", [fam_ragged_bf16, fam_ragged_f32, fam_k9, fam_k17], ids=lambda f: f.__name__)
def test_hostpool_parity_small_families(make):
    fam = make()
    base, experts = fam.host_arrays()
    run_case(fam, base, experts, ("avg", "ties", "ties1", "dare", "ties_masked"), FRACS, host_experts=True)


def test_hostpool_multi_segment_matches_oracle_and_device_path(pool):  # noqa: F811
    """Qwen2.5-0.5B shapes (494M params, 16 segments), K=8: TA and TIES against the oracle's
    catalog, thresholds and plans, sampled merged blocks, and the device-resident run"""
    fam = synth.qwen25_05b()
    K = fam.K
    base_d, experts_d = fam.device_arrays()
    experts_h = [e.cpu().pin_memory() for e in experts_d]
    offs, nums, _ = fam.layout()
    tensors = list(zip(offs.tolist(), nums.tolist()))
    mf_dev = mp.family(tensors, base_d, experts_d, fam.block_elems, fam.dtype, 0)
    mf_host = mp.family(tensors, base_d, experts_h, fam.block_elems, fam.dtype, 1)
    bo, bl, bt = fam.block_table()
    rng = np.random.default_rng(3)
    samples = sorted({0, fam.n_blocks - 1, *[int(x) for x in rng.choice(fam.n_blocks, 10, replace=False)]})
    for gop, oop in [(mp.make_op(mp.MP_OP_TA, alpha=[0.3] * K), oracle.Op(oracle.TA, K, alpha=[0.3] * K)),
                     (mp.make_op(mp.MP_OP_TIES, density=0.2), oracle.Op(oracle.TIES, K, density=0.2))]:
        ties = oop.kind == oracle.TIES
        o_norm, o_max, o_nnz, o_tau = oracle_catalog(pool, ("qwen25_05b", ()), fam, 0.2 if ties else None)
        i_dev = mp.mp_index_blocks(mf_dev, gop)
        i_host = mp.mp_index_blocks(mf_host, gop)
        s_dev = mp.mp_index_stats(i_dev)
        s_host = mp.mp_index_stats(i_host)
        for a, b in zip(s_dev, s_host):
            assert np.array_equal(a.view(np.uint32), b.view(np.uint32))
        assert np.array_equal(s_host[0].view(np.uint32), o_norm.view(np.uint32))
        assert np.array_equal(s_host[1].view(np.uint32), o_max.view(np.uint32))
        assert np.array_equal(s_host[2], o_nnz)
        if ties:
            assert np.array_equal(s_host[3], o_tau)
        for f in (1.0, 0.25):
            B = mp.mp_budget_from_fraction(mf_host, f)
            p_dev, p_host = mp.mp_plan(i_dev, gop, B), mp.mp_plan(i_host, gop, B)
            pi = mp.mp_plan_info(p_host, i_host)
            opl = oracle.plan(K, bl, bt, len(fam.tensors), fam.elem_size, oop, o_norm, o_max, o_nnz, o_tau, B)
            assert pi["digest"] == opl["digest"] and np.array_equal(pi["mask"], opl["mask"])
            assert pi["digest"] == mp.mp_plan_info(p_dev, i_dev)["digest"]
            o_dev, o_host = torch.empty_like(base_d), torch.empty_like(base_d)
            m_dev = mp.mp_merge(mf_dev, i_dev, p_dev, o_dev)
            m_host = mp.mp_merge(mf_host, i_host, p_host, o_host)
            mi = mp.mp_manifest_info(m_host, K)
            assert mi["realized_total"] == pi["chat"] <= B
            assert torch.equal(o_dev.view(torch.int16), o_host.view(torch.int16))
            for b in samples:
                hb, hex_ = fam.block_host(b)
                tau_k = o_tau[:, bt[b]] if ties else None
                want = oracle.merge_block(fam.dtype, int(bo[b]), hb, hex_, int(opl["mask"][b]), oop, tau_k)
                got = host(fam, o_host[int(bo[b]):int(bo[b] + bl[b])])
                assert np.array_equal(got, want), (f, b)
            for h in (m_dev, m_host, p_dev, p_host):
                h.free()
        i_dev.free()
        i_host.free()
