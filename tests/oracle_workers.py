"""Process-pool workers that run the CPU oracle over a whole full-size family.

Each worker regenerates the blocks it is given on the host (from the seeded
generator, never from the GPU) and computes the oracle's statistics; for TIES it
works tensor by tensor and also returns the trim thresholds.  Used only by the
full-size parity tests; the pool is started with the 'spawn' method.
"""
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

_FAMILIES = {}


def init_worker():
    if ROOT not in sys.path:
        sys.path.insert(0, ROOT)


def family(spec):
    """spec = (constructor name, kwargs tuple)"""
    if spec not in _FAMILIES:
        from paper_2605_29489_gb300 import synth

        name, kw = spec
        _FAMILIES[spec] = getattr(synth, name)(**dict(kw))
    return _FAMILIES[spec]


def block_stats(spec, blocks):
    """oracle (norm, maxabs, nnz) [K, len(blocks)] for the given blocks"""
    import oracle

    fam = family(spec)
    K = fam.K
    out_n = np.zeros((K, len(blocks)), np.float32)
    out_m = np.zeros((K, len(blocks)), np.float32)
    out_z = np.zeros((K, len(blocks)), np.uint32)
    for j, b in enumerate(blocks):
        base, experts = fam.block_host(int(b))
        for i in range(K):
            n, m, z, _ = oracle.block_stats(fam.dtype, base, experts[i])
            out_n[i, j], out_m[i, j], out_z[i, j] = n, m, z
    return blocks, out_n, out_m, out_z


def tensor_stats_and_tau(spec, t, density):
    """oracle statistics of every block of tensor t and its TIES thresholds tau[K]"""
    import oracle

    fam = family(spec)
    K = fam.K
    bo, bl, bt = fam.block_table()
    blocks = np.nonzero(bt == t)[0]
    hist = [np.zeros(32768, np.uint64) for _ in range(K)]
    out_n = np.zeros((K, len(blocks)), np.float32)
    out_m = np.zeros((K, len(blocks)), np.float32)
    out_z = np.zeros((K, len(blocks)), np.uint32)
    for j, b in enumerate(blocks):
        base, experts = fam.block_host(int(b))
        for i in range(K):
            n, m, z, _ = oracle.block_stats(fam.dtype, base, experts[i])
            out_n[i, j], out_m[i, j], out_z[i, j] = n, m, z
            oracle.key_hist(fam.dtype, base, experts[i], hist[i])
    numel = int(bl[blocks].sum())
    tau = np.array([oracle.tau_from_hist(hist[i], numel, density) for i in range(K)], np.uint32)
    return t, blocks, out_n, out_m, out_z, tau


def merged_hashes(spec, blocks, cases):
    """the oracle's merge of each given block under every budget's mask of every case,
    hashed like the catalog's blocks.  cases: [(op_args, masks [n_budgets, len(blocks)],
    tau [K, n_tensors] or None)], op_args = (kind, K, kwargs) of oracle.Op (trim group =
    tensor).  Returns (blocks, [uint64 [n_budgets, len(blocks)] per case]); each block is
    regenerated once for all cases."""
    import oracle

    fam = family(spec)
    bo, bl, bt = fam.block_table()
    ops = [oracle.Op(a[0], a[1], **dict(a[2])) for a, _, _ in cases]
    outs = [np.zeros((m.shape[0], len(blocks)), np.uint64) for _, m, _ in cases]
    for j, b in enumerate(blocks):
        base, experts = fam.block_host(int(b))
        for (args, masks, tau), op, out in zip(cases, ops, outs):
            tau_k = None if tau is None else np.ascontiguousarray(tau[:, bt[b]])
            for k in range(masks.shape[0]):
                merged = oracle.merge_block(fam.dtype, int(bo[b]), base, experts, int(masks[k, j]), op, tau_k)
                out[k, j] = oracle.block_hash(merged.tobytes())
    return blocks, outs
