"""Seeded synthetic checkpoint families (input generator shared by the oracle's
test inputs and the GPU path).

A family is a base checkpoint and K experts in one flat buffer each.  Tensors
lie in checkpoint order, each starting on a 16-byte boundary, and are split
into blocks of ``block_elems`` contiguous elements (the last block of a tensor
may be partial; no block crosses a tensor).  Expert i differs from the base by
a per-(expert, block) scale times an approximate standard normal variate:

* active blocks: scale ~ lognormal(log_mu, log_sigma);
* inactive blocks: scale = ``inactive_scale`` (1e-7; bf16 storage rounds it away
  for about 99.9 % of the elements, all but those whose base is near zero).

The active set is either one set shared by all experts (a seeded choice of
exactly floor(active_frac * n_blocks) blocks) or an independent set per expert.
The element recipe lives in ``synth_core.h``; this module only builds the block
and scale tables and calls the host (C, pthreads) or device (CUDA) fill.
Nothing here computes any part of the merge method.
"""
from __future__ import annotations

import ctypes
import math
import os
from dataclasses import dataclass, field

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))

BF16 = 0
F32 = 1
_GAMMA = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)


def _mix64(z: np.ndarray) -> np.ndarray:
    """SplitMix64 output function on a uint64 array (wrapping arithmetic)."""
    z = np.asarray(z, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = (z ^ (z >> np.uint64(30))) * _M1
        z = (z ^ (z >> np.uint64(27))) * _M2
    return z ^ (z >> np.uint64(31))


def _stream_key(seed: int, stream: int) -> np.uint64:
    with np.errstate(over="ignore"):
        v = np.uint64(seed & 0xFFFFFFFFFFFFFFFF) + _GAMMA * np.uint64(stream + 1)
    return _mix64(np.array([v], dtype=np.uint64))[0]


def _uniform01(seed: int, stream: int, idx: np.ndarray) -> np.ndarray:
    """uniforms in (0, 1] from a keyed SplitMix64 stream, 53-bit resolution"""
    key = _stream_key(seed, stream)
    with np.errstate(over="ignore"):
        w = _mix64(key + _GAMMA * (idx.astype(np.uint64) + np.uint64(1)))
    return ((w >> np.uint64(11)).astype(np.float64) + 1.0) * (1.0 / 9007199254740992.0)


@dataclass
class Family:
    """A synthetic checkpoint family: tensor shapes, block size, K and delta model."""

    name: str
    dtype: int                       # BF16 or F32
    tensors: list                    # [(name, numel)] in checkpoint order
    block_elems: int
    K: int
    active_frac: float
    log_mu: float
    log_sigma: float
    per_expert_active: bool = False
    inactive_scale: float = 1e-7
    seed: int = 0
    _cache: dict = field(default_factory=dict, repr=False, compare=False)

    @property
    def elem_size(self) -> int:
        return 2 if self.dtype == BF16 else 4

    @property
    def torch_dtype(self):
        import torch
        return torch.bfloat16 if self.dtype == BF16 else torch.float32

    @property
    def np_dtype(self):
        return np.uint16 if self.dtype == BF16 else np.float32

    def layout(self):
        """(offsets, numels, total_elems): each tensor starts on a 16-byte boundary"""
        if "layout" not in self._cache:
            align = 16 // self.elem_size
            off, offs, nums = 0, [], []
            for _, n in self.tensors:
                off = (off + align - 1) // align * align
                offs.append(off)
                nums.append(int(n))
                off += int(n)
            total = (off + align - 1) // align * align
            self._cache["layout"] = (np.array(offs, np.uint64), np.array(nums, np.uint64), total)
        return self._cache["layout"]

    @property
    def total_elems(self) -> int:
        return self.layout()[2]

    @property
    def n_params(self) -> int:
        return int(sum(int(n) for _, n in self.tensors))

    def block_table(self):
        """(blk_off uint64, blk_len uint32, blk_tensor uint32) in global block order"""
        if "blocks" not in self._cache:
            offs, nums, _ = self.layout()
            E = self.block_elems
            bo, bl, bt = [], [], []
            for t, (o, n) in enumerate(zip(offs.tolist(), nums.tolist())):
                nb = (n + E - 1) // E
                starts = o + E * np.arange(nb, dtype=np.uint64)
                lens = np.minimum(np.uint64(E), np.uint64(o + n) - starts)
                bo.append(starts)
                bl.append(lens.astype(np.uint32))
                bt.append(np.full(nb, t, np.uint32))
            self._cache["blocks"] = (np.concatenate(bo) if bo else np.zeros(0, np.uint64),
                                     np.concatenate(bl) if bl else np.zeros(0, np.uint32),
                                     np.concatenate(bt) if bt else np.zeros(0, np.uint32))
        return self._cache["blocks"]

    @property
    def n_blocks(self) -> int:
        return int(self.block_table()[0].shape[0])

    def active_mask(self) -> np.ndarray:
        """bool [K, n_blocks]: which (expert, block) pairs carry a lognormal-scale delta"""
        nb = self.n_blocks
        n_act = int(math.floor(self.active_frac * nb))
        act = np.zeros((self.K, nb), dtype=bool)
        b = np.arange(nb, dtype=np.uint64)
        sets = range(self.K) if self.per_expert_active else [None]
        for s in sets:
            stream = 0x1000 + (0 if s is None else 1 + s)
            key = _stream_key(self.seed, stream)
            with np.errstate(over="ignore"):
                rank_key = _mix64(key + _GAMMA * (b + np.uint64(1)))
            chosen = np.argsort(rank_key, kind="stable")[:n_act]
            if s is None:
                act[:, chosen] = True
            else:
                act[s, chosen] = True
        return act

    def scales(self) -> np.ndarray:
        """float32 [K, n_blocks] per-(expert, block) delta scale"""
        if "scales" not in self._cache:
            nb = self.n_blocks
            act = self.active_mask()
            sc = np.full((self.K, nb), np.float32(self.inactive_scale), dtype=np.float32)
            idx = np.arange(nb, dtype=np.uint64)
            for i in range(self.K):
                u1 = _uniform01(self.seed, 0x2000 + 2 * i, idx)
                u2 = _uniform01(self.seed, 0x2001 + 2 * i, idx)
                g = np.sqrt(-2.0 * np.log(u1)) * np.cos(2.0 * np.pi * u2)
                s = np.exp(self.log_mu + self.log_sigma * g).astype(np.float32)
                sc[i, act[i]] = s[act[i]]
            self._cache["scales"] = sc
        return self._cache["scales"]

    # ---- host fill -------------------------------------------------------------------
    def fill_base_host(self, j0: int = 0, n: int | None = None, nthreads: int = 0) -> np.ndarray:
        n = self.total_elems - j0 if n is None else n
        out = np.empty(n, dtype=self.np_dtype)
        _host_fill(self, 0, j0, n, None, out, nthreads)
        return out

    def fill_expert_host(self, i: int, base_stored: np.ndarray, j0: int = 0, nthreads: int = 0) -> np.ndarray:
        n = int(base_stored.shape[0])
        out = np.empty(n, dtype=self.np_dtype)
        _host_fill(self, 1 + i, j0, n, base_stored, out, nthreads)
        return out

    def host_arrays(self, nthreads: int = 0):
        """(base, [experts]) as numpy arrays of the storage dtype (uint16 bits for bf16)"""
        base = self.fill_base_host(nthreads=nthreads)
        return base, [self.fill_expert_host(i, base, nthreads=nthreads) for i in range(self.K)]

    def block_host(self, b: int):
        """(base, [experts]) for block b alone, regenerated on the host"""
        bo, bl, _ = self.block_table()
        j0, n = int(bo[b]), int(bl[b])
        base = self.fill_base_host(j0, n, nthreads=1)
        return base, [self.fill_expert_host(i, base, j0, nthreads=1) for i in range(self.K)]

    # ---- device fill -----------------------------------------------------------------
    def device_arrays(self, device="cuda", stream=None):
        """(base, [experts]) as torch tensors on the GPU (bf16 or fp32)"""
        import torch
        lib = _dev_lib()
        st = torch.cuda.current_stream(device) if stream is None else stream
        n = self.total_elems
        bo, bl, _ = self.block_table()
        d_bo = torch.from_numpy(bo.view(np.int64)).to(device)
        d_bl = torch.from_numpy(bl.view(np.int32)).to(device)
        base = torch.empty(n, dtype=self.torch_dtype, device=device)
        rc = lib.syn_dev_fill_base(self.dtype, ctypes.c_uint64(self.seed), ctypes.c_uint64(n),
                                   ctypes.c_void_p(base.data_ptr()), ctypes.c_void_p(st.cuda_stream))
        if rc != 0:
            raise RuntimeError(f"synthetic base fill failed ({rc})")
        sc = torch.from_numpy(self.scales()).to(device)
        experts = []
        maxlen = int(bl.max()) if bl.size else 0
        for i in range(self.K):
            e = torch.empty(n, dtype=self.torch_dtype, device=device)
            rc = lib.syn_dev_fill_expert(self.dtype, ctypes.c_uint64(self.seed), ctypes.c_uint32(i),
                                         ctypes.c_uint64(n), ctypes.c_uint64(self.n_blocks),
                                         ctypes.c_void_p(d_bo.data_ptr()), ctypes.c_void_p(d_bl.data_ptr()),
                                         ctypes.c_void_p(sc[i].data_ptr()), ctypes.c_uint32(maxlen),
                                         ctypes.c_void_p(base.data_ptr()), ctypes.c_void_p(e.data_ptr()),
                                         ctypes.c_void_p(st.cuda_stream))
            if rc != 0:
                raise RuntimeError(f"synthetic expert fill failed ({rc})")
            experts.append(e)
        st.synchronize()
        return base, experts


# ---- shapes of the checkpoint families --------------------------------------------------

def _qwen2_tensors(hidden, layers, n_q, n_kv, inter, vocab, head_dim=None):
    hd = head_dim or hidden // n_q
    kv = n_kv * hd
    t = [("embed_tokens", vocab * hidden)]
    for l in range(layers):
        p = f"layers.{l}."
        t += [(p + "input_layernorm", hidden),
              (p + "q_proj.weight", hidden * n_q * hd), (p + "q_proj.bias", n_q * hd),
              (p + "k_proj.weight", kv * hidden), (p + "k_proj.bias", kv),
              (p + "v_proj.weight", kv * hidden), (p + "v_proj.bias", kv),
              (p + "o_proj.weight", hidden * n_q * hd),
              (p + "post_attention_layernorm", hidden),
              (p + "gate_proj", inter * hidden), (p + "up_proj", inter * hidden),
              (p + "down_proj", hidden * inter)]
    t.append(("norm", hidden))
    return t


def _llama_tensors(hidden, layers, n_q, n_kv, inter, vocab, embeddings=True):
    hd = hidden // n_q
    kv = n_kv * hd
    t = [("embed_tokens", vocab * hidden)] if embeddings else []
    for l in range(layers):
        p = f"layers.{l}."
        t += [(p + "input_layernorm", hidden),
              (p + "q_proj", hidden * hidden), (p + "k_proj", kv * hidden), (p + "v_proj", kv * hidden),
              (p + "o_proj", hidden * hidden), (p + "post_attention_layernorm", hidden),
              (p + "gate_proj", inter * hidden), (p + "up_proj", inter * hidden),
              (p + "down_proj", hidden * inter)]
    t += [("norm", hidden), ("lm_head", vocab * hidden)] if embeddings else [("norm", hidden)]
    return t


def tiny(seed: int = 0) -> Family:
    """8 fp32 tensors of 512x512, 4096-element blocks, K=4, lognormal(ln 1e-3, 1) on 30% of blocks"""
    return Family("tiny-fp32", F32, [(f"w{t}", 512 * 512) for t in range(8)], 4096, 4,
                  active_frac=0.3, log_mu=math.log(1e-3), log_sigma=1.0, seed=seed)


def qwen25_05b(seed: int = 0, K: int = 8, layers: int = 24) -> Family:
    """Qwen2.5-0.5B shapes (hidden 896, 24 layers, 14/2 heads, inter 4864, vocab 151936 tied), bf16"""
    name = "qwen2.5-0.5b" if layers == 24 else f"qwen2.5-0.5b-{layers}l"
    return Family(name, BF16, _qwen2_tensors(896, layers, 14, 2, 4864, 151936), 65536, K,
                  active_frac=0.3, log_mu=math.log(1e-3), log_sigma=1.0, seed=seed)


def llama3_8b(seed: int = 0, K: int = 4, layers: int = 32) -> Family:
    """Llama-3-8B shapes (hidden 4096, 32 layers, 32/8 heads, inter 14336, vocab 128256 untied), bf16.
    With fewer layers (a profiling case) the embedding and lm_head are left out as well, so
    that the family holds only transformer layers (218,112,000 parameters each) and a norm."""
    if layers == 32:
        return Family("llama-3-8b", BF16, _llama_tensors(4096, 32, 32, 8, 14336, 128256), 65536, K,
                      active_frac=0.4, log_mu=math.log(2e-4), log_sigma=1.2, seed=seed)
    return Family(f"llama-3-8b-{layers}l", BF16, _llama_tensors(4096, layers, 32, 8, 14336, 128256, False), 65536,
                  K, active_frac=0.4, log_mu=math.log(2e-4), log_sigma=1.2, seed=seed)


def qwen25_15b(seed: int = 0, K: int = 16, layers: int = 28) -> Family:
    """Qwen2.5-1.5B shapes (hidden 1536, 28 layers, 12/2 heads, inter 8960, vocab 151936 tied), bf16,
    per-expert active subsets of 25% of blocks"""
    name = "qwen2.5-1.5b" if layers == 28 else f"qwen2.5-1.5b-{layers}l"
    return Family(name, BF16, _qwen2_tensors(1536, layers, 12, 2, 8960, 151936), 65536, K,
                  active_frac=0.25, log_mu=math.log(1e-3), log_sigma=1.0, per_expert_active=True, seed=seed)


def missing_entries(fam: Family, K: int, seed: int = 2605, pair_frac: float = 0.10,
                    entry_frac: float = 0.001) -> np.ndarray:
    """A seeded pattern of catalog entries without statistics, bool [K, n_blocks]: every entry
    of a pair_frac share of the (expert, tensor) pairs (always the largest tensor of expert
    0) and an entry_frac share of the other entries.  Input generation only: which entries
    a saved catalog lacks."""
    _, _, bt = fam.block_table()
    rng = np.random.default_rng(seed)
    n_t = int(bt.max()) + 1
    pairs = rng.random((K, n_t)) < pair_frac
    pairs[0, int(np.argmax(np.bincount(bt)))] = True
    return pairs[:, bt] | (rng.random((K, bt.size)) < entry_frac)


def custom(shapes, dtype=BF16, block_elems=4096, K=3, active_frac=0.5, log_mu=math.log(1e-2),
           log_sigma=1.0, per_expert_active=False, seed=0, name="custom") -> Family:
    """A small family for tests: shapes is a list of element counts"""
    return Family(name, dtype, [(f"t{t}", int(n)) for t, n in enumerate(shapes)], block_elems, K,
                  active_frac=active_frac, log_mu=log_mu, log_sigma=log_sigma,
                  per_expert_active=per_expert_active, seed=seed)


# ---- native fills -------------------------------------------------------------------------

_host = None
_dev = None


def _host_lib():
    global _host
    if _host is None:
        from .. import build as _b
        path = _b.build_synth_host()
        lib = ctypes.CDLL(path)
        lib.syn_fill_range.restype = ctypes.c_int
        lib.syn_fill_range.argtypes = [ctypes.c_int, ctypes.c_uint64, ctypes.c_uint32, ctypes.c_uint64,
                                       ctypes.c_uint64, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                                       ctypes.c_uint64, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int]
        lib.syn_mix64_export.restype = ctypes.c_uint64
        lib.syn_mix64_export.argtypes = [ctypes.c_uint64]
        _host = lib
    return _host


def _dev_lib():
    global _dev
    if _dev is None:
        from .. import build as _b
        path = _b.build_synth_dev()
        lib = ctypes.CDLL(path)
        lib.syn_dev_fill_base.restype = ctypes.c_int
        lib.syn_dev_fill_base.argtypes = [ctypes.c_int, ctypes.c_uint64, ctypes.c_uint64, ctypes.c_void_p,
                                          ctypes.c_void_p]
        lib.syn_dev_fill_expert.restype = ctypes.c_int
        lib.syn_dev_fill_expert.argtypes = [ctypes.c_int, ctypes.c_uint64, ctypes.c_uint32, ctypes.c_uint64,
                                            ctypes.c_uint64, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                                            ctypes.c_uint32, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p]
        _dev = lib
    return _dev


def _host_fill(fam: Family, stream: int, j0: int, n: int, base_stored, out: np.ndarray, nthreads: int):
    lib = _host_lib()
    if nthreads <= 0:
        nthreads = min(16, os.cpu_count() or 1)
    bo, bl, _ = fam.block_table()
    if stream == 0:
        rc = lib.syn_fill_range(fam.dtype, fam.seed, 0, j0, n, None, None, None, 0, None,
                                out.ctypes.data, nthreads)
    else:
        sc = np.ascontiguousarray(fam.scales()[stream - 1])
        base_stored = np.ascontiguousarray(base_stored)
        rc = lib.syn_fill_range(fam.dtype, fam.seed, stream, j0, n, bo.ctypes.data, bl.ctypes.data,
                                sc.ctypes.data, bo.shape[0], base_stored.ctypes.data, out.ctypes.data,
                                nthreads)
    if rc != 0:
        raise RuntimeError(f"synthetic host fill failed ({rc})")
