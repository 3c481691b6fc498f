"""Pin of the oracle's Philox4x32-10 to an independent implementation of the same
published generator: cuRAND's device Philox4_32_10 (curand_init + curand4), run on
the GPU through a small probe compiled here.  cuRAND's state for (seed, subsequence,
offset = 4*c) evaluates the generator at key = (seed low, seed high) and counter =
(c low, c high, subsequence low, subsequence high), then steps the counter by one per
curand4 call."""
import ctypes
import os
import subprocess
import tempfile

import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))


@pytest.fixture(scope="module")
def probe():
    from paper_2605_29489_gb300 import build

    d = tempfile.mkdtemp(prefix="philox_probe_")
    so = os.path.join(d, "probe.so")
    subprocess.check_call([build.nvcc(), *build.ARCH, "-O2", "-Xcompiler", "-fPIC", "-shared",
                           os.path.join(HERE, "probes", "curand_philox_probe.cu"), "-o", so])
    L = ctypes.CDLL(so)
    L.curand_philox_probe.restype = ctypes.c_int
    L.curand_philox_probe.argtypes = [ctypes.c_void_p] * 3 + [ctypes.c_uint, ctypes.c_uint, ctypes.c_void_p]
    return L


def test_oracle_philox_matches_curand(probe):
    rng = np.random.default_rng(7)
    count, n = 64, 3
    seed = rng.integers(0, 2 ** 63, count, dtype=np.uint64)
    seed[:4] = [0, 1, 0xFFFFFFFF, 0x123456789ABCDEF0]
    subseq = rng.integers(0, 2 ** 40, count, dtype=np.uint64)
    subseq[:4] = [0, 5, 0x44415245, 2 ** 33 + 7]
    c = rng.integers(0, 2 ** 40, count, dtype=np.uint64)
    c[:4] = [0, 1, 2 ** 32 - 1, 2 ** 32]
    offset = c * np.uint64(4)
    d = [torch.from_numpy(x.view(np.int64)).cuda() for x in (seed, subseq, offset)]
    out = torch.zeros(count * n * 4, dtype=torch.int32, device="cuda")
    assert probe.curand_philox_probe(d[0].data_ptr(), d[1].data_ptr(), d[2].data_ptr(), n, count, out.data_ptr()) == 0
    got = out.cpu().numpy().view(np.uint32).reshape(count, n, 4)
    for t in range(count):
        for k in range(n):
            cc = int(c[t]) + k
            ctr = [cc & 0xFFFFFFFF, cc >> 32, int(subseq[t]) & 0xFFFFFFFF, int(subseq[t]) >> 32]
            key = [int(seed[t]) & 0xFFFFFFFF, int(seed[t]) >> 32]
            assert np.array_equal(oracle.philox4x32_10(ctr, key), got[t, k]), (t, k)
