"""The merge kernel's TIES mean divides by a count c <= 32 with a reciprocal and one
Markstein correction step; that helper must round exactly like IEEE division.  This
checks it exhaustively against the CUDA division on the GPU: every finite fp32
numerator but -0 (never a TIES numerator: the kernel divides +0 when no sign wins), every
c in 1..32, through a probe compiled here from the kernel's own header."""
import ctypes
import os
import subprocess
import tempfile

import pytest
import torch

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(os.path.dirname(HERE), "paper_2605_29489_gb300", "csrc")


def test_small_count_division_is_ieee_exact():
    from paper_2605_29489_gb300 import build

    d = tempfile.mkdtemp(prefix="small_div_probe_")
    so = os.path.join(d, "probe.so")
    subprocess.check_call([build.nvcc(), *build.ARCH, "-O3", "-fmad=false", "-I", CSRC, "-Xcompiler", "-fPIC",
                           "-shared", os.path.join(HERE, "probes", "small_div_probe.cu"), "-o", so])
    L = ctypes.CDLL(so)
    L.small_div_probe.restype = ctypes.c_int
    L.small_div_probe.argtypes = [ctypes.c_void_p, ctypes.c_void_p]
    bad = torch.zeros(1, dtype=torch.int64, device="cuda")
    first = torch.zeros(3, dtype=torch.int32, device="cuda")
    assert L.small_div_probe(bad.data_ptr(), first.data_ptr()) == 0
    f = first.cpu().tolist()
    assert int(bad.item()) == 0, f"mismatch at a=0x{f[0] & 0xFFFFFFFF:08x}, c={f[1]}"
